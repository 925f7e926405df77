"""Pins for the oracle's log-softmax / top-k step (§2.3, §4.3).

Checked against things other than the oracle itself: scipy's logsumexp, the
normalisation of a distribution, a pure-Python sort, and the planted peaks of the
tiny workload.
"""

import numpy as np
import pytest
import scipy.special
import torch

import synth
from oracle import presto_oracle as O

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def _rows(seed, R, V, quant=None):
    rng = np.random.default_rng(seed)
    x = rng.normal(0, 3, size=(R, V))
    if quant:
        x = np.round(x * quant) / quant          # many exact ties
    return x


def test_lse_matches_scipy_and_normalises():
    x = _rows(0, 7, 1001)
    _, _, lse = O.topk_logsoftmax(x, 5)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(x, axis=1), rtol=0, atol=1e-12)
    total = np.exp(x - lse[:, None]).sum(axis=1)
    np.testing.assert_allclose(total, 1.0, rtol=0, atol=1e-12)


def test_bf16_inputs_are_taken_exactly():
    x = torch.randn(3, 513, generator=torch.Generator().manual_seed(1)).to(torch.bfloat16)
    ids, logq, lse = O.topk_logsoftmax(x.float().numpy(), 4)
    xd = x.double().numpy()
    np.testing.assert_allclose(lse, scipy.special.logsumexp(xd, axis=1), atol=1e-12)
    np.testing.assert_array_equal(np.take_along_axis(xd, ids, 1) - lse[:, None], logq)


@pytest.mark.parametrize("quant", [None, 1, 4])
def test_ids_match_python_sort_with_ties(quant):
    x = _rows(2, 9, 300, quant)
    for k in (1, 3, 8, 300):
        ids, logq, lse = O.topk_logsoftmax(x, k)
        for r in range(x.shape[0]):
            want = sorted(range(x.shape[1]), key=lambda v: (-x[r, v], v))[:k]
            assert ids[r].tolist() == want
        assert np.all(np.diff(logq, axis=1) <= 0)


def test_tie_goes_to_lower_id():
    x = np.array([[1.0, 3.0, 3.0, 2.0, 3.0]])
    ids, _, _ = O.topk_logsoftmax(x, 2)
    assert ids[0].tolist() == [1, 2]


def test_planted_peak_rank_by_counting():
    """The planted token's rank is the number of entries that beat it (larger
    value, or equal value and lower id); where that rank is below k it must sit
    there in the top-k list."""
    w = synth.WORKLOADS["tiny"]
    x = synth.drafter_logits(w).reshape(w.B * w.L, w.V).numpy().astype(np.float64)
    ids, logq, _ = O.topk_logsoftmax(x, w.k)
    peaks = torch.cat([synth.workloads.planted_peaks(w, b) for b in range(w.B)]).numpy()
    at_zero = 0
    for r, p in enumerate(peaks):
        rank = int(np.sum(x[r] > x[r, p]) + np.sum((x[r] == x[r, p]) & (np.arange(w.V) < p)))
        if rank < w.k:
            assert ids[r, rank] == p
        at_zero += rank == 0
    assert at_zero >= len(peaks) // 2
    assert np.all(logq <= 0)


def test_dominant_logit_has_log_prob_near_zero():
    x = np.zeros((1, 50))
    x[0, 17] = 60.0
    ids, logq, _ = O.topk_logsoftmax(x, 1)
    assert ids[0, 0] == 17 and abs(logq[0, 0]) < 1e-20


def test_bad_k_rejected():
    with pytest.raises(ValueError):
        O.topk_logsoftmax(np.zeros((1, 4)), 5)
