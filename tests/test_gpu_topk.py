"""presto_topk (GPU, through the C ABI) vs the oracle: ids bit-exact, log q and
lse within 1e-5 * max(1, |x|)."""

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import GPU, rel_close

pytestmark = GPU


def _check(logits_cpu, k, view=None):
    """logits_cpu: [B, L, V] CPU tensor; view(t) may return a strided view on device."""
    B, L, V = logits_cpu.shape
    dev = logits_cpu.cuda()
    if view is not None:
        dev = view(dev)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ids, logq, lse = P.presto_topk(dev, k, dev_status=st)
    torch.cuda.synchronize()
    oids, ologq, olse = O.topk_logsoftmax(logits_cpu.reshape(B * L, V).double().numpy(), k)
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(B * L, k), oids)
    assert rel_close(logq.cpu().numpy().reshape(B * L, k), ologq) <= 1e-5
    assert rel_close(lse.cpu().numpy().reshape(-1), olse) <= 1e-5
    return int(st.item())


@pytest.mark.parametrize("name", ["tiny", "qwen3_8b", "self_spec", "long_ctx", "batched_ragged"])
def test_topk_workloads(name):
    w = synth.WORKLOADS[name]
    x = synth.drafter_logits(w)
    assert _check(x, w.k) == 0


def test_topk_few_rows_spread_over_many_ctas():
    """A handful of long rows: each row spans more CTAs than one cluster holds and
    the spans merge through the workspace."""
    g = torch.Generator().manual_seed(11)
    for B, L in ((1, 1), (1, 4), (2, 3)):
        x = (torch.randn(B, L, 151936, generator=g) * 2).to(torch.bfloat16)
        assert _check(x, 10) == 0


@pytest.mark.parametrize("V,dtype,k", [(4097, torch.float32, 4), (1001, torch.bfloat16, 7),
                                       (16, torch.float32, 16), (31, torch.bfloat16, 1),
                                       (151936, torch.bfloat16, 16), (8, torch.bfloat16, 8),
                                       (70000, torch.float32, 10)])
def test_topk_ragged_vocab_and_k(V, dtype, k):
    g = torch.Generator().manual_seed(V + k)
    x = (torch.randn(3, 5, V, generator=g) * 3).to(dtype)
    assert _check(x, k) == 0


def test_topk_unaligned_rows_use_plain_loads():
    g = torch.Generator().manual_seed(7)
    for dtype in (torch.float32, torch.bfloat16):
        wide = (torch.randn(2, 6, 5003, generator=g) * 2).to(dtype)
        V = 4999
        sub = wide[:, :, :V].contiguous()       # the oracle sees the same values
        assert _check(sub, 6, view=lambda t, w=wide: w.cuda()[:, :, :V]) == 0


def test_topk_many_ties_and_masked_vocab():
    g = torch.Generator().manual_seed(3)
    x = torch.round(torch.randn(2, 8, 20000, generator=g) * 2) / 2   # values on a 0.5 grid
    x[:, :, ::3] = -float("inf")                                       # masked tokens
    assert _check(x.to(torch.bfloat16), 9) == 0
    assert _check(x, 16) == 0


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_topk_candidate_overflow_in_register_kernel(dtype):
    """Few rows (the register-resident kernel) whose spans hold far more elements at
    or above the threshold than the candidate buffer: constant rows, two-valued rows
    and a row whose top values repeat; the threshold is raised over the kept data
    until the keys fit, and ties go to the lower id."""
    g = torch.Generator().manual_seed(21)
    V = 151936
    x = torch.randn(1, 4, V, generator=g)
    x[0, 0] = 1.25                                                  # constant
    x[0, 1] = (torch.rand(V, generator=g) < 0.5).float()            # two values
    x[0, 2, ::7] = 9.0                                              # repeated maximum
    x[0, 3, 100000:] = 5.0                                          # tied tail
    assert _check(x.to(dtype), 8) == 0
    assert _check(x[:, :2, :20000].contiguous().to(dtype), 16) == 0


def test_topk_large_magnitudes():
    g = torch.Generator().manual_seed(4)
    x = torch.randn(1, 4, 30000, generator=g) * 40
    assert _check(x, 5) == 0


def test_topk_all_masked_row_reports_nonfinite():
    x = torch.full((1, 2, 300), -float("inf"))
    x[0, 1, 5] = 1.0
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_topk(x.cuda(), 2, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x100


@pytest.mark.parametrize("V,dtype,k", [(151936, torch.bfloat16, 8), (1001, torch.bfloat16, 7),
                                       (4097, torch.float32, 16), (16, torch.float32, 16),
                                       (70000, torch.float32, 10)])
def test_topk_many_rows_stream(V, dtype, k):
    """More rows than one wave of the register-resident kernel holds: the launch
    streams the rows through a ring of bulk copies instead."""
    g = torch.Generator().manual_seed(V * 3 + k)
    x = (torch.randn(8, 60, V, generator=g) * 3).to(dtype)
    assert _check(x, k) == 0


def test_topk_stream_ties_masks_and_adversarial_rows():
    """Ties on a grid with a masked vocabulary; constant rows (every element a
    candidate); increasing rows (every chunk beats the threshold of the last):
    the candidate buffer overflows and the thresholds are raised exactly."""
    g = torch.Generator().manual_seed(12)
    x = torch.round(torch.randn(8, 50, 20000, generator=g) * 2) / 2
    x[:, :, ::3] = -float("inf")
    assert _check(x.to(torch.bfloat16), 9) == 0
    assert _check(x, 16) == 0
    y = torch.randn(8, 50, 70000, generator=g)
    y[0, :5] = 1.25                                             # constant rows
    y[1, :5] = torch.linspace(-20, 20, 70000)                   # increasing rows
    y[2, :5] = torch.linspace(20, -20, 70000)                   # decreasing rows
    assert _check(y, 12) == 0


@pytest.mark.parametrize("dtype,Vw,off,V,k", [(torch.float32, 70008, 3, 70003, 11),
                                              (torch.bfloat16, 151944, 5, 151937, 8)])
def test_topk_streaming_plan_misaligned_base_and_tail(dtype, Vw, off, V, k):
    """Many long rows (the streaming plan: equal pieces that cross row boundaries,
    partials merged per row) whose base is not 16-byte aligned while the row stride
    is: every row has the same few head elements before its first aligned vector and
    a tail after its last."""
    g = torch.Generator().manual_seed(Vw + off)
    wide = (torch.randn(4, 32, Vw, generator=g) * 3).to(dtype)
    sub = wide[:, :, off:off + V].contiguous()
    assert _check(sub, k, view=lambda t, w=wide: w.cuda()[:, :, off:off + V]) == 0
