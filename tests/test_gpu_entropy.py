"""presto_topk_entropy (GPU, C ABI) vs the oracle: the top-k outputs exactly as
presto_topk's, each row's entropy H_d and the adaptive lambda_d(H_d) of App. F.

Tolerances.  H = ln s - ln2 t / s comes from float32 sums of exp2 terms (the
same sums as lse), so it is held to the lse bound: |H - H_oracle| <= 1e-5 max(1, H).
lambda = beta H / (H + C) moves by |dlambda/dH| = beta C / (H + C)^2 per unit of H,
so its bound is that slope times the H bound, plus a few float32 roundings."""

import math

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import GPU, LOGQ_TOL, assert_tree_close, rel_close, to_dev, tree_host

pytestmark = GPU

BETA, C = 0.5, 2.0


def _check(x_cpu, k, beta=BETA, c=C):
    B, L, V = x_cpu.shape
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ids, logq, lse, H, lam = P.presto_topk_entropy(x_cpu.cuda(), k, beta, c, dev_status=st)
    torch.cuda.synchronize()
    rows = x_cpu.reshape(B * L, V).double().numpy()
    oids, ologq, olse = O.topk_logsoftmax(rows, k)
    oH = O.drafter_entropy(rows)
    olam = O.entropy_adaptive_lambda(oH, beta, c)
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(B * L, k), oids)
    assert rel_close(logq.cpu().numpy().reshape(B * L, k), ologq) <= LOGQ_TOL
    assert rel_close(lse.cpu().numpy().reshape(-1), olse) <= LOGQ_TOL
    gH = H.cpu().numpy().reshape(-1).astype(np.float64)
    hb = LOGQ_TOL * np.maximum(1.0, oH)
    assert np.all(np.abs(gH - oH) <= hb), float(np.max(np.abs(gH - oH) / hb))
    glam = lam.cpu().numpy().reshape(-1).astype(np.float64)
    lb = beta * c / (oH + c) ** 2 * hb + 4 * 2.0 ** -24 * olam
    assert np.all(np.abs(glam - olam) <= lb), float(np.max(np.abs(glam - olam) / lb))
    return int(st.item()), gH, oH


@pytest.mark.parametrize("name", ["tiny", "qwen3_8b", "self_spec", "batched_ragged"])
def test_entropy_workloads(name):
    w = synth.WORKLOADS[name]
    assert _check(synth.drafter_logits(w), w.k)[0] == 0


@pytest.mark.parametrize("V,dtype,k,scale", [(4097, torch.float32, 4, 3.0), (1001, torch.bfloat16, 7, 1.0),
                                             (31, torch.bfloat16, 1, 0.1), (151936, torch.bfloat16, 16, 8.0),
                                             (70000, torch.float32, 10, 30.0)])
def test_entropy_ragged_vocab_and_sharpness(V, dtype, k, scale):
    g = torch.Generator().manual_seed(V + k)
    x = (torch.randn(3, 5, V, generator=g) * scale).to(dtype)
    assert _check(x, k)[0] == 0


def test_entropy_few_long_rows_merge_across_a_cluster():
    g = torch.Generator().manual_seed(3)
    for B, L in ((1, 1), (1, 4), (2, 3)):
        x = (torch.randn(B, L, 151936, generator=g) * 2).to(torch.bfloat16)
        assert _check(x, 10)[0] == 0


def test_entropy_closed_forms_on_the_gpu():
    """Uniform rows give log V, a single finite entry 0, two finite entries the
    binary entropy; -inf entries (a masked vocabulary) add nothing."""
    V = 151936
    x = torch.full((1, 4, V), float("-inf"))
    x[0, 0] = 1.5                                  # uniform
    x[0, 1, 12345] = 7.0                           # one finite entry
    x[0, 2, 3], x[0, 2, V - 1] = 2.0, -1.0         # two finite entries, one in the tail
    x[0, 3, : V // 2] = torch.linspace(-3, 3, V // 2)  # half the vocabulary masked
    st, gH, oH = _check(x, 1)
    assert st == 0
    assert abs(gH[0] - math.log(V)) <= LOGQ_TOL * math.log(V)
    assert 0.0 <= gH[1] <= LOGQ_TOL
    p = 1 / (1 + math.exp(-3.0))
    assert abs(gH[2] - (-(p * math.log(p) + (1 - p) * math.log(1 - p)))) <= LOGQ_TOL


def test_entropy_only_and_bad_arguments():
    x = torch.randn(1, 2, 999).cuda()
    ids, logq, lse, H, lam = P.presto_topk_entropy(x, 3)      # no beta, C: entropy only
    torch.cuda.synchronize()
    assert lam is None
    oH = O.drafter_entropy(x.cpu().double().numpy().reshape(2, 999))
    assert np.all(np.abs(H.cpu().numpy().reshape(-1) - oH) <= LOGQ_TOL * np.maximum(1, oH))
    for beta, c in ((0.0, 1.0), (1.0, 0.0), (-1.0, 1.0), (1.0, float("inf"))):
        with pytest.raises(P.PrestoError):
            P.presto_topk_entropy(x, 3, beta, c)
    with pytest.raises(P.PrestoError):
        P.presto_topk_entropy(x, 3, with_entropy=False)        # neither output


def test_adaptive_lambda_chain_matches_oracle_chain():
    """topk_entropy -> build with lambda_d on the GPU vs the oracle's float64 chain
    with its own lambda_d.  Scores differ by at most sum_d |dlambda_d| |log rho| on top
    of the top-k bound; node sets agree away from near-ties at the budget edge."""
    for name in ("tiny", "qwen3_8b"):
        w = synth.WORKLOADS[name]
        x = synth.drafter_logits(w)
        ctx = synth.ctx_tokens(w).numpy()
        a, bb, t, lr = synth.trigram_entries(w)
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, w.table_log2_cap, w.miss_logrho)
        ids_d, logq_d, _, _, lam_d = P.presto_topk_entropy(x.cuda(), w.k, BETA, C)
        out = P.presto_score_build_tree(ids_d, logq_d, to_dev(ctx), ngram, 0.0, w.N, lambda_d=lam_d)
        g = tree_host(out)
        rows = x.reshape(w.rows, w.V).double().numpy()
        oids, ologq, _ = O.topk_logsoftmax(rows, w.k)
        olam = O.entropy_adaptive_lambda(O.drafter_entropy(rows), BETA, C).reshape(w.B, w.L)
        table = O.make_table(a, bb, t, lr)
        dlam = float(np.max(np.abs(lam_d.cpu().numpy().astype(np.float64) - olam)))
        worst = max(abs(w.miss_logrho), float(np.max(np.abs(lr))))
        tol = LOGQ_TOL + w.L * dlam * worst
        assert_tree_close(g, oids.reshape(w.B, w.L, w.k), ologq.reshape(w.B, w.L, w.k), ctx, table,
                          w.miss_logrho, olam, w.N, tol=tol)
