"""presto_score_build_tree (GPU, C ABI) vs the oracle's best-first search with its
decisions taken in float32 (the kernel's precision): topology, order, n_nodes and
the float32 path scores bit-exact on the same inputs."""

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import (GPU, assert_tree_close, assert_tree_exact, reachable_table,
                        synthetic_candidates, to_dev, tree_host)

pytestmark = GPU

MISS = -12.0


def _run(ids, logq, ctx, entries, lam, N, b=None, log2_cap=18):
    B, L, k = ids.shape
    table = None
    ngram = None
    if entries is not None:
        a, bb, t, lr = entries
        table = O.make_table(a, bb, t, lr)
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, log2_cap, MISS)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), ngram,
                                    lam, N, b=b, dev_status=st)
    torch.cuda.synchronize()
    g = tree_host(out)
    o = O.best_first_tree(ids, logq, ctx, table, MISS, lam, b or k, N, "fp32")
    return g, o, int(st.item())


CASES = [
    # B, L, k, b, N, lam, table, quant
    (2, 8, 4, None, 16, 0.2, True, None),        # tiny-shaped
    (1, 16, 8, None, 64, 0.2, True, None),       # Qwen3-8B round
    (16, 16, 8, None, 128, 0.2, True, None),     # batched serving
    (4, 32, 6, None, 256, 0.0, False, None),     # self-speculative, marginal-only
    (8, 16, 10, None, 256, 0.2, True, None),     # long context round
    (3, 6, 8, 3, 100, 0.5, True, None),          # b < k
    (2, 12, 5, None, 200, 0.0, False, 4),        # many exact score ties
    (2, 10, 6, None, 150, 0.2, True, 8),         # ties with a prefix signal
    (1, 1, 16, None, 256, 0.2, True, None),      # one level
    (1, 2, 2, None, 10, 0.2, True, None),        # budget above the candidate tree (7 nodes)
    (2, 5, 3, None, 1, 0.2, True, None),         # root only
]


@pytest.mark.parametrize("B,L,k,b,N,lam,with_table,quant", CASES + [(2, 16, 8, None, 1024, 0.2, True, None)])
def test_fused_mask_matches_oracle(B, L, k, b, N, lam, with_table, quant):
    """presto_score_build_tree_mask: the tree as presto_score_build_tree builds it,
    and the mask and position ids of the oracle's tree, bit-exact."""
    rng = np.random.default_rng(B * 1000 + L * 31 + k * 7 + N)
    vocab = rng.choice(200000, 300, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, 200000, quant=quant, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    entries = reachable_table(rng, ids, ctx) if with_table else None
    table = ngram = None
    if entries is not None:
        a, bb, t, lr = entries
        table = O.make_table(a, bb, t, lr)
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, 18, MISS)
    kv = rng.integers(0, 40000, size=B)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), ngram,
                                    lam, N, b=b, dev_status=st, kv_len=to_dev(kv))
    torch.cuda.synchronize()
    g = tree_host({k2: v for k2, v in out.items() if k2 not in ("mask", "pos_ids")})
    o = O.best_first_tree(ids, logq, ctx, table, MISS, lam, b or k, N, "fp32")
    assert int(st.item()) == 0
    assert_tree_exact(g, o, B)
    omask, opos = O.tree_mask(o["parent"], o["depth"], o["n_nodes"], kv, N)
    np.testing.assert_array_equal(out["mask"].cpu().numpy().view(np.uint32), omask)
    np.testing.assert_array_equal(out["pos_ids"].cpu().numpy(), opos)


@pytest.mark.parametrize("B,L,k,b,N,lam,with_table,quant", CASES)
def test_build_matches_oracle_fp32(B, L, k, b, N, lam, with_table, quant):
    rng = np.random.default_rng(B * 1000 + L * 31 + k * 7 + N)
    vocab = rng.choice(200000, 300, replace=False)          # small pool: contexts repeat
    ids, logq = synthetic_candidates(rng, B, L, k, 200000, quant=quant, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    entries = reachable_table(rng, ids, ctx) if with_table else None
    g, o, st = _run(ids, logq, ctx, entries, lam, N, b=b)
    assert st == 0
    assert_tree_exact(g, o, B)


def test_build_table_in_global_memory():
    """L*k^3 floats above the shared-memory budget: the score table lives in the
    workspace instead."""
    rng = np.random.default_rng(5)
    B, L, k, N = 1, 40, 16, 256
    vocab = rng.choice(100000, 200, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, 100000, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    entries = reachable_table(rng, ids, ctx, density=0.05)
    assert P.presto_build_workspace(B, L, k, N) >= L * k ** 3 * 4
    g, o, st = _run(ids, logq, ctx, entries, 0.2, N, log2_cap=20)
    assert st == 0
    assert_tree_exact(g, o, B)


def test_build_chain_from_gpu_topk_matches_oracle_chain():
    """topk -> build on the GPU vs oracle topk -> oracle build (float64): scores
    within 1e-5, node sets equal away from near-ties at the budget boundary."""
    for name in ("tiny", "qwen3_8b"):
        w = synth.WORKLOADS[name]
        x = synth.drafter_logits(w)
        ctx = synth.ctx_tokens(w).numpy()
        a, bb, t, lr = synth.trigram_entries(w)
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, w.table_log2_cap, w.miss_logrho)
        ids_d, logq_d, _ = P.presto_topk(x.cuda(), w.k)
        out = P.presto_score_build_tree(ids_d, logq_d, to_dev(ctx), ngram, w.lam, w.N)
        g = tree_host(out)
        oids, ologq, _ = O.topk_logsoftmax(x.reshape(w.rows, w.V).double().numpy(), w.k)
        oids = oids.reshape(w.B, w.L, w.k)
        ologq = ologq.reshape(w.B, w.L, w.k)
        table = O.make_table(a, bb, t, lr)
        assert_tree_close(g, oids, ologq, ctx, table, w.miss_logrho, w.lam, w.N)


def test_duplicate_candidates_are_reported():
    ids = np.array([[[5, 5, 6], [7, 8, 9]]])
    logq = -np.ones((1, 2, 3))
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev([[1, 2]]), None,
                              0.0, 8, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x40


def test_positive_scores_are_reported():
    ids = np.array([[[5, 6], [7, 8]]])
    logq = np.array([[[-1.0, 0.5], [-1.0, -2.0]]])
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev([[1, 2]]), None,
                              0.0, 8, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x10
