"""The paper's large node budgets (N = 512, 1024; Table 1 sweeps to 1024) through the
C ABI: tree build (best-first, beam, printed Alg. 2) bit-exact against the oracle's
float32 search, the selection scratch in shared memory or in the workspace, the
mask and acceptance bit-exact, and the top-k -> build chain at Qwen3-8B shapes."""

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


def _case(seed, B, L, k, with_table, quant=None):
    rng = np.random.default_rng(seed)
    vocab = rng.choice(200000, 400, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, 200000, quant=quant, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    entries = reachable_table(rng, ids, ctx) if with_table else None
    return ids, logq, ctx, entries


def _build(ids, logq, ctx, entries, lam, N, policy, W):
    ngram = None
    if entries is not None:
        a, bb, t, lr = entries
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, 18, MISS)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), ngram,
                                    lam, N, dev_status=st, policy=policy, beam_width=W)
    torch.cuda.synchronize()
    return tree_host(out), int(st.item())


CASES = [
    # B, L, k, N, table, quant: qwen3-like rows; a small k (scratch fits shared memory);
    # many exact ties; marginal-only scoring
    (1, 16, 8, 1024, True, None),
    (2, 16, 8, 512, True, None),
    (2, 8, 4, 1024, True, None),
    (2, 12, 5, 1024, False, 4),
    (3, 32, 6, 512, False, None),
]


@pytest.mark.parametrize("B,L,k,N,with_table,quant", CASES)
@pytest.mark.parametrize("policy,W", [("best_first", 1), ("beam", 10), ("beam", 64), ("eager", 1)])
def test_large_budget_build_matches_oracle_fp32(B, L, k, N, with_table, quant, policy, W):
    ids, logq, ctx, entries = _case(B * 7 + L * 3 + k + N, B, L, k, with_table, quant)
    lam = 0.2 if with_table else 0.0
    pol = {"best_first": P.SEARCH_BEST_FIRST, "beam": P.SEARCH_BEAM, "eager": P.SEARCH_EAGER}[policy]
    g, st = _build(ids, logq, ctx, entries, lam, N, pol, W)
    table = None
    if entries is not None:
        a, bb, t, lr = entries
        table = O.make_table(a, bb, t, lr)
    if policy == "best_first":
        o = O.best_first_tree(ids, logq, ctx, table, MISS, lam, k, N, "fp32")
    elif policy == "beam":
        o = O.beam_search_tree(ids, logq, ctx, table, MISS, lam, k, N, W, "fp32")
    else:
        o = O.eager_tree(ids, logq, ctx, table, MISS, lam, k, N, "fp32")
    assert st == 0
    assert_tree_exact(g, o, B)


def test_large_budget_workspace_size_covers_the_scratch():
    """N = 1024 with k = 8 needs the selection scratch in the workspace."""
    ws = P.presto_build_workspace(1, 16, 8, 1024, 64)
    assert ws > 300 * 1024
    assert P.presto_build_workspace(1, 16, 8, 64) == 256


def test_mask_and_accept_at_1024_nodes():
    rng = np.random.default_rng(31)
    B, L, k, N = 3, 16, 8, 1024
    ids, logq = synthetic_candidates(rng, B, L, k, 5000)
    ctx = rng.integers(0, 5000, size=(B, 2))
    t = O.best_first_tree(ids, logq, ctx, None, 0.0, 0.0, k, N, "fp64")
    kv = rng.integers(0, 40000, size=B)
    mask, pos = P.presto_tree_mask(to_dev(t["parent"]), to_dev(t["depth"]), to_dev(t["n_nodes"]),
                                   to_dev(kv))
    omask, opos = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, N)
    np.testing.assert_array_equal(mask.cpu().numpy().view(np.uint32), omask)
    np.testing.assert_array_equal(pos.cpu().numpy(), opos)
    for trial in range(3):
        tgt = np.full((B, N), -1, np.int64)
        for b in range(B):            # follow the root path of a random node
            j = int(rng.integers(1, N))
            path = []
            while j > 0:
                path.append(j)
                j = int(t["parent"][b, j])
            prev = 0
            for j in reversed(path):
                tgt[b, prev] = t["token"][b, j]
                prev = j
        acc, apath, bonus = P.presto_accept(to_dev(t["token"]), to_dev(t["parent"]),
                                            to_dev(t["depth"]), mask, to_dev(t["n_nodes"]),
                                            to_dev(tgt), L)
        oacc, opath, obonus = O.accept(t["token"], t["parent"], t["n_nodes"], tgt, L)
        np.testing.assert_array_equal(acc.cpu().numpy(), oacc)
        np.testing.assert_array_equal(apath.cpu().numpy(), opath)
        np.testing.assert_array_equal(bonus.cpu().numpy(), obonus)


def test_topk_build_chain_at_1024_nodes():
    w = synth.WORKLOADS["qwen3_8b"].scaled(N=1024, k=10)
    x = synth.drafter_logits(w)
    ctx = synth.ctx_tokens(w).numpy()
    a, bb, t, lr = synth.trigram_entries(w)
    ngram = P.Ngram3Table.from_entries(a, bb, t, lr, w.table_log2_cap, w.miss_logrho)
    ids_d, logq_d, _ = P.presto_topk(x.cuda(), w.k)
    out = P.presto_score_build_tree(ids_d, logq_d, to_dev(ctx), ngram, w.lam, w.N)
    g = tree_host(out)
    oids, ologq, _ = O.topk_logsoftmax(x.reshape(w.rows, w.V).double().numpy(), w.k)
    table = O.make_table(a, bb, t, lr)
    assert_tree_close(g, oids.reshape(w.B, w.L, w.k), ologq.reshape(w.B, w.L, w.k), ctx, table,
                      w.miss_logrho, w.lam, w.N)
