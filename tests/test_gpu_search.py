"""presto_score_build_tree_ex (GPU, C ABI) vs the oracle, decisions in float32:
beam search with global retention (Alg. 1), Alg. 2 as printed (eager), and a
per-row lambda (App. F) -- topology, order, n_nodes and the float32 path scores
bit-exact on the same inputs."""

import numpy as np
import pytest
import torch

import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import (GPU, assert_tree_exact, reachable_table, synthetic_candidates, to_dev,
                        tree_host)

pytestmark = GPU

MISS = -12.0


def _case(seed, B, L, k, N, with_table, quant=None):
    rng = np.random.default_rng(seed)
    vocab = rng.choice(200000, 300, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, 200000, quant=quant, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    entries = reachable_table(rng, ids, ctx) if with_table else None
    return ids, logq, ctx, entries


def _gpu(ids, logq, ctx, entries, lam, N, b, policy, W, lambda_d=None):
    ngram = None
    if entries is not None:
        a, bb, t, lr = entries
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, 18, MISS)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), ngram,
                                    lam, N, b=b, dev_status=st, policy=policy, beam_width=W,
                                    lambda_d=None if lambda_d is None
                                    else torch.as_tensor(lambda_d, dtype=torch.float32).cuda())
    torch.cuda.synchronize()
    return tree_host(out), int(st.item())


def _table(entries):
    if entries is None:
        return None
    a, bb, t, lr = entries
    return O.make_table(a, bb, t, lr)


BEAM_CASES = [
    # B, L, k, b, N, lam, table, W, quant
    (1, 16, 10, None, 64, 0.2, True, 10, None),     # the paper's default: W = k = 10
    (1, 16, 8, None, 64, 0.2, True, 4, None),       # Qwen3-8B round, narrow beam
    (16, 16, 8, None, 128, 0.2, True, 10, None),    # batched serving
    (4, 32, 6, None, 256, 0.0, False, 10, None),    # self-speculative, marginal-only
    (2, 8, 4, None, 16, 0.2, True, 1, None),        # greedy beam
    (3, 6, 8, 3, 100, 0.5, True, 16, None),         # b < k, wide beam
    (2, 12, 5, None, 200, 0.0, False, 64, 4),       # many exact score ties
    (2, 10, 6, None, 150, 0.2, True, 200, 8),       # beam wider than N
    (1, 2, 2, None, 10, 0.2, True, 2, None),        # budget above the tree
    (2, 5, 3, None, 1, 0.2, True, 3, None),         # root only
]


@pytest.mark.parametrize("B,L,k,b,N,lam,with_table,W,quant", BEAM_CASES)
def test_beam_matches_oracle_fp32(B, L, k, b, N, lam, with_table, W, quant):
    ids, logq, ctx, entries = _case(B * 1000 + L * 31 + k * 7 + N + W, B, L, k, N, with_table,
                                    quant)
    g, st = _gpu(ids, logq, ctx, entries, lam, N, b, P.SEARCH_BEAM, W)
    o = O.beam_search_tree(ids, logq, ctx, _table(entries), MISS, lam, b or k, N, W, "fp32")
    assert st == 0
    assert_tree_exact(g, o, B)


EAGER_CASES = [
    (2, 8, 4, None, 16, 0.2, True, None),
    (1, 16, 8, None, 64, 0.2, True, None),
    (16, 16, 8, None, 128, 0.2, True, None),
    (4, 32, 6, None, 256, 0.0, False, None),
    (3, 6, 8, 3, 100, 0.5, True, None),
    (2, 12, 5, None, 200, 0.0, False, 4),
    (1, 2, 2, None, 10, 0.2, True, None),
    (2, 5, 3, None, 1, 0.2, True, None),
]


@pytest.mark.parametrize("B,L,k,b,N,lam,with_table,quant", EAGER_CASES)
def test_eager_matches_oracle_fp32(B, L, k, b, N, lam, with_table, quant):
    ids, logq, ctx, entries = _case(B * 977 + L * 13 + k + N, B, L, k, N, with_table, quant)
    g, st = _gpu(ids, logq, ctx, entries, lam, N, b, P.SEARCH_EAGER, 1)
    o = O.eager_tree(ids, logq, ctx, _table(entries), MISS, lam, b or k, N, "fp32")
    assert st == 0
    assert_tree_exact(g, o, B)


@pytest.mark.parametrize("policy", ["best_first", "beam", "eager"])
def test_per_row_lambda_matches_oracle_fp32(policy):
    B, L, k, N = 4, 16, 8, 64
    ids, logq, ctx, entries = _case(4242, B, L, k, N, True)
    rng = np.random.default_rng(5)
    lam_d = rng.uniform(0.0, 0.6, size=(B, L)).astype(np.float32)
    pol = {"best_first": P.SEARCH_BEST_FIRST, "beam": P.SEARCH_BEAM, "eager": P.SEARCH_EAGER}[policy]
    g, st = _gpu(ids, logq, ctx, entries, 0.0, N, None, pol, 10, lambda_d=lam_d)
    table = _table(entries)
    lam64 = lam_d.astype(np.float64)
    if policy == "best_first":
        o = O.best_first_tree(ids, logq, ctx, table, MISS, lam64, k, N, "fp32")
    elif policy == "beam":
        o = O.beam_search_tree(ids, logq, ctx, table, MISS, lam64, k, N, 10, "fp32")
    else:
        o = O.eager_tree(ids, logq, ctx, table, MISS, lam64, k, N, "fp32")
    assert st == 0
    assert_tree_exact(g, o, B)


def test_negative_lambda_row_is_reported():
    ids, logq, ctx, entries = _case(17, 1, 4, 3, 8, True)
    lam_d = np.array([[0.2, -0.5, 0.2, 0.2]], dtype=np.float32)
    _, st = _gpu(ids, logq, ctx, entries, 0.2, 8, None, P.SEARCH_BEST_FIRST, 1, lambda_d=lam_d)
    assert st & 0x10
