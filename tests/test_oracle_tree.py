"""Pins for the oracle's prefix-aligned scoring (§4.1) and best-first tree (§4.2).

Independent checks: hand-computed scores of a small example (closed form), the
definition of the target tree written as exhaustive enumeration + sort, the
surrogate objective of Eq. surrogate-objective maximised over every prefix-closed
subset, the prefix-blind special case (Eq. marginal-surrogate), non-triviality
(Def. 2.1) and linear drafting as the k = 1 special case.
"""

import itertools
import math

import numpy as np
import pytest

from oracle import presto_oracle as O

KEYS = ("token", "parent", "depth", "n_nodes", "rank")


def _hand_case():
    # depth 1 candidates: tokens 1, 2; depth 2 candidates: tokens 3, 4.
    ids = np.array([[[1, 2], [3, 4]]])
    logq = np.array([[[-0.5, -1.0], [-0.25, -2.0]]])
    ctx = np.array([[7, 8]])
    table = {(7, 8, 1): -1.0, (8, 1, 3): -4.0, (8, 2, 4): 0.0}
    return ids, logq, ctx, table, -8.0, 0.5


def test_hand_computed_scores_and_order():
    ids, logq, ctx, table, miss, lam = _hand_case()
    # s(1)   = -0.5  + 0.5*(-1)  = -1.0      (hit  7,8,1)
    # s(2)   = -1.0  + 0.5*(-8)  = -5.0      (miss 7,8,2)
    # s(1,3) = -0.25 + 0.5*(-4)  = -2.25     (hit  8,1,3) -> S = -3.25
    # s(1,4) = -2.0  + 0.5*(-8)  = -6.0      (miss 8,1,4) -> S = -7.0
    # s(2,3) = -0.25 + 0.5*(-8)  = -4.25     (miss 8,2,3) -> S = -9.25
    # s(2,4) = -2.0  + 0.5*0     = -2.0      (hit  8,2,4) -> S = -7.0
    # order: root, (1), (1,3), (2), then the S = -7 tie at equal depth and token
    # goes to the parent placed first: (1,4) before (2,4); then (2,3).
    for prec in ("fp32", "fp64"):
        t = O.best_first_tree(ids, logq, ctx, table, miss, lam, 2, 7, prec)
        assert t["token"][0].tolist() == [8, 1, 3, 2, 4, 4, 3]
        assert t["parent"][0].tolist() == [-1, 0, 1, 0, 1, 3, 3]
        assert t["depth"][0].tolist() == [0, 1, 2, 1, 2, 2, 2]
        assert t["score"][0].tolist() == [0.0, -1.0, -3.25, -5.0, -7.0, -7.0, -9.25]
        assert t["score64"][0].tolist() == [0.0, -1.0, -3.25, -5.0, -7.0, -7.0, -9.25]
        t5 = O.best_first_tree(ids, logq, ctx, table, miss, lam, 2, 5, prec)
        assert t5["token"][0].tolist() == [8, 1, 3, 2, 4]
        assert int(t5["n_nodes"][0]) == 5
    # budget above the candidate tree's size: every node, n_nodes < N.
    t = O.best_first_tree(ids, logq, ctx, table, miss, lam, 2, 10)
    assert int(t["n_nodes"][0]) == 7 and t["token"][0, 7:].tolist() == [-1, -1, -1]


def test_branching_keeps_top_b_by_token_score():
    ids, logq, ctx, table, miss, lam = _hand_case()
    t = O.best_first_tree(ids, logq, ctx, table, miss, lam, 1, 10)
    # b = 1: root -> 1 (s=-1 beats -5) -> 3 (s=-2.25 beats -6): a chain.
    assert t["token"][0, :3].tolist() == [8, 1, 3] and int(t["n_nodes"][0]) == 3


def _lazy_vs_eager_case():
    # L = 3, k = 2, no prefix signal. Depth-1 log q: A=-1, B=-5; depth 2: C=-0.1,
    # D=-5; depth 3: E=-0.1, F=-9.  So S(A)=-1, S(AC)=-1.1, S(ACE)=-1.2, S(B)=-5.
    A, B, C, D, E, F = 11, 12, 13, 14, 15, 16
    ids = np.array([[[A, B], [C, D], [E, F]]])
    logq = np.array([[[-1.0, -5.0], [-0.1, -5.0], [-0.1, -9.0]]])
    return ids, logq, np.array([[0, 1]]), (A, B, C, D, E, F)


def test_lazy_reading_beats_printed_eager_variant():
    ids, logq, ctx, (A, B, C, D, E, F) = _lazy_vs_eager_case()
    lazy = O.best_first_tree(ids, logq, ctx, None, 0.0, 0.0, 2, 4, "fp64")
    assert lazy["token"][0].tolist() == [1, A, C, E]
    eager = O.eager_tree(ids, logq, ctx, None, 0.0, 0.0, 2, 4, "fp64")
    assert eager["token"][0].tolist() == [1, A, C, B]
    obj = lambda S: sum(math.exp(s) for s in S)          # Eq. surrogate-objective
    assert obj([0, -1, -1.1, -1.2]) > obj([0, -1, -1.1, -5])


def _random_case(rng, L, k, V, with_table):
    ids = np.stack([rng.choice(V, k, replace=False) for _ in range(L)])[None]
    logq = -np.abs(np.round(rng.normal(0, 1.5, size=(1, L, k)) * 4) / 4)
    ctx = rng.integers(0, V, size=(1, 2))
    table = None
    if with_table:
        table = {}
        for _ in range(3 * V):
            key = tuple(int(v) for v in rng.integers(0, V, 3))
            table[key] = -float(rng.integers(0, 16)) / 8
    return ids, logq, ctx, table


@pytest.mark.parametrize("prec", ["fp32", "fp64"])
def test_best_first_equals_enumeration_definition(prec):
    rng = np.random.default_rng(123)
    cases = 0
    for L in (1, 2, 3, 4):
        for k in (1, 2, 3):
            for bfac in range(1, k + 1):
                for with_table in (False, True):
                    for lam in ((0.0,) if not with_table else (0.0, 0.2, 0.5)):
                        ids, logq, ctx, table = _random_case(rng, L, k, 6, with_table)
                        for N in (1, 2, 5, 13, 200):
                            got = O.best_first_tree(ids, logq, ctx, table, -2.0, lam, bfac, N, prec)
                            want = O.brute_force_tree(ids, logq, ctx, table, -2.0, lam, bfac, N, prec)
                            for key in KEYS:
                                np.testing.assert_array_equal(got[key], want[key], err_msg=key)
                            np.testing.assert_array_equal(got["score"], want["score"])
                            cases += 1
    assert cases > 300


def test_top_n_maximises_surrogate_objective():
    """Eq. surrogate-objective: over all prefix-closed subsets of the candidate tree
    of size N (root included), the best-first tree has the largest sum of exp(S)."""
    rng = np.random.default_rng(7)
    for _ in range(25):
        ids, logq, ctx, table = _random_case(rng, 3, 2, 5, True)
        nodes = O.candidate_tree_nodes(ids[0], logq[0], ctx[0], table, -2.0, 0.3, 2, "fp64")
        S = {p: float(s) for p, s, _ in nodes}
        nonroot = [p for p in S if p]
        for N in (2, 3, 4, 6):
            best = -1.0
            for combo in itertools.combinations(nonroot, N - 1):
                cs = set(combo) | {()}
                if all(p[:-1] in cs for p in combo):
                    best = max(best, sum(math.exp(S[p]) for p in cs))
            t = O.best_first_tree(ids, logq, ctx, table, -2.0, 0.3, 2, N, "fp64")
            got = sum(math.exp(s) for s in t["score64"][0, :N])
            assert got >= best - 1e-12


def test_marginal_only_is_prefix_blind():
    """lambda = 0 (or no table): s = log q whatever the context (Eq.
    marginal-surrogate), and S of a path is the sum of its log-marginals."""
    rng = np.random.default_rng(5)
    ids, logq, ctx, table = _random_case(rng, 4, 3, 7, True)
    with_t = O.best_first_tree(ids, logq, ctx, table, -2.0, 0.0, 3, 30, "fp64")
    without = O.best_first_tree(ids, logq, ctx, None, -2.0, 0.0, 3, 30, "fp64")
    for key in KEYS:
        np.testing.assert_array_equal(with_t[key], without[key])
    for i in range(1, int(without["n_nodes"][0])):
        j, total = i, 0.0
        while j > 0:
            total += logq[0, without["depth"][0, j] - 1, without["rank"][0, j]]
            j = without["parent"][0, j]
        assert without["score64"][0, i] == pytest.approx(total, abs=1e-12)


def test_prefix_aligned_score_is_nontrivial():
    """Def. 2.1: with lambda > 0 and a context-dependent rho, the same (d, t)
    scores differently under two prefixes."""
    ids, logq, ctx, table, miss, lam = _hand_case()
    s_after_1 = O.children(ids[0], logq[0], ctx[0], table, miss, lam, 2, (1,), "fp64")
    s_after_2 = O.children(ids[0], logq[0], ctx[0], table, miss, lam, 2, (2,), "fp64")
    d1 = {t: s for s, t, _ in s_after_1}
    d2 = {t: s for s, t, _ in s_after_2}
    assert d1[3] != d2[3] and d1[4] != d2[4]
    s0 = O.children(ids[0], logq[0], ctx[0], table, miss, 0.0, 2, (1,), "fp64")
    s0b = O.children(ids[0], logq[0], ctx[0], table, miss, 0.0, 2, (2,), "fp64")
    assert s0 == s0b


def test_linear_drafting_is_the_k1_chain():
    """§1 linear drafting: with one candidate per position the tree is the top-1
    chain t_1, ..., t_L."""
    rng = np.random.default_rng(9)
    ids, logq, ctx, table = _random_case(rng, 5, 1, 9, True)
    t = O.best_first_tree(ids, logq, ctx, table, -2.0, 0.2, 1, 100)
    assert int(t["n_nodes"][0]) == 6
    assert t["token"][0, 1:6].tolist() == ids[0, :, 0].tolist()
    assert t["parent"][0, :6].tolist() == [-1, 0, 1, 2, 3, 4]


def test_structure_invariants_on_random_trees():
    rng = np.random.default_rng(11)
    for _ in range(20):
        ids, logq, ctx, table = _random_case(rng, 6, 4, 30, True)
        t = O.best_first_tree(ids, logq, ctx, table, -3.0, 0.2, 3, 40)
        n = int(t["n_nodes"][0])
        S = t["score"][0]
        assert t["depth"][0, 0] == 0 and S[0] == 0
        for i in range(1, n):
            p = t["parent"][0, i]
            assert 0 <= p < i
            assert t["depth"][0, i] == t["depth"][0, p] + 1
            assert S[i] <= S[p]                             # s <= 0 down a path
            assert S[i] <= S[i - 1]                          # output in score order
            # A3 additivity in float64
            sc = O.token_score(logq[0, t["depth"][0, i] - 1, t["rank"][0, i]],
                               None if table is None else table.get(
                                   O.trigram_context(ctx[0], _path(t, i)[:-1]) + (int(t["token"][0, i]),), -3.0),
                               0.2, "fp64")
            assert t["score64"][0, i] - t["score64"][0, p] == pytest.approx(sc, abs=1e-12)
        sib = {}
        for i in range(1, n):
            sib.setdefault(t["parent"][0, i], []).append(int(t["token"][0, i]))
        assert all(len(v) == len(set(v)) for v in sib.values())


def _path(t, i):
    out = []
    while i > 0:
        out.append(int(t["token"][0, i]))
        i = int(t["parent"][0, i])
    return tuple(reversed(out))


def test_competing_pairs_flags_near_ties():
    t = {"score64": np.array([[0.0, -1.0, -1.0 - 1e-7, -2.0]]), "n_nodes": np.array([4])}
    assert O.competing_pairs(t, 0) == [(1, 2)]
