"""Pins for the oracle's beam search with global retention (§4.2, Alg. 1) and for
Alg. 2 as printed (the eager variant of reading R7).

Independent checks: with an unbounded beam width, Alg. 1 keeps the N best nodes of
the candidate tree truncated at the depth where |T| first reaches N (exhaustive
enumeration + sort); with width 1 it follows the greedy path; with b = 1 it is
linear drafting; |T| follows a closed-form count; the eager variant expands nodes in
the lazy best-first order, so its output is the lazy prefix of X nodes followed by
the best of their unexpanded children.
"""

import math

import numpy as np
import pytest

from oracle import presto_oracle as O

KEYS = ("token", "parent", "depth", "n_nodes", "rank")


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


def _ranked(nodes):
    """Enumerated nodes (path, S, ranks) sorted by the total order R6 written
    recursively on paths: (-S, depth, token, key(parent))."""
    by_path = {p: (S, r) for p, S, r in nodes}
    memo = {}

    def key(p):
        if p not in memo:
            memo[p] = () if not p else (-float(by_path[p][0]), len(p), p[-1], key(p[:-1]))
        return memo[p]

    return sorted(by_path, key=key), by_path


def _as_rows(chosen, by_path, root_token):
    index = {p: i for i, p in enumerate(chosen)}
    return {
        "token": [root_token if not p else p[-1] for p in chosen],
        "parent": [-1 if not p else index[p[:-1]] for p in chosen],
        "depth": [len(p) for p in chosen],
        "score": [float(by_path[p][0]) for p in chosen],
    }


def _check(got, want, n):
    assert got["n_nodes"][0] == n
    for key in ("token", "parent", "depth", "score"):
        np.testing.assert_array_equal(got[key][0, :n], np.asarray(want[key]), err_msg=key)


@pytest.mark.parametrize("prec", ["fp32", "fp64"])
def test_unbounded_beam_keeps_top_n_of_the_expanded_depths(prec):
    rng = np.random.default_rng(7)
    cases = 0
    for L in (1, 2, 3, 4):
        for k in (2, 3):
            for bfac in range(1, k + 1):
                for with_table in (False, True):
                    ids, logq, ctx, table = _random_case(rng, L, k, 6, with_table)
                    lam = 0.3 if with_table else 0.0
                    nodes = O.candidate_tree_nodes(ids[0], logq[0], ctx[0], table, -2.0, lam,
                                                   bfac, prec)
                    for N in (1, 2, 4, 9, 30, 500):
                        # the depths Alg. 1 expands: while |T| < N, one more depth
                        count, dstar = 1, 0
                        while dstar < L and count < N:
                            dstar += 1
                            count += sum(1 for p, _, _ in nodes if len(p) == dstar)
                        order, by_path = _ranked([e for e in nodes if len(e[0]) <= dstar])
                        chosen = order[:N]
                        got = O.beam_search_tree(ids, logq, ctx, table, -2.0, lam, bfac, N,
                                                 10 ** 6, prec)
                        _check(got, _as_rows(chosen, by_path, int(ctx[0, 1])), len(chosen))
                        cases += 1
    assert cases > 80


def test_width_one_follows_the_greedy_path():
    rng = np.random.default_rng(8)
    for trial in range(40):
        L, k = 4, 3
        ids, logq, ctx, table = _random_case(rng, L, k, 7, trial % 2 == 1)
        lam = 0.25 if table is not None else 0.0
        bfac, N = 3, 12
        nodes = O.candidate_tree_nodes(ids[0], logq[0], ctx[0], table, -2.0, lam, bfac, "fp64")
        order, by_path = _ranked(nodes)
        rank = {p: i for i, p in enumerate(order)}
        # greedy path: from the root, the best child (order R6) at each depth; T is the
        # root plus every child of the path's nodes, for as long as |T| < N
        T, g = [()], ()
        while len(g) < L and len(T) < N:
            kids = [p for p in by_path if len(p) == len(g) + 1 and p[:-1] == g]
            T += kids
            g = min(kids, key=rank.get)
        chosen = sorted(T, key=rank.get)[:N]
        got = O.beam_search_tree(ids, logq, ctx, table, -2.0, lam, bfac, N, 1, "fp64")
        _check(got, _as_rows(chosen, by_path, int(ctx[0, 1])), len(chosen))


def test_single_child_is_linear_drafting():
    rng = np.random.default_rng(9)
    L, k = 6, 4
    ids, logq, ctx, _ = _random_case(rng, L, k, 20, False)
    for W in (1, 3):
        for N in (3, 7, 50):
            got = O.beam_search_tree(ids, logq, ctx, None, -2.0, 0.0, 1, N, W, "fp64")
            n = min(N, L + 1)
            top1 = [int(ids[0, d, np.lexsort((ids[0, d], -logq[0, d]))[0]]) for d in range(L)]
            assert got["n_nodes"][0] == n
            assert got["token"][0, 1:n].tolist() == top1[: n - 1]
            assert got["parent"][0, :n].tolist() == list(range(-1, n - 1))


@pytest.mark.parametrize("W,bfac,L,N", [(2, 3, 3, 100), (2, 3, 3, 11), (1, 2, 5, 100),
                                        (4, 2, 4, 100), (3, 3, 2, 5)])
def test_tree_size_follows_the_closed_form(W, bfac, L, N):
    rng = np.random.default_rng(W * 100 + bfac * 10 + L)
    ids, logq, ctx, _ = _random_case(rng, L, bfac, 12, False)
    got = O.beam_search_tree(ids, logq, ctx, None, -2.0, 0.0, bfac, N, W, "fp64")
    size, beam = 1, 1
    for _ in range(L):
        if size >= N:
            break
        new = beam * bfac          # every beam node has b children
        size += new
        beam = min(W, new)
    assert got["n_nodes"][0] == min(N, size)


def test_eager_is_the_lazy_prefix_then_its_best_unexpanded_children():
    rng = np.random.default_rng(10)
    cases = 0
    for L in (2, 3, 4):
        for k in (2, 3):
            for with_table in (False, True):
                ids, logq, ctx, table = _random_case(rng, L, k, 6, with_table)
                lam = 0.3 if with_table else 0.0
                bfac = k
                nodes = O.candidate_tree_nodes(ids[0], logq[0], ctx[0], table, -2.0, lam, bfac,
                                               "fp32")
                order, by_path = _ranked(nodes)
                for N in (2, 4, 7, 15):
                    # expansions happen in the order R6 (the lazy pop order); stop once
                    # |T| = 1 + (children of the expanded nodes) reaches N
                    size, X = 1, 0
                    while size < N and X < len(order):
                        size += sum(1 for p in by_path if len(p) == len(order[X]) + 1
                                    and p[:-1] == order[X])
                        X += 1
                    expanded = set(order[:X])
                    T = {()} | {p for p in by_path if p and p[:-1] in expanded}
                    chosen = [p for p in order if p in T][:N]
                    got = O.eager_tree(ids, logq, ctx, table, -2.0, lam, bfac, N, "fp32")
                    _check(got, _as_rows(chosen, by_path, int(ctx[0, 1])), len(chosen))
                    cases += 1
    assert cases >= 40


def test_per_row_lambda_matches_enumeration_and_special_cases():
    """App. F: a lambda_d per position.  Best-first, beam and eager with a [B, L]
    lambda against exhaustive enumeration scored from scratch; a constant array
    equals the scalar; a zero row is prefix-blind at that depth."""
    rng = np.random.default_rng(11)
    for trial in range(30):
        L, k = 4, 3
        ids, logq, ctx, table = _random_case(rng, L, k, 6, True)
        lam_d = rng.choice([0.0, 0.125, 0.25, 0.5, 1.0], size=(1, L))
        N = int(rng.integers(2, 20))
        want = O.brute_force_tree(ids, logq, ctx, table, -2.0, lam_d, k, N, "fp32")
        got = O.best_first_tree(ids, logq, ctx, table, -2.0, lam_d, k, N, "fp32")
        for key in KEYS:
            np.testing.assert_array_equal(got[key], want[key], err_msg=key)
        const = np.full((1, L), 0.25)
        for fn, extra in ((O.best_first_tree, ()), (O.eager_tree, ()),
                          (O.beam_search_tree, (3,))):
            a = fn(ids, logq, ctx, table, -2.0, const, k, N, *extra)
            s = fn(ids, logq, ctx, table, -2.0, 0.25, k, N, *extra)
            for key in KEYS + ("score",):
                np.testing.assert_array_equal(a[key], s[key], err_msg=key)
    # a zero row: depth-1 scores are log q alone
    ids, logq, ctx, table = _random_case(rng, 3, 3, 6, True)
    lam_d = np.array([[0.0, 0.5, 0.5]])
    t = O.best_first_tree(ids, logq, ctx, table, -2.0, lam_d, 3, 4, "fp64")
    for i in range(1, int(t["n_nodes"][0])):
        if t["depth"][0, i] == 1:
            assert t["score"][0, i] == logq[0, 0, t["rank"][0, i]]
