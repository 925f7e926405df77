"""Pins of the oracle's tree search at the paper's large budgets (N = 512, 1024;
the budget sweep of Table 1 goes to 1024): best-first equals exhaustive
enumeration of a candidate tree with more than N nodes, in both precisions, and
the mask / acceptance steps keep their invariants at that size."""

import numpy as np
import pytest

from oracle import presto_oracle as O

KEYS = ("token", "parent", "depth", "n_nodes", "rank")


def _case(seed, L, k, V=40, quant=None):
    rng = np.random.default_rng(seed)
    ids = np.stack([rng.choice(V, k, replace=False) for _ in range(L)])[None]
    logq = -np.abs(rng.normal(0, 1.5, size=(1, L, k)))
    if quant:
        logq = -np.round(-logq * quant) / quant
    ctx = rng.integers(0, V, size=(1, 2))
    table = {}
    for _ in range(4 * V):
        key = tuple(int(v) for v in rng.integers(0, V, 3))
        table[key] = -float(rng.integers(0, 24)) / 8
    return ids, logq, ctx, table


@pytest.mark.parametrize("N", [512, 1024])
@pytest.mark.parametrize("prec", ["fp32", "fp64"])
def test_best_first_equals_enumeration_at_large_budgets(N, prec):
    # k = 4, L = 6: 5461 nodes in the candidate tree; quantised log q adds exact ties
    for seed, quant in ((1, None), (2, 4)):
        ids, logq, ctx, table = _case(seed, 6, 4, quant=quant)
        want = O.brute_force_tree(ids, logq, ctx, table, -3.0, 0.25, 4, N, prec)
        got = O.best_first_tree(ids, logq, ctx, table, -3.0, 0.25, 4, N, prec)
        assert int(got["n_nodes"][0]) == N
        for key in KEYS:
            np.testing.assert_array_equal(got[key], want[key], err_msg=key)


def test_mask_and_acceptance_invariants_at_1024_nodes():
    ids, logq, ctx, table = _case(3, 6, 4)
    t = O.best_first_tree(ids, logq, ctx, table, -3.0, 0.25, 4, 1024, "fp32")
    mask, pos = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], np.array([77]), 1024)
    dense = O.mask_to_dense(mask, 1024)[0]
    assert dense.shape == (1024, 1024)
    np.testing.assert_array_equal(dense.sum(axis=1), t["depth"][0] + 1)   # ancestors-or-self
    for i in range(1, 1024):
        p = int(t["parent"][0, i])
        assert np.all(dense[i] >= dense[p]) and dense[i, i]
    np.testing.assert_array_equal(pos[0], 77 + t["depth"][0])
    # the target follows the path of the last node: it is accepted, with its depth
    leaf = 1023
    path = []
    j = leaf
    while j > 0:
        path.append(j)
        j = int(t["parent"][0, j])
    target = np.full((1, 1024), -5)
    prev = 0
    for j in reversed(path):
        target[0, prev] = t["token"][0, j]
        prev = j
    acc, apath, bonus = O.accept(t["token"], t["parent"], t["n_nodes"], target, 6)
    assert acc[0] == t["depth"][0, leaf]
    assert list(apath[0][: acc[0] + 1]) == [0] + list(reversed(path))
