"""Pins for the oracle's tree mask / position ids (App. C (I), (IV)) and greedy
acceptance (§2.1, App. A, App. C (I)).

Independent checks: the App. C / Fig. 3 worked example (tests/golden), mask
ancestry invariants, the lower-triangular chain special case, the Obs. 1 coverage
bound (§3) with equality for an exhaustive tree, and linear-drafting acceptance.
"""

import json
import os

import numpy as np
import pytest

from oracle import presto_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))


def _random_tree(rng, L=5, k=3, V=40, N=30):
    ids = np.stack([rng.choice(V, k, replace=False) for _ in range(L)])[None]
    logq = -np.abs(rng.normal(0, 1.5, size=(1, L, k)))
    ctx = rng.integers(0, V, size=(1, 2))
    return ids, logq, ctx, O.best_first_tree(ids, logq, ctx, None, 0.0, 0.0, k, N, "fp64")


def test_mask_ancestry_invariants():
    rng = np.random.default_rng(0)
    for _ in range(10):
        _, _, _, t = _random_tree(rng, N=int(rng.integers(1, 70)))
        N = t["token"].shape[1]
        kv = np.array([int(rng.integers(0, 5000))])
        mask, pos = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, N)
        dense = O.mask_to_dense(mask, N)[0]
        n = int(t["n_nodes"][0])
        assert dense[0].tolist() == [True] + [False] * (N - 1)        # root row = {0}
        for i in range(n):
            assert dense[i].sum() == t["depth"][0, i] + 1              # popcount = depth + 1
            assert dense[i, i]
            assert not dense[i, i + 1:].any()                          # ancestors precede
            p = t["parent"][0, i]
            if p >= 0:
                assert np.all(dense[i] >= dense[p])                     # superset of parent's row
            assert pos[0, i] == kv[0] + t["depth"][0, i]
        assert not dense[n:].any() and np.all(pos[0, n:] == -1)


def test_chain_mask_is_lower_triangular():
    N = 37
    parent = np.array([[-1] + list(range(N - 1))])
    depth = np.arange(N)[None]
    mask, pos = O.tree_mask(parent, depth, [N], [100], N)
    dense = O.mask_to_dense(mask, N)[0]
    np.testing.assert_array_equal(dense, np.tril(np.ones((N, N), bool)))
    assert pos[0].tolist() == list(range(100, 100 + N))


def test_appc_fig3_worked_example():
    g = json.load(open(os.path.join(HERE, "golden", "appc_fig3_accept.json")))
    acc, path, bonus = O.accept(np.array([g["node_token"]]), np.array([g["node_parent"]]),
                                [len(g["node_token"])], np.array([g["target_token"]]), g["L"])
    assert int(acc[0]) == g["expected"]["accept_len"]
    assert path[0].tolist() == g["expected"]["accept_path"]
    assert int(bonus[0]) == g["expected"]["bonus"]


def _target_fn(seed, V):
    def f(path):
        h = hash((seed,) + tuple(path)) & 0xFFFFFFFF
        return int(np.random.default_rng(h).integers(0, V))
    return f


def test_accept_within_coverage_bound_and_equal_for_full_tree():
    rng = np.random.default_rng(3)
    hits = 0
    for trial in range(60):
        L, k, V = 4, 3, 5                 # small V: the target often hits candidates
        ids = np.stack([rng.choice(V, k, replace=False) for _ in range(L)])[None]
        logq = -np.abs(rng.normal(0, 1.5, size=(1, L, k)))
        ctx = rng.integers(0, V, size=(1, 2))
        f = _target_fn(trial, V)
        sets = [set(ids[0, d].tolist()) for d in range(L)]
        bound = O.coverage_bound(f, sets, L)
        full = sum(k ** d for d in range(L + 1))
        for N, exhaustive in ((7, False), (full, True)):
            t = O.best_first_tree(ids, logq, ctx, None, 0.0, 0.0, k, N, "fp64")
            n = int(t["n_nodes"][0])
            paths = [_path(t, i) for i in range(n)]
            tgt = np.full((1, N), -1)
            tgt[0, :n] = [f(p) for p in paths]
            acc, path, bonus = O.accept(t["token"], t["parent"], t["n_nodes"], tgt, L)
            assert acc[0] <= bound
            if exhaustive:
                assert acc[0] == bound
                hits += bound > 0
            deepest = path[0, acc[0]]
            assert t["depth"][0, deepest] == acc[0]
            assert bonus[0] == tgt[0, deepest]
            chain = path[0, : acc[0] + 1].tolist()
            assert chain[0] == 0 and all(path[0, acc[0] + 1:] == -1)
            assert all(t["parent"][0, chain[j]] == chain[j - 1] for j in range(1, len(chain)))
    assert hits > 10


def _path(t, i):
    out = []
    while i > 0:
        out.append(int(t["token"][0, i]))
        i = int(t["parent"][0, i])
    return tuple(reversed(out))


def test_linear_drafting_acceptance_counts_leading_matches():
    L = 6
    toks = [5, 6, 7, 8, 9, 10]
    parent = np.array([[-1, 0, 1, 2, 3, 4, 5]])
    node_token = np.array([[99] + toks])
    for agree in range(L + 1):
        # the target agrees with the chain for `agree` tokens, then diverges
        target = np.array([[toks[i] if i < agree else 1000 + i for i in range(L)] + [2000]])
        acc, path, bonus = O.accept(node_token, parent, [L + 1], target, L)
        assert acc[0] == agree
        assert path[0, : agree + 1].tolist() == list(range(agree + 1))
        assert bonus[0] == target[0, agree]


def test_accept_rejects_bad_parent():
    with pytest.raises(ValueError):
        O.accept(np.array([[1, 2]]), np.array([[-1, 5]]), [2], np.array([[2, 3]]), 3)
