"""Pins for the oracle's tree attention (§5.1 tree-masked verification, App. C (I)).

Independent checks: torch's scaled_dot_product_attention on the CPU in float64
(a library routine) for the root-only case (plain decode attention), for a chain
(causal attention over prefix + chain) and for a general tree with an explicit
boolean mask; constant values; invariance under permuting the prefix keys; scipy's
logsumexp for the returned lse.
"""

import math

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

from oracle import presto_oracle as O


def _inputs(rng, B, N, Hq, Hkv, D, T, kv_len=None):
    r = lambda *s: rng.normal(size=s)
    kv_len = np.full(B, T) if kv_len is None else np.asarray(kv_len)
    return r(B, N, Hq, D), r(B, Hkv, T, D), r(B, Hkv, T, D), kv_len, r(B, N, Hkv, D), r(B, N, Hkv, D)


def _sdpa(q, k, v, mask=None):
    """q [n, D], k/v [m, D] float64 -> [n, D]."""
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))[None, None]
    m = None if mask is None else torch.from_numpy(mask)[None, None]
    return F.scaled_dot_product_attention(t(q), t(k), t(v), attn_mask=m)[0, 0].numpy()


def _tree(rng, N, L=6, k=3, V=50):
    ids = np.stack([rng.choice(V, k, replace=False) for _ in range(L)])[None]
    logq = -np.abs(rng.normal(0, 1.5, size=(1, L, k)))
    return O.best_first_tree(ids, logq, np.array([[1, 2]]), None, 0.0, 0.0, k, N, "fp64")


def test_root_only_is_decode_attention():
    rng = np.random.default_rng(0)
    q, kc, vc, kv, kt, vt = _inputs(rng, 2, 1, 8, 2, 16, 40, kv_len=[40, 17])
    mask = np.ones((2, 1, 1), np.uint32)
    out, lse = O.tree_attention(q, kc, vc, kv, kt, vt, mask, [1, 1])
    for b in range(2):
        T = kv[b]
        for h in range(8):
            g = h // 4
            K = np.concatenate([kc[b, g, :T], kt[b, :1, g]])
            Vv = np.concatenate([vc[b, g, :T], vt[b, :1, g]])
            np.testing.assert_allclose(out[b, 0, h], _sdpa(q[b, :1, h], K, Vv)[0], atol=1e-12)
            sc = q[b, 0, h] @ K.T / math.sqrt(16)
            assert lse[b, 0, h] == pytest.approx(scipy.special.logsumexp(sc), abs=1e-12)


def test_chain_is_causal_attention():
    rng = np.random.default_rng(1)
    N, T, D = 9, 30, 8
    q, kc, vc, kv, kt, vt = _inputs(rng, 1, N, 2, 1, D, T)
    parent = np.array([[-1] + list(range(N - 1))])
    mask, _ = O.tree_mask(parent, np.arange(N)[None], [N], kv, N)
    out, _ = O.tree_attention(q, kc, vc, kv, kt, vt, mask, [N])
    causal = np.tril(np.ones((N, N), bool))
    full = np.concatenate([np.ones((N, T), bool), causal], axis=1)
    for h in range(2):
        K = np.concatenate([kc[0, 0], kt[0, :, 0]])
        Vv = np.concatenate([vc[0, 0], vt[0, :, 0]])
        np.testing.assert_allclose(out[0, :, h], _sdpa(q[0, :, h], K, Vv, full), atol=1e-12)


def test_general_tree_matches_masked_sdpa_and_unused_rows_are_zero():
    rng = np.random.default_rng(2)
    N = 24
    t = _tree(rng, N)
    n = int(t["n_nodes"][0])
    q, kc, vc, kv, kt, vt = _inputs(rng, 1, N, 4, 2, 16, 33, kv_len=[21])
    mask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, N)
    # a tree with fewer nodes than the budget leaves unused slots
    n_used = [min(n, 19)]
    mask[0, n_used[0]:] = 0
    out, lse = O.tree_attention(q, kc, vc, kv, kt, vt, mask, n_used)
    dense = O.mask_to_dense(mask, N)[0]
    for h in range(4):
        g = h // 2
        K = np.concatenate([kc[0, g, :21], kt[0, : n_used[0], g]])
        Vv = np.concatenate([vc[0, g, :21], vt[0, : n_used[0], g]])
        m = np.concatenate([np.ones((n_used[0], 21), bool), dense[: n_used[0], : n_used[0]]], 1)
        np.testing.assert_allclose(out[0, : n_used[0], h], _sdpa(q[0, : n_used[0], h], K, Vv, m),
                                   atol=1e-12)
    assert not out[0, n_used[0]:].any() and np.all(np.isinf(lse[0, n_used[0]:]))


def test_constant_values_give_constant_output():
    rng = np.random.default_rng(3)
    q, kc, vc, kv, kt, vt = _inputs(rng, 1, 5, 2, 1, 8, 12)
    vc[:] = 0.75
    vt[:] = 0.75
    t = _tree(rng, 5)
    mask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, 5)
    out, _ = O.tree_attention(q, kc, vc, kv, kt, vt, mask, t["n_nodes"])
    n = int(t["n_nodes"][0])
    np.testing.assert_allclose(out[0, :n], 0.75, atol=1e-14)


def test_prefix_permutation_invariance():
    rng = np.random.default_rng(4)
    q, kc, vc, kv, kt, vt = _inputs(rng, 1, 6, 4, 2, 8, 50)
    t = _tree(rng, 6)
    mask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, 6)
    a, la = O.tree_attention(q, kc, vc, kv, kt, vt, mask, t["n_nodes"])
    perm = rng.permutation(50)
    b, lb = O.tree_attention(q, kc[:, :, perm], vc[:, :, perm], kv, kt, vt, mask, t["n_nodes"])
    np.testing.assert_allclose(a, b, atol=1e-12)
    np.testing.assert_allclose(la, lb, atol=1e-12)
