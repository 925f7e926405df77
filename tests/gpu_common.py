"""Helpers shared by the GPU parity tests: synthetic candidate sets, trigram tables,
tree comparisons.  Expected values always come from ``oracle``; the CUDA path's
outputs are only ever compared, never fed back into the oracle."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import presto_oracle as O

requires_gpu = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
GPU = [pytest.mark.gpu, requires_gpu]

LOGQ_TOL = 1e-5      # |gpu - oracle| <= LOGQ_TOL * max(1, |oracle|) for log q, lse, S
ATTN_TOL = 2e-2      # max abs error of bf16 attention output vs float64


def rel_close(got, want, tol=LOGQ_TOL):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    both_inf = np.isinf(got) & np.isinf(want) & (np.sign(got) == np.sign(want))
    err = np.where(both_inf, 0.0, np.abs(got - want) / np.maximum(1.0, np.abs(want)))
    return float(np.max(err)) if err.size else 0.0


def synthetic_candidates(rng, B, L, k, V, quant=None, vocab=None):
    """Distinct candidate tokens per row and log-probabilities <= 0 (not sorted)."""
    pool = np.arange(V) if vocab is None else np.asarray(vocab)
    ids = np.stack([np.stack([rng.choice(pool, k, replace=False) for _ in range(L)])
                    for _ in range(B)]).astype(np.int64)
    logq = -np.abs(rng.normal(0, 2.0, size=(B, L, k)))
    if quant:
        logq = -np.round(-logq * quant) / quant
    logq = logq.astype(np.float32).astype(np.float64)
    return ids, logq


def reachable_table(rng, ids, ctx, density=0.4, extra=2000, V=1 << 17):
    """A trigram table (a, b, t, logrho) covering part of the triples a tree over
    these candidates can query, plus random background triples."""
    B, L, k = ids.shape
    trip = set()
    for b in range(B):
        c0, c1 = int(ctx[b, 0]), int(ctx[b, 1])
        for d in range(L):
            for t in ids[b, d]:
                if d == 0:
                    cands = [(c0, c1)]
                elif d == 1:
                    cands = [(c1, int(x)) for x in ids[b, 0]]
                else:
                    cands = [(int(x), int(y)) for x in ids[b, d - 2] for y in ids[b, d - 1]]
                for (x, y) in cands:
                    if rng.random() < density:
                        trip.add((x, y, int(t)))
    for _ in range(extra):
        trip.add(tuple(int(v) for v in rng.integers(0, V, 3)))
    trip = sorted(trip)
    a = np.array([t[0] for t in trip], np.int64)
    bb = np.array([t[1] for t in trip], np.int64)
    t = np.array([t[2] for t in trip], np.int64)
    logrho = (-rng.integers(0, 64, len(trip)) / 8.0).astype(np.float32)
    return a, bb, t, logrho


def to_dev(x, dtype=torch.int32):
    return torch.as_tensor(np.ascontiguousarray(x)).to(dtype).cuda()


def tree_host(out):
    return {k: v.cpu().numpy() for k, v in out.items()}


def path_of(token, parent, i):
    p = []
    while i > 0:
        p.append(int(token[i]))
        i = int(parent[i])
    return tuple(reversed(p))


def assert_tree_exact(g, o, B):
    for b in range(B):
        n = int(o["n_nodes"][b])
        assert int(g["n_nodes"][b]) == n, (b, int(g["n_nodes"][b]), n)
        for key in ("token", "parent", "depth"):
            np.testing.assert_array_equal(g[key][b], o[key][b], err_msg=f"{key} seq {b}")
        np.testing.assert_array_equal(g["score"][b].astype(np.float32),
                                      o["score"][b].astype(np.float32), err_msg=f"score seq {b}")


def path_score64(ids_b, logq_b, ctx_b, table, miss, lam, path):
    """float64 S of a token path through the candidate sets (oracle functions)."""
    S = 0.0
    for d in range(1, len(path) + 1):
        j = int(np.nonzero(ids_b[d - 1] == path[d - 1])[0][0])
        rho = None
        if table is not None:
            rho = table.get(O.trigram_context(ctx_b, path[: d - 1]) + (path[d - 1],), miss)
        S += O.token_score(logq_b[d - 1, j], rho, O._lam_at(lam, d - 1), "fp64")
    return S


def assert_tree_close(g, ids, logq, ctx, table, miss, lam, N, tol=LOGQ_TOL):
    """GPU tree built from GPU log q vs the oracle's float64 tree from the oracle's
    log q.  Scores agree within tol; node sets agree except for near-ties at the
    budget boundary; when the oracle flags no near-tie the trees are identical."""
    o = O.best_first_tree(ids, logq, ctx, table, miss, lam, ids.shape[2], N, "fp64")
    B = ids.shape[0]
    for b in range(B):
        n = int(o["n_nodes"][b])
        assert int(g["n_nodes"][b]) == n
        gp = [path_of(g["token"][b], g["parent"][b], i) for i in range(n)]
        op = [path_of(o["token"][b], o["parent"][b], i) for i in range(n)]
        gS = [path_score64(ids[b], logq[b], ctx[b], table, miss, O._lam_of(lam, b), p) for p in gp]
        err = rel_close(g["score"][b][:n], gS)
        assert err <= tol, (b, err)
        assert all(gS[i + 1] <= gS[i] + tol * max(1, abs(gS[i])) for i in range(n - 1))
        edge = o["score64"][b][n - 1]
        band = tol * max(1.0, abs(edge))
        for p, s in zip(op, o["score64"][b][:n]):
            if s > edge + band:
                assert p in set(gp), (b, p)
        for p, s in zip(gp, gS):
            if s > edge + band:
                assert p in set(op), (b, p)
        if not O.competing_pairs(o, b, tol) and gp == op:
            np.testing.assert_array_equal(g["parent"][b][:n], o["parent"][b][:n])
