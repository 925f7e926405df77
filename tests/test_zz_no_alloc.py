"""presto_score_build_tree_noalloc: the tree build for callers that cannot allocate
device memory (a plugin whose host framework owns every byte of the GPU, a C program
with no allocator, or a loop that must never block in cudaMalloc).  At large node
budgets the build keeps its selection scratch in global memory; this entry point
keeps it in a fixed device array inside the library instead of a caller workspace.

Called through the C ABI twice in a row on each input, it must give the same trees
(and masks and position ids) as the workspace entry point presto_score_build_tree_mask:
token, parent, depth, node count, mask and position ids bit-exact, and the float32
scores bitwise equal, as the other tree tests require.  Kept in its own file so
that it runs after every other test."""

import ctypes

import numpy as np
import pytest
import torch

import paper_2607_22634_gb300 as P
from paper_2607_22634_gb300 import _lib
from gpu_common import GPU, reachable_table, synthetic_candidates, to_dev

pytestmark = GPU

MISS = -12.0
LIMIT = 1 << 20  # PRESTO_BUILD_STATIC_SCRATCH_BYTES


def _inputs(seed, B, L, k, with_table):
    rng = np.random.default_rng(seed)
    vocab = rng.choice(200000, 400, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, 200000, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    ngram = None
    if with_table:
        a, bb, t, lr = reachable_table(rng, ids, ctx)
        ngram = P.Ngram3Table.from_entries(a, bb, t, lr, 18, MISS)
    return to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), ngram


def _outputs(B, N, dev="cuda"):
    W = (N + 31) // 32
    return {"token": torch.full((B, N), -7, dtype=torch.int32, device=dev),
            "parent": torch.full((B, N), -7, dtype=torch.int32, device=dev),
            "depth": torch.full((B, N), -7, dtype=torch.int32, device=dev),
            "score": torch.full((B, N), float("nan"), dtype=torch.float32, device=dev),
            "n_nodes": torch.full((B,), -7, dtype=torch.int32, device=dev),
            "mask": torch.full((B, N, W), -7, dtype=torch.int32, device=dev),
            "pos_ids": torch.full((B, N), -7, dtype=torch.int32, device=dev)}


def _noalloc(ids, logq, ctx, ngram, lam, N, policy, W, kv_len):
    """One call of presto_score_build_tree_noalloc through ctypes."""
    lib = P.load()
    B, L, k = ids.shape
    o = _outputs(B, N)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    desc = None if ngram is None else ctypes.byref(ngram.desc)
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = lib.presto_score_build_tree_noalloc(
        p(ids), p(logq), B, L, k, k, p(ctx), desc, ctypes.c_float(lam), None, policy, W, N,
        p(o["token"]), p(o["parent"]), p(o["depth"]), p(o["score"]), p(o["n_nodes"]),
        p(kv_len), p(o["mask"]), p(o["pos_ids"]), p(st),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    return rc, o, int(st.item())


CASES = [
    # B, L, k, N, table, policy, W: the selection scratch of two N = 1024 trees, the
    # child tables of four N = 512 trees (beam search), marginal-only scoring
    (2, 16, 8, 1024, True, P.SEARCH_BEST_FIRST, 1),
    (4, 16, 8, 512, True, P.SEARCH_BEAM, 10),
    (2, 32, 6, 1024, False, P.SEARCH_BEST_FIRST, 1),
]


@pytest.mark.parametrize("B,L,k,N,with_table,policy,W", CASES)
def test_noalloc_build_matches_workspace_entry_point(B, L, k, N, with_table, policy, W):
    # the shape really uses scratch outside shared memory, and it fits the array
    need = P.presto_build_workspace(B, L, k, N, W)
    assert 256 < need <= LIMIT
    ids, logq, ctx, ngram = _inputs(B * 31 + L + k + N, B, L, k, with_table)
    lam = 0.2 if with_table else 0.0
    kv = to_dev(np.arange(B) * 1000 + 17)
    ref = P.presto_score_build_tree(ids, logq, ctx, ngram, lam, N, policy=policy, beam_width=W,
                                    kv_len=kv)
    torch.cuda.synchronize()
    # an unrelated call (other seed and shape, the largest budget) first leaves the
    # shared array full of its own data; then two checked calls in a row, each on the
    # scratch the previous call left
    oi, ol, oc, og = _inputs(B * 131 + 7, 1, 24, 10, True)
    rc, _, st = _noalloc(oi, ol, oc, og, 0.3, 1024, P.SEARCH_BEST_FIRST, 1, to_dev([5]))
    assert rc == 0 and st == 0
    for _ in range(2):  # two calls in a row share the one scratch array
        rc, got, st = _noalloc(ids, logq, ctx, ngram, lam, N, policy, W, kv)
        assert rc == 0 and st == 0
        assert torch.equal(got["n_nodes"], ref["n_nodes"])
        assert int(got["n_nodes"].min()) > 256
        for key in ("mask", "pos_ids"):
            assert torch.equal(got[key], ref[key]), key
        for b in range(B):
            n = int(ref["n_nodes"][b])
            for key in ("token", "parent", "depth"):
                assert torch.equal(got[key][b, :n], ref[key][b, :n]), key
            assert torch.equal(got["score"][b, :n].view(torch.int32),
                               ref["score"][b, :n].view(torch.int32))


def test_noalloc_build_rejects_shapes_beyond_its_scratch():
    """Three N = 1024 trees need more scratch than the array holds: the call is
    refused on the host with PRESTO_ERR_UNSUPPORTED and nothing is written."""
    B, L, k, N = 3, 16, 8, 1024
    assert P.presto_build_workspace(B, L, k, N) > LIMIT
    ids, logq, ctx, ngram = _inputs(5, B, L, k, True)
    kv = to_dev(np.zeros(B))
    rc, got, st = _noalloc(ids, logq, ctx, ngram, 0.2, N, P.SEARCH_BEST_FIRST, 1, kv)
    assert rc == -2
    assert "limit" in _lib.load().presto_status_string(rc).decode()
    assert int(got["n_nodes"].max()) == -7 and st == 0
