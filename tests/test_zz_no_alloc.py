"""presto_topk_noalloc: the top-k entry point for callers that cannot allocate
device memory (for example a plugin whose host framework owns every byte of the
GPU, or a loop that must never block in cudaMalloc).  It keeps its scratch in a
fixed device array inside the library instead of a caller workspace.

Called through the C ABI twice in a row on each input, its results must match
the workspace entry point presto_topk within the top-k tolerances of the other
tests (ids exact; log q and lse within 1e-5 * max(1, |x|)).  Kept in its own file
so that it runs after every other test."""

import ctypes

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from gpu_common import GPU, rel_close

pytestmark = GPU


def _noalloc(lib, x, k):
    B, L, V = x.shape
    dtype = 0 if x.dtype == torch.float32 else 1
    ids = torch.full((B, L, k), -7, dtype=torch.int32, device=x.device)
    logq = torch.full((B, L, k), float("nan"), dtype=torch.float32, device=x.device)
    lse = torch.full((B, L), float("nan"), dtype=torch.float32, device=x.device)
    st = torch.zeros(1, dtype=torch.int32, device=x.device)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lib.presto_topk_noalloc(ctypes.c_void_p(x.data_ptr()), dtype, B, L, V, x.stride(1), k,
                                 ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(logq.data_ptr()),
                                 ctypes.c_void_p(lse.data_ptr()), ctypes.c_void_p(st.data_ptr()),
                                 stream)
    torch.cuda.synchronize()
    return rc, ids, logq, lse, int(st.item())


@pytest.mark.parametrize("name", ["tiny", "qwen3_8b", "self_spec", "qwen3_8b_4rows"])
def test_noalloc_topk_matches_workspace_entry_point(name):
    lib = P.load()
    if name == "qwen3_8b_4rows":   # few long rows: the shape whose spans merge in scratch
        w = synth.WORKLOADS["qwen3_8b"].scaled(L=4)
    else:
        w = synth.WORKLOADS[name]
    x = synth.drafter_logits(w).cuda()
    ref_ids, ref_logq, ref_lse = P.presto_topk(x, w.k)
    torch.cuda.synchronize()
    for _ in range(2):                       # two calls in a row share the scratch array
        rc, ids, logq, lse, st = _noalloc(lib, x, w.k)
        assert rc == 0 and st == 0
        assert torch.equal(ids, ref_ids)
        assert rel_close(logq.cpu().numpy(), ref_logq.cpu().numpy()) <= 1e-5
        assert rel_close(lse.cpu().numpy(), ref_lse.cpu().numpy()) <= 1e-5


def test_noalloc_widest_shape_fits_its_scratch():
    """The widest shape the ABI allows (near-2^18 float32 vocabulary, k = 16) needs
    no more scratch than the fixed array holds, and matches presto_topk."""
    lib = P.load()
    B, L, V, k = 1, 9, 262143, 16
    assert P.presto_topk_workspace(B, L, V, k) <= (1 << 14)
    g = torch.Generator().manual_seed(9)
    x = (torch.randn(B, L, V, generator=g) * 3).cuda()
    ref_ids, ref_logq, ref_lse = P.presto_topk(x, k)
    torch.cuda.synchronize()
    rc, ids, logq, lse, st = _noalloc(lib, x, k)
    assert rc == 0 and st == 0
    assert torch.equal(ids, ref_ids)
    assert rel_close(logq.cpu().numpy(), ref_logq.cpu().numpy()) <= 1e-5
    assert rel_close(lse.cpu().numpy(), ref_lse.cpu().numpy()) <= 1e-5
