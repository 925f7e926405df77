"""presto_tree_attention (tcgen05 kernel, C ABI) vs the float64 oracle: bf16
output within 2e-2 max abs, lse within 2e-3.  Covers both head dims, GQA ratios,
ragged and empty prefixes, root-only and chain trees, trees smaller than the
budget, split-KV and single-split launches, and the full-size workloads on a
seeded sample of (sequence, kv head) pairs."""

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import ATTN_TOL, GPU, synthetic_candidates, to_dev

pytestmark = GPU


def _tree(seed, B, N, L=8, k=4, n_used=None):
    rng = np.random.default_rng(seed)
    ids, logq = synthetic_candidates(rng, B, L, k, 1000)
    t = O.best_first_tree(ids, logq, rng.integers(0, 1000, size=(B, 2)), None, 0.0, 0.0, k, N,
                          "fp64")
    if n_used is not None:
        for b in range(B):
            n = min(int(t["n_nodes"][b]), n_used[b])
            t["n_nodes"][b] = n
            for key in ("token", "parent", "depth"):
                t[key][b, n:] = -1
    return t


def _inputs(B, N, Hq, Hkv, D, T, kv_len, seed, device="cuda"):
    g = torch.Generator(device=device).manual_seed(seed)
    rn = lambda *s: torch.randn(*s, generator=g, device=device).to(torch.bfloat16)
    return dict(q=rn(B, N, Hq, D), k_cache=rn(B, Hkv, T, D), v_cache=rn(B, Hkv, T, D),
                k_tree=rn(B, N, Hkv, D), v_tree=rn(B, N, Hkv, D),
                kv_len=torch.as_tensor(kv_len, dtype=torch.int32, device=device))


def _np(t):
    return t.float().cpu().double().numpy()


def _run_and_check(inp, t, N, seqs=None, kv_heads=None, tol=ATTN_TOL):
    B = inp["q"].shape[0]
    omask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], inp["kv_len"].cpu().numpy(), N)
    mask = to_dev(omask.view(np.int32))
    n_nodes = to_dev(t["n_nodes"])
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out, lse = P.presto_tree_attention(inp["q"], inp["k_cache"], inp["v_cache"], inp["kv_len"],
                                       inp["k_tree"], inp["v_tree"], mask, n_nodes, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    Hkv = inp["k_cache"].shape[1]
    G = inp["q"].shape[2] // Hkv
    seqs = range(B) if seqs is None else seqs
    kv_heads = range(Hkv) if kv_heads is None else kv_heads
    sl = lambda x, b: x[b:b + 1]
    for b in seqs:
        oo, ol = O.tree_attention(_np(sl(inp["q"], b)), _np(sl(inp["k_cache"], b)),
                                  _np(sl(inp["v_cache"], b)), inp["kv_len"][b:b + 1].cpu().numpy(),
                                  _np(sl(inp["k_tree"], b)), _np(sl(inp["v_tree"], b)),
                                  omask[b:b + 1], t["n_nodes"][b:b + 1], kv_heads=list(kv_heads))
        heads = [g * G + h for g in kv_heads for h in range(G)]
        got = out[b].float().cpu().numpy()[:, heads]
        err = np.max(np.abs(got - oo[0][:, heads]))
        assert err <= tol, (b, err)
        gl = lse[b].cpu().numpy()[:, heads]
        wl = ol[0][:, heads]
        fin = np.isfinite(wl)
        assert np.array_equal(np.isfinite(gl), fin)
        if fin.any():
            assert np.max(np.abs(gl[fin] - wl[fin])) <= 2e-3


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("Hq,Hkv", [(4, 1), (32, 8), (8, 8), (16, 2)])
def test_attention_small(D, Hq, Hkv):
    B, N, T = 2, 24, 300
    t = _tree(D + Hq, B, N, n_used=[24, 17])
    inp = _inputs(B, N, Hq, Hkv, D, T, [300, 129], seed=D * Hq)
    _run_and_check(inp, t, N)


def test_attention_tiny_workload():
    w = synth.WORKLOADS["tiny"]
    inp = synth.attention_inputs(w, device="cuda")
    t = _tree(1, w.B, w.N)
    _run_and_check(inp, t, w.N)


@pytest.mark.parametrize("kv", [[0, 1], [127, 128], [129, 255], [256, 4]])
def test_attention_ragged_and_empty_prefix(kv):
    B, N = 2, 40
    t = _tree(sum(kv), B, N)
    inp = _inputs(B, N, 8, 2, 128, 256, kv, seed=sum(kv) + 1)
    _run_and_check(inp, t, N)


def test_attention_root_only_and_chain():
    B, N = 1, 1
    t = _tree(3, B, N)
    inp = _inputs(B, N, 32, 8, 128, 1000, [1000], seed=3)
    _run_and_check(inp, t, N)
    # chain: k = 1 gives a lower-triangular tree mask
    N = 20
    t = _tree(4, 1, N, L=30, k=1)
    inp = _inputs(1, N, 32, 8, 128, 513, [513], seed=4)
    _run_and_check(inp, t, N)


def test_attention_two_tree_tiles():
    """N = 256: the tree keys span two 128-key tiles."""
    B, N = 1, 256
    t = _tree(5, B, N, L=16, k=6)
    inp = _inputs(B, N, 8, 8, 64, 700, [650], seed=5)
    _run_and_check(inp, t, N)


def test_attention_qwen3_8b_round_full():
    w = synth.WORKLOADS["qwen3_8b"]
    inp = synth.attention_inputs(w, device="cuda")
    t = _tree(6, w.B, w.N, L=w.L, k=w.k)
    _run_and_check(inp, t, w.N)


def test_attention_launch_count():
    """presto_attn_launches: the Qwen3-8B-shaped call splits its KV range over plain CTAs
    and merges them in a second kernel; self_spec takes the long-run schedule (one
    kernel, splits merged inside its clusters); refused shapes launch nothing."""
    q = synth.WORKLOADS["qwen3_8b"]
    assert P.presto_attn_launches(q.B, q.N, q.Hq, q.Hkv, q.D, q.T) == 2
    s = synth.WORKLOADS["self_spec"]
    assert P.presto_attn_launches(s.B, s.N, s.Hq, s.Hkv, s.D, s.T) == 1
    assert P.presto_attn_launches(1, 8, 4, 1, 128, 16) == 1  # one KV tile: no split
    assert P.presto_attn_launches(1, 8, 6, 4, 128, 16) == 0  # Hq not a multiple of Hkv
    assert P.presto_attn_launches(1, 8, 4, 1, 96, 16) == 0   # unsupported D


def test_attention_batched_ragged_sampled():
    w = synth.WORKLOADS["batched_ragged"]
    inp = synth.attention_inputs(w, device="cuda")
    t = _tree(7, w.B, w.N, L=w.L, k=w.k)
    _run_and_check(inp, t, w.N, seqs=[0, 9], kv_heads=[0, 5])


def test_attention_self_spec_sampled():
    w = synth.WORKLOADS["self_spec"]
    inp = synth.attention_inputs(w, device="cuda")
    t = _tree(8, w.B, w.N, L=w.L, k=w.k)
    _run_and_check(inp, t, w.N, seqs=[3], kv_heads=[2])


def test_attention_long_ctx_layer_sampled():
    w = synth.WORKLOADS["long_ctx"]
    inp = synth.attention_inputs(w, layer=17, device="cuda")
    t = _tree(9, w.B, w.N, L=w.L, k=w.k)
    _run_and_check(inp, t, w.N, seqs=[5], kv_heads=[7])


def test_attention_long_run_d64():
    """D = 64 with many (sequence, kv head) pairs and long prefixes: one KV split per
    row block, 17 KV tiles per CTA (the long-run schedule); ragged prefix lengths."""
    B, N, Hq, Hkv, T = 16, 64, 32, 8, 2048
    t = _tree(11, B, N, L=12, k=6)
    kv = [2048 - 61 * b for b in range(B)]
    inp = _inputs(B, N, Hq, Hkv, 64, T, kv, seed=11)
    _run_and_check(inp, t, N, seqs=[0, 7, 15], kv_heads=[0, 3, 7])


def test_attention_kv_len_above_capacity_is_reported():
    B, N = 1, 8
    t = _tree(10, B, N)
    inp = _inputs(B, N, 8, 2, 64, 128, [500], seed=10)
    omask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], [128], N)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_tree_attention(inp["q"], inp["k_cache"], inp["v_cache"], inp["kv_len"], inp["k_tree"],
                            inp["v_tree"], to_dev(omask.view(np.int32)), to_dev(t["n_nodes"]),
                            dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x4


@pytest.mark.parametrize("D,T,kv", [(128, 700, [650]), (128, 4096, [4096]), (64, 300, [0])])
def test_attention_large_tree_budgets(D, T, kv):
    """N = 1024 (and 512 for D = 64): up to eight tree-key tiles, dealt out to the KV
    splits together with the prefix tiles; an empty prefix leaves only tree keys."""
    B = 1
    N = 1024 if D == 128 else 512
    t = _tree(9 + T, B, N, L=16, k=8)
    inp = _inputs(B, N, 32, 8, D, T, kv, seed=9 + T)
    _run_and_check(inp, t, N, kv_heads=[0, 5])
