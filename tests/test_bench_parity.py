"""bench.py's parity check of the benched round (oracle_check), on the CPU: given the
oracle's own round on the Qwen3-8B-shaped workload's inputs, as the GPU arm hands it
over (candidates, tree, mask as 32-bit words, attention inputs and output), every
check passes; a planted mistake in the mask or in the attention output fails its
check."""

import os
import tempfile

import numpy as np
import pytest

import bench
import synth


@pytest.fixture(scope="module")
def round0():
    w = synth.WORKLOADS["qwen3_8b"]
    inp = bench.oracle_inputs(w, attn_f64=True)
    res = bench.oracle_round(w, inp)
    att = synth.attention_inputs(w, device="cpu")
    g = {"ids": res["ids"], "logq": res["logq"].astype(np.float32),
         "mask": res["mask"].view(np.int32),  # as a torch int32 tensor arrives
         "pos_ids": res["pos"], "attn": res["attn"], "accept_len": res["accept_len"],
         "accept_path": res["accept_path"], "bonus": res["bonus"], "target": inp["target"],
         "kv_len": np.asarray(inp["kv_len"], np.int32),
         "token": res["token"], "parent": res["parent"], "depth": res["depth"],
         "score": np.asarray(res["score"], np.float32), "n_nodes": res["n_nodes"]}
    g.update({k: att[k].float().numpy() for k in ("q", "k_cache", "v_cache", "k_tree", "v_tree")})
    return w, g


def _check(w, g):
    fd, path = tempfile.mkstemp(suffix=".npz")
    os.close(fd)
    try:
        np.savez(path, **g)
        return bench.oracle_check(w, path)
    finally:
        os.unlink(path)


def test_oracle_round_passes_every_check(round0):
    w, g = round0
    c = _check(w, g)
    assert c["tree"] and c["tree_scores_equal"] and c["mask"] and c["pos_ids"] and c["accept"]
    assert c["attention_max_abs"] <= 1e-12


def test_planted_mask_bit_fails(round0):
    w, g = round0
    bad = dict(g)
    m = g["mask"].view(np.uint32).copy()
    n = int(g["n_nodes"][0])
    m[0, n - 1, 0] ^= np.uint32(1 << 31)  # a word's sign bit
    bad["mask"] = m.view(np.int32)
    c = _check(w, bad)
    assert not c["mask"] and c["mask_rows_differ"] == 1


def test_planted_attention_error_fails(round0):
    w, g = round0
    bad = dict(g)
    a = g["attn"].copy()
    a[0, 3, 5, 7] += 0.05
    bad["attn"] = a
    c = _check(w, bad)
    assert c["attention_max_abs"] == pytest.approx(0.05, rel=1e-9)
