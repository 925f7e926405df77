#!/usr/bin/env python
"""Benchmark of one PRESTO draft-and-verify round on GB300.

A step is one round of the whole hot path on one batch of synthetic input:
presto_topk -> presto_score_build_tree -> presto_tree_mask ->
presto_tree_attention (per layer) -> presto_accept, replayed from a CUDA graph.
The default workload is the Qwen3-8B-shaped dedicated-drafter round (B=1, L=16,
V=151936, k=8, N=64, GQA 32/8, D=128, T=4096, one attention layer).

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle instead.
Multi-GPU (torchrun): independent replicas, no collective on the data path.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tree draft+verify steps/s at Qwen3-8B shapes; top-k HBM % & tree-attn TC % peak"
L2_BYTES = 129 * 1024 * 1024
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20000)
    p.add_argument("--warmup", type=int, default=50)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="qwen3_8b")
    p.add_argument("--no-graph", action="store_true")
    p.add_argument("--kernel-steps", type=int, default=20,
                   help="graph replays (each n_sets launches) of the per-call timing pass")
    p.add_argument("--e2e-steps", type=int, default=2000)
    p.add_argument("--cpu-seconds", type=float, default=15.0)
    p.add_argument("--repeats", type=int, default=5,
                   help="timed regions of --steps rounds each (at least)")
    p.add_argument("--repeat-seconds", type=float, default=1.0,
                   help="keep repeating the timed region for at least this long")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-variants", action="store_true",
                   help="skip timing the search policies, adaptive lambda and slot top-k")
    p.add_argument("--oracle-worker", action="store_true", help=argparse.SUPPRESS)
    p.add_argument("--oracle-mode", choices=["round", "mp", "subset", "check"], default="round",
                   help=argparse.SUPPRESS)
    p.add_argument("--check-in", default=None, help=argparse.SUPPRESS)
    p.add_argument("--parity-out", default=None, help=argparse.SUPPRESS)
    return p.parse_args(argv)


def workload_desc(w):
    return (f"{w.name}: B={w.B} L={w.L} V={w.V} k={w.k} N={w.N} lambda={w.lam} "
            f"table={'trigram' if w.use_table else 'none'} GQA {w.Hq}/{w.Hkv} D={w.D} "
            f"T={w.T_min}..{w.T} layers={w.layers} logits={w.logits_dtype}")


# ---------------------------------------------------------------- CPU oracle
# The oracle runs only here: in the cpu_baseline leg of the GPU arm and in the
# reference arm, always in a subprocess that sees no GPU.

# workloads whose attention the oracle times on a subset of (sequence, kv head)
# pairs, scaled to the whole round by flops
ATTN_SUBSET = {"batched_ragged": ([0, 1], [0]), "long_ctx": ([0], [0])}


def oracle_inputs(w, attn_f64=True):
    """Set 0 of the workload (the GPU arm's input set 0) for the oracle: logits,
    context, table, the tree's target tokens, one attention layer (float64, or
    float32 arrays the oracle converts slice by slice when attn_f64 is False)."""
    import numpy as np
    import synth
    from oracle import presto_oracle as O
    logits = synth.drafter_logits(w)
    a, b, t, lr = synth.trigram_entries(w)
    att = synth.attention_inputs(w, device="cpu")
    conv = (lambda x: x.double().numpy()) if attn_f64 else (lambda x: x.float().numpy())
    ids, logq, _ = O.topk_logsoftmax(logits.reshape(w.rows, w.V).double().numpy(), w.k)
    table = O.make_table(a, b, t, lr) if w.use_table else None
    ctx = synth.ctx_tokens(w).numpy()
    tree = O.best_first_tree(ids.reshape(w.B, w.L, w.k), logq.reshape(w.B, w.L, w.k), ctx, table,
                             w.miss_logrho, w.lam, w.branching, w.N, "fp32")
    target = synth.target_tokens(w, logits, tree["token"], tree["parent"], tree["n_nodes"]).numpy()
    layer = {k: conv(v) for k, v in att.items() if k != "kv_len"}
    layer["q"] = att["q"].double().numpy()
    return {"logits": logits.reshape(w.rows, w.V).double().numpy(), "ctx": ctx, "table": table,
            "kv_len": att["kv_len"].numpy(), "layer": layer, "target": target,
            "n_entries": int(np.size(a))}


def oracle_round(w, inp, seqs=None, kv_heads=None, clock=None, n_layers=None):
    """One draft-and-verify round with the CPU oracle (float64; the tree search in
    float32, as the kernels take its decisions).  Attention runs on every layer (or
    n_layers of them), or on the (seqs, kv_heads) subset of each.  `clock`
    (optional dict) collects the seconds of each step."""
    import time as _t
    from oracle import presto_oracle as O
    t0 = _t.perf_counter()
    ids, logq, lse = O.topk_logsoftmax(inp["logits"], w.k)
    t1 = _t.perf_counter()
    ids3, logq3 = ids.reshape(w.B, w.L, w.k), logq.reshape(w.B, w.L, w.k)
    tree = O.best_first_tree(ids3, logq3, inp["ctx"], inp["table"], w.miss_logrho, w.lam,
                             w.branching, w.N, "fp32")
    mask, pos = O.tree_mask(tree["parent"], tree["depth"], tree["n_nodes"], inp["kv_len"], w.N)
    t2 = _t.perf_counter()
    lay = inp["layer"]
    out = None
    for _ in range(w.layers if n_layers is None else n_layers):
        out, _ = O.tree_attention(lay["q"], lay["k_cache"], lay["v_cache"], inp["kv_len"],
                                  lay["k_tree"], lay["v_tree"], mask, tree["n_nodes"],
                                  seqs=seqs, kv_heads=kv_heads)
    t3 = _t.perf_counter()
    acc, path, bonus = O.accept(tree["token"], tree["parent"], tree["n_nodes"], inp["target"], w.L)
    t4 = _t.perf_counter()
    if clock is not None:
        for key, dt in (("topk", t1 - t0), ("build_mask", t2 - t1), ("attention", t3 - t2),
                        ("accept", t4 - t3)):
            clock[key] = clock.get(key, 0.0) + dt
    return {"ids": ids, "logq": logq, "lse": lse, "token": tree["token"],
            "parent": tree["parent"], "depth": tree["depth"], "score": tree["score"],
            "n_nodes": tree["n_nodes"], "mask": mask, "pos": pos, "attn": out,
            "accept_len": acc, "accept_path": path, "bonus": bonus}


def attention_flops(w, kv_len, n_nodes, mask, seqs=None, kv_heads=None):
    """4 Hq' D sum_b sum_i (T_b + |anc(i)|) over the sequences and kv heads given
    (all by default), Hq' = the query heads of those kv heads; one layer."""
    import numpy as np
    G = w.Hq // w.Hkv
    heads = (w.Hkv if kv_heads is None else len(kv_heads)) * G
    total = 0
    for b in (range(w.B) if seqs is None else seqs):
        n = int(n_nodes[b])
        anc = int(np.unpackbits(np.asarray(mask[b, :n], np.uint32).view(np.uint8)).sum())
        total += int(kv_len[b]) * n + anc
    return 4.0 * heads * w.D * total


# -- multi-process oracle: one process per host core, each holding the inputs
_MP = {}


def _mp_init(workload):
    import synth
    w = synth.WORKLOADS[workload]
    _MP["w"] = w
    _MP["inp"] = oracle_inputs(w)


def _mp_topk(rows):
    from oracle import presto_oracle as O
    return O.topk_logsoftmax(_MP["inp"]["logits"][rows[0]:rows[1]], _MP["w"].k)


def _mp_tree(args):
    from oracle import presto_oracle as O
    w, inp = _MP["w"], _MP["inp"]
    b, ids_b, logq_b = args
    return O.best_first_tree(ids_b, logq_b, inp["ctx"][b:b + 1], inp["table"], w.miss_logrho,
                             w.lam, w.branching, w.N, "fp32")


def _mp_attn(args):
    from oracle import presto_oracle as O
    w, inp = _MP["w"], _MP["inp"]
    b, g, mask, n_nodes = args
    lay = inp["layer"]
    G = w.Hq // w.Hkv
    out, _ = O.tree_attention(lay["q"], lay["k_cache"], lay["v_cache"], inp["kv_len"],
                              lay["k_tree"], lay["v_tree"], mask, n_nodes, seqs=[b], kv_heads=[g])
    return out[b, :, g * G:(g + 1) * G]


def oracle_round_mp(w, inp, pool, procs):
    """oracle_round with its independent pieces spread over a process pool: top-k
    rows, one tree per sequence, attention per (sequence, kv head); the mask and
    the acceptance (microseconds) stay in the parent."""
    import numpy as np
    from oracle import presto_oracle as O
    R = w.rows
    cuts = [(R * i // procs, R * (i + 1) // procs) for i in range(procs)]
    parts = pool.map(_mp_topk, [c for c in cuts if c[1] > c[0]])
    ids = np.concatenate([p[0] for p in parts]).reshape(w.B, w.L, w.k)
    logq = np.concatenate([p[1] for p in parts]).reshape(w.B, w.L, w.k)
    trees = pool.map(_mp_tree, [(b, ids[b:b + 1], logq[b:b + 1]) for b in range(w.B)])
    tree = {key: np.concatenate([t[key] for t in trees]) for key in trees[0]}
    mask, _ = O.tree_mask(tree["parent"], tree["depth"], tree["n_nodes"], inp["kv_len"], w.N)
    for _ in range(w.layers):
        pool.map(_mp_attn, [(b, g, mask, tree["n_nodes"]) for b in range(w.B)
                            for g in range(w.Hkv)])
    O.accept(tree["token"], tree["parent"], tree["n_nodes"], inp["target"], w.L)


def oracle_worker(args):
    """Runs in a fresh process with one BLAS thread and no GPU.  Modes:
    round  full rounds on one thread (and, with --parity-out, input set 0's round
           results saved for the GPU arm to compare with);
    mp     full rounds with one process per host core;
    subset the round's steps on one thread, attention on ATTN_SUBSET's pairs,
           scaled to the whole round (all layers) by flops."""
    import synth
    w = synth.WORKLOADS[args.workload]
    budget = args.cpu_seconds
    mode = args.oracle_mode
    if mode == "check":
        print(json.dumps(oracle_check(w, args.check_in)))
        return
    if mode == "subset":
        seqs, heads = ATTN_SUBSET[args.workload]
        inp = oracle_inputs(w, attn_f64=False)
        clock = {}
        res = oracle_round(w, inp, seqs=seqs, kv_heads=heads, clock=clock, n_layers=1)
        full = attention_flops(w, inp["kv_len"], res["n_nodes"], res["mask"]) * w.layers
        sub = attention_flops(w, inp["kv_len"], res["n_nodes"], res["mask"], seqs, heads)
        attn_s = clock["attention"] * full / sub
        secs = clock["topk"] + clock["build_mask"] + attn_s + clock["accept"]
        print(json.dumps({"seconds_per_round": secs, "steps": clock,
                          "attention_scaled_seconds": attn_s, "attention_scale": full / sub,
                          "subset": {"seqs": seqs, "kv_heads": heads}}))
        return
    inp = oracle_inputs(w)
    pool, procs = None, 1
    if mode == "mp":
        import multiprocessing as mp
        procs = max(1, os.cpu_count() or 1)
        pool = mp.get_context("spawn").Pool(procs, initializer=_mp_init, initargs=(args.workload,))
        step = lambda: oracle_round_mp(w, inp, pool, procs)
    else:
        step = lambda: oracle_round(w, inp)
    t0 = time.perf_counter()
    for _ in range(max(1, args.warmup)):          # warm-up rounds, untimed
        step()
    first = time.perf_counter() - t0
    n, t_start = 0, time.perf_counter()
    while n < max(1, args.steps) and (n == 0 or time.perf_counter() - t_start < budget):
        step()
        n += 1
    dt = time.perf_counter() - t_start
    if pool is not None:
        pool.close()
        pool.join()
    if args.parity_out:
        import numpy as np
        np.savez(args.parity_out, **oracle_round(w, inp))
    print(json.dumps({"rounds": n, "seconds": dt, "warmup_seconds": first,
                      "warmup": max(1, args.warmup), "procs": procs}))


def oracle_check(w, gpu_file):
    """Each step of the GPU's round on input set 0 against the oracle applied to that
    step's inputs as the GPU had them (so floating-point near-ties upstream cannot
    make later steps differ): the tree from the GPU's candidates, the mask and
    position ids from the GPU's tree, attention with the GPU's mask, acceptance on
    the GPU's tree with its target tokens.  Exact, except scores (1e-5 relative) and
    attention (2e-2 max abs)."""
    import numpy as np
    import synth
    from oracle import presto_oracle as O
    g = dict(np.load(gpu_file))
    g["mask"] = np.ascontiguousarray(g["mask"]).view(np.uint32)  # 32-bit words, unsigned
    a, b, t, lr = synth.trigram_entries(w)
    table = O.make_table(a, b, t, lr) if w.use_table else None
    ctx = synth.ctx_tokens(w).numpy()
    ids = g["ids"].astype(np.int64).reshape(w.B, w.L, w.k)
    logq = g["logq"].astype(np.float64).reshape(w.B, w.L, w.k)
    tree = O.best_first_tree(ids, logq, ctx, table, w.miss_logrho, w.lam, w.branching, w.N, "fp32")
    c = {}
    c["tree"] = bool(all(np.array_equal(tree[k], g[k]) for k in ("token", "parent", "depth",
                                                                  "n_nodes")))
    c["tree_scores_equal"] = bool(np.array_equal(np.asarray(tree["score"], np.float32),
                                                 g["score"].astype(np.float32)))
    mask, pos = O.tree_mask(g["parent"], g["depth"], g["n_nodes"], g["kv_len"], w.N)
    c["mask"] = bool(np.array_equal(mask, g["mask"]))
    if not c["mask"]:
        bad = np.argwhere((mask != g["mask"]).any(axis=2))
        b0, i0 = (int(bad[0][0]), int(bad[0][1])) if len(bad) else (0, 0)
        c["mask_rows_differ"] = int(len(bad))
        c["mask_first_diff"] = {"seq": b0, "node": i0, "gpu": g["mask"][b0, i0].tolist(),
                                "oracle": mask[b0, i0].tolist(),
                                "shapes": [list(mask.shape), list(g["mask"].shape)]}
    c["pos_ids"] = bool(np.array_equal(pos, g["pos_ids"]))
    if w.layers == 1:
        # the layer's Q / K / V exactly as the GPU read them (bf16 widened to float32)
        f64 = lambda x: np.asarray(x, np.float64)
        out, _ = O.tree_attention(f64(g["q"]), f64(g["k_cache"]), f64(g["v_cache"]),
                                  g["kv_len"], f64(g["k_tree"]), f64(g["v_tree"]),
                                  g["mask"], g["n_nodes"])
        c["attention_max_abs"] = float(np.abs(out - g["attn"]).max())
    else:
        c["attention_max_abs"] = None  # the GPU output is the last layer's; checked in tests
    acc, path, bonus = O.accept(g["token"], g["parent"], g["n_nodes"], g["target"], w.L)
    c["accept"] = bool(np.array_equal(acc, g["accept_len"]) and np.array_equal(path, g["accept_path"])
                       and np.array_equal(bonus, g["bonus"]))
    return c


def run_oracle(workload, seconds, max_steps, warmup=1, mode="round", parity_out=None,
               check_in=None):
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "NUMEXPR_NUM_THREADS"):
        env[v] = "1"
    env["CUDA_VISIBLE_DEVICES"] = ""
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-worker", "--workload", workload,
           "--cpu-seconds", str(seconds), "--steps", str(max_steps), "--warmup", str(warmup),
           "--oracle-mode", mode]
    if parity_out:
        cmd += ["--parity-out", parity_out]
    if check_in:
        cmd += ["--check-in", check_in]
    r = subprocess.run(cmd, capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError("oracle worker failed:\n" + r.stderr[-3000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


def bench_config(w, world):
    """The `config` both arms print (so the driver sees the same workload)."""
    return {"workload": workload_desc(w), "parallelism": "replicas" if world > 1 else "1 GPU"}


def run_reference(args):
    import synth
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    w = synth.WORKLOADS[args.workload]
    res = run_oracle(args.workload, seconds=min(60.0, max(10.0, 2.0 * args.steps)),
                     max_steps=args.steps, warmup=args.warmup, mode="mp")
    value = res["rounds"] / res["seconds"]
    sample = (f"{res['rounds']} full oracle rounds of {args.steps} requested (float64 numpy; "
              f"top-k rows, trees and attention (sequence, kv head) pairs spread over "
              f"{res['procs']} processes, one per host core): {workload_desc(w)}")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s",
        "n_gpus": args.gpus, "steps": res["rounds"], "warmup": res["warmup"],
        "ms_per_step": 1e3 / value, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": bench_config(w, world),
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": res["procs"],
                         "host_cores": os.cpu_count(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


# ---------------------------------------------------------------- GPU path

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons around a region."""

    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.out = ""

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu_id)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self, t_start, t_end):
        import datetime
        mhz, max_mhz, reasons = [], None, set()
        for line in self.out.strip().splitlines():
            r = [x.strip() for x in line.split(",")]
            if len(r) < 9:
                continue
            try:
                ts = datetime.datetime.strptime(r[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                clk, mx = float(r[1]), float(r[2])
            except ValueError:
                continue
            if not (t_start - 0.05 <= ts <= t_end + 0.05):
                continue
            mhz.append(clk)
            max_mhz = mx
            for name, val in zip(self.NAMES, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(mhz) if mhz else None, "sm_max_mhz": max_mhz,
                "reasons": sorted(reasons), "samples": len(mhz)}


def gpu_smi_id(dev):
    """Identifier nvidia-smi -i accepts for this torch device (its UUID)."""
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
        return vis.split(",")[dev.index].strip() if vis else str(dev.index)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def source_digest(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2607_22634_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel):
    """DRAM bytes per launch from the committed ncu summary, if the kernel's
    source has not changed since the capture (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f).get(kernel)
    if not rec or rec.get("source_digest") != source_digest(rec["sources"]):
        return None
    return rec.get("dram_bytes_per_launch")


def time_variants(args, P, w, step, sets, side, ngram):
    import torch
    import synth
    dev = step.device
    B, L, k, N = w.B, w.L, w.k, w.N
    f32, i32 = torch.float32, torch.int32
    lam_d = torch.full((B, L), w.lam, dtype=f32, device=dev)
    ent = torch.empty(B, L, dtype=f32, device=dev)
    lam_out = torch.empty(B, L, dtype=f32, device=dev)
    ws_b = torch.empty(max(P.presto_build_workspace(B, L, k, N, 10), 256), dtype=torch.uint8,
                       device=dev)
    tree = {key: torch.empty_like(v) for key, v in step.tree.items()}
    # slot logits of every node of the tree: [B, N, L + 1, V]; set s accepts node
    # 1 + s (mod N - 1) of every sequence, so each launch reads other rows
    esz = sets[0]["logits"].element_size()
    slots = None
    if B * N * (L + 1) * w.V * esz <= (4 << 30):
        g = torch.Generator(device=dev)
        g.manual_seed(w.seed + 77)
        slots = torch.randn(B, N, L + 1, w.V, generator=g, device=dev).to(sets[0]["logits"].dtype)
        acc_len = torch.ones(B, dtype=i32, device=dev)
        paths = []
        for s in range(len(sets)):
            pth = torch.full((B, L + 1), -1, dtype=i32, device=dev)
            pth[:, 0] = 0
            pth[:, 1] = 1 + s % max(1, N - 1)
            paths.append(pth)
    calls = {
        "build_beam10": lambda st, s, i: P.presto_score_build_tree(
            step.topk_ids, step.topk_logq, st["ctx"], ngram, w.lam, N, b=w.branching,
            out=tree, ws=ws_b, stream=s, policy=P.SEARCH_BEAM, beam_width=10),
        "build_eager": lambda st, s, i: P.presto_score_build_tree(
            step.topk_ids, step.topk_logq, st["ctx"], ngram, w.lam, N, b=w.branching,
            out=tree, ws=ws_b, stream=s, policy=P.SEARCH_EAGER),
        "build_lambda_d": lambda st, s, i: P.presto_score_build_tree(
            step.topk_ids, step.topk_logq, st["ctx"], ngram, w.lam, N, b=w.branching,
            out=tree, ws=ws_b, stream=s, lambda_d=lam_d),
        "topk_entropy": lambda st, s, i: P.presto_topk_entropy(
            st["logits"], k, 0.5, 2.0, step.topk_ids, step.topk_logq, step.lse, ent, lam_out,
            ws=step.ws_topk, stream=s),
    }
    if slots is not None:
        calls["topk_slots"] = lambda st, s, i: P.presto_topk_slots(
            slots, acc_len, paths[i], 1, L, k, topk_ids=step.topk_ids, topk_logq=step.topk_logq,
            lse=step.lse, ws=step.ws_topk, stream=s)
    # one whole round at the largest budget the paper sweeps (N = 1024, k = 10)
    w2 = w.scaled(N=1024, k=10)
    step2 = P.DraftVerifyStep(w2.B, w2.L, w2.V, w2.k, w2.N, w2.Hq, w2.Hkv, w2.D, w2.T,
                              logits_dtype=sets[0]["logits"].dtype, b=w2.branching, lam=w2.lam,
                              ngram=ngram, device=dev)
    att2 = synth.attention_inputs(w2, device=dev)
    kv2 = att2.pop("kv_len").to(torch.int32)
    tgt2 = torch.zeros(w2.B, w2.N, dtype=i32, device=dev)
    g2 = step2.capture(sets[0]["logits"], sets[0]["ctx"], [att2], kv2, tgt2)
    out = {}
    for _ in range(3):
        g2.replay()
    ea = torch.cuda.Event(enable_timing=True)
    eb = torch.cuda.Event(enable_timing=True)
    ea.record()
    for _ in range(args.kernel_steps):
        g2.replay()
    eb.record()
    torch.cuda.synchronize()
    out["round_N1024_k10"] = ea.elapsed_time(eb) * 1e3 / args.kernel_steps
    del g2, step2, att2
    for name, fn in calls.items():
        def run(s, fn=fn):
            for i, st in enumerate(sets):
                fn(st, s, i)
        with torch.cuda.stream(side):
            run(side)
        side.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            run(side)
        with torch.cuda.stream(side):
            for _ in range(3):
                g.replay()
            ea = torch.cuda.Event(enable_timing=True)
            eb = torch.cuda.Event(enable_timing=True)
            ea.record(side)
            for _ in range(args.kernel_steps):
                g.replay()
            eb.record(side)
        side.synchronize()
        out[name] = ea.elapsed_time(eb) * 1e3 / (args.kernel_steps * len(sets))
        del g
    del slots
    torch.cuda.synchronize()
    if int(step.dev_status.item()) != 0:
        raise RuntimeError(f"device status after variants: "
                           f"{P.dev_status_names(int(step.dev_status.item()))}")
    return out


def cpu_baseline(args, w):
    """The oracle timed on the host cores, each leg in a subprocess without a GPU:
    one thread (full rounds of the workload's input set 0, whose results come back
    in a temporary file), one process per host core (full rounds), and for the two
    large workloads one round on a subset of (sequence, kv head) pairs, scaled to
    the whole round by attention flops.  Returns (cpu_baseline dict, results file)."""
    import tempfile
    host = os.cpu_count()
    fd, path = tempfile.mkstemp(suffix=".npz")
    os.close(fd)
    out = {"value": None, "unit": "steps/s", "cores": None, "host_cores": host, "kind": "oracle",
           "sample": None}
    try:
        r1 = run_oracle(args.workload, args.cpu_seconds, 10 ** 6, mode="round", parity_out=path)
        one = {"value": r1["rounds"] / r1["seconds"], "unit": "steps/s", "cores": 1,
               "sample": f"{r1['rounds']} full oracle rounds ({r1['seconds']:.1f} s), one thread"}
        out["single_thread"] = one
        out.update(value=one["value"], cores=1, sample=one["sample"])
    except Exception as e:  # reported, not fatal
        out["sample"] = f"failed: {e}"[:300]
        os.unlink(path)
        return out, None
    try:
        r2 = run_oracle(args.workload, args.cpu_seconds, 10 ** 6, mode="mp")
        out.update(value=r2["rounds"] / r2["seconds"], cores=r2["procs"],
                   sample=(f"{r2['rounds']} full oracle rounds ({r2['seconds']:.1f} s) of the "
                           f"same workload (input set 0), numpy float64, with top-k rows, "
                           f"trees and attention (sequence, kv head) pairs spread over "
                           f"{r2['procs']} processes, one per host core"))
    except Exception as e:
        out["multi_process"] = f"failed: {e}"[:300]
    by = {}
    for name in ATTN_SUBSET:
        try:
            r = run_oracle(name, 0, 1, mode="subset")
            by[name] = {"seconds_per_round": r["seconds_per_round"],
                        "steps_per_s": 1.0 / r["seconds_per_round"], "cores": 1,
                        "step_seconds": r["steps"],
                        "sample": (f"one round on one thread: top-k, tree, mask and accept in "
                                   f"full; attention of sequences {r['subset']['seqs']} x kv "
                                   f"heads {r['subset']['kv_heads']} of one layer, scaled by "
                                   f"attention flops (x{r['attention_scale']:.1f}) to every "
                                   f"sequence, head and layer")}
        except Exception as e:
            by[name] = {"failed": f"{e}"[:300]}
    out["by_workload"] = by
    return out, path


def round_parity(w, step, st0, graph0, oracle_file):
    """Replays the round on input set 0 (the graph the timed region replays) and checks
    it against the oracle: the top-k against the oracle's top-k of the same logits
    (ids exact; log q and lse within 1e-5 relative), then every later step against
    the oracle applied to that step's inputs as the GPU had them (oracle_check).  The
    tree of the oracle's own chain may differ where float32 near-ties decide a node;
    `chain_tree_equal` reports whether it did."""
    import tempfile
    import numpy as np
    import torch
    o = dict(np.load(oracle_file))
    step.dev_status.zero_()
    if graph0 is not None:
        graph0.replay()
    else:
        step.run(st0["logits"], st0["ctx"], st0["layers"], st0["kv_len"], st0["target"])
    torch.cuda.synchronize()
    h = lambda t: t.cpu().numpy()

    def rel(a, b):
        a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
        both = np.isinf(a) & np.isinf(b) & (np.sign(a) == np.sign(b))
        e = np.where(both, 0.0, np.abs(a - b) / np.maximum(1.0, np.abs(b)))
        return float(e.max()) if e.size else 0.0

    R = w.rows
    g = {"ids": h(step.topk_ids).reshape(R, w.k), "logq": h(step.topk_logq).reshape(R, w.k),
         "mask": h(step.mask).view(np.uint32), "pos_ids": h(step.pos_ids),
         "attn": h(step.attn_out.float()).astype(np.float64), "accept_len": h(step.accept_len),
         "accept_path": h(step.accept_path), "bonus": h(step.bonus), "target": h(st0["target"]),
         "kv_len": h(st0["kv_len"])}
    g.update({k: h(v) for k, v in step.tree.items()})
    if w.layers == 1:  # the attention inputs are drawn on the GPU: hand them over as read
        g.update({k: h(st0["layers"][0][k].float()) for k in ("q", "k_cache", "v_cache",
                                                               "k_tree", "v_tree")})
    c = {"topk_ids": bool(np.array_equal(g["ids"], o["ids"])),
         "logq_rel_err": rel(g["logq"], o["logq"]),
         "lse_rel_err": rel(h(step.lse).reshape(R), o["lse"]),
         "chain_tree_equal": bool(all(np.array_equal(g[k], o[k]) for k in ("token", "parent",
                                                                          "depth", "n_nodes"))),
         "dev_status": int(step.dev_status.item())}
    fd, path = tempfile.mkstemp(suffix=".npz")
    os.close(fd)
    try:
        np.savez(path, **g)
        c.update(run_oracle(w.name, 0, 1, mode="check", check_in=path))
    except Exception as e:  # reported
        c["check_failed"] = f"{e}"[:300]
    finally:
        os.unlink(path)
    ok = (c["topk_ids"] and c["logq_rel_err"] <= 1e-5 and c["lse_rel_err"] <= 1e-5
          and c.get("tree", False) and c.get("tree_scores_equal", False) and c.get("mask", False)
          and c.get("pos_ids", False) and c.get("accept", False) and c["dev_status"] == 0
          and (c.get("attention_max_abs") is None or c["attention_max_abs"] <= 2e-2))
    return {"ok": ok, "input_set": 0, "checks": c,
            "against": ("the CPU oracle: top-k from the same logits; every later step from "
                        "that step's inputs as the GPU had them")}


def max_over_ranks(x, device=None):
    """The largest of every rank's x (the job's time is its slowest replica's); x
    itself on a single process."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world, steps_per_rank, seconds):
    """Whole-job rounds per second: every rank ran steps_per_rank rounds (replicas,
    weak scaling) within the slowest rank's seconds."""
    return world * steps_per_rank / seconds


def time_workload_rooflines(args, P, hbm, tc, tc_sus):
    """Top-k and one attention layer of the larger workloads, each timed the way the
    per-call numbers are (a graph of launches over inputs that together exceed L2),
    against the measured peaks: the kernels' rooflines where the work is large enough
    to approach them."""
    import numpy as np
    import torch

    import synth
    dev = torch.device("cuda", torch.cuda.current_device())
    out = {}
    for name in ("self_spec", "batched_ragged", "long_ctx"):
        w = synth.WORKLOADS[name]
        x0 = synth.drafter_logits(w).to(dev)
        nbytes = x0.numel() * x0.element_size()
        R = max(2, math.ceil(300e6 / nbytes))
        xs = [x0] + [torch.roll(x0, shifts=i, dims=2) for i in range(1, R)]
        ids = torch.empty(w.B, w.L, w.k, dtype=torch.int32, device=dev)
        lq = torch.empty(w.B, w.L, w.k, dtype=torch.float32, device=dev)
        lse = torch.empty(w.B, w.L, dtype=torch.float32, device=dev)
        ws_t = torch.empty(max(P.presto_topk_workspace(w.B, w.L, w.V, w.k), 256), dtype=torch.uint8,
                           device=dev)
        topk_us = _graph_time(args, lambda s: [P.presto_topk(x, w.k, ids, lq, lse, ws=ws_t, stream=s)
                                               for x in xs], len(xs))
        del xs, x0
        # one attention layer over a full k-ary tree of N nodes (every node used)
        att = synth.attention_inputs(w, device=dev)
        kv = att.pop("kv_len").to(torch.int32)
        par = [-1] + [(i - 1) // w.k for i in range(1, w.N)]
        dep = [0] * w.N
        for i in range(1, w.N):
            dep[i] = dep[par[i]] + 1
        parent = torch.tensor([par] * w.B, dtype=torch.int32, device=dev)
        depth = torch.tensor([dep] * w.B, dtype=torch.int32, device=dev)
        nn = torch.full((w.B,), w.N, dtype=torch.int32, device=dev)
        mask, _ = P.presto_tree_mask(parent, depth, nn, kv)
        ws_a = torch.empty(max(P.presto_attn_workspace(w.B, w.N, w.Hq, w.Hkv, w.D, w.T), 256),
                           dtype=torch.uint8, device=dev)
        o = torch.empty(w.B, w.N, w.Hq, w.D, dtype=torch.bfloat16, device=dev)
        ol = torch.empty(w.B, w.N, w.Hq, dtype=torch.float32, device=dev)
        attn_us = _graph_time(args, lambda s: P.presto_tree_attention(
            att["q"], att["k_cache"], att["v_cache"], kv, att["k_tree"], att["v_tree"], mask, nn,
            out=o, lse=ol, ws=ws_a, stream=s), 1)
        kvh = kv.cpu().numpy()
        anc = w.B * (sum(dep) + w.N)
        flops = 4.0 * w.Hq * w.D * (w.N * int(kvh.sum()) + anc)
        abytes = 2 * w.Hkv * w.D * 2 * (int(kvh.sum()) + w.B * w.N) + 2 * w.B * w.N * w.Hq * w.D * 2
        out[name] = {
            "topk_us": topk_us, "topk_gbs": nbytes / (topk_us * 1e-6) / 1e9,
            "topk_hbm_frac": nbytes / (topk_us * 1e-6) / 1e9 / hbm,
            "attention_layer_us": attn_us,
            "attention_tflops": flops / (attn_us * 1e-6) / 1e12,
            "attention_tensor_frac": flops / (attn_us * 1e-6) / 1e12 / tc,
            "attention_tensor_frac_sustained": flops / (attn_us * 1e-6) / 1e12 / tc_sus,
            "attention_hbm_frac": abytes / (attn_us * 1e-6) / 1e9 / hbm,
        }
        del att, mask
        torch.cuda.synchronize()
    return out


def time_full_depth(args, P):
    """The long-context workload's whole round with every one of its 36 attention layers
    (independent seeded Q/K/V, ~39 GB of KV cache resident): the full-depth
    tree-verify time per round."""
    import numpy as np
    import torch

    import synth
    w = synth.WORKLOADS["long_ctx"]
    dev = torch.device("cuda", torch.cuda.current_device())
    kv_bytes = w.layers * 2 * w.B * w.Hkv * w.T * w.D * 2
    free, _ = torch.cuda.mem_get_info(dev)
    if free < kv_bytes * 1.2 + (8 << 30):
        return {"skipped": f"needs about {kv_bytes * 1.2 / 1e9:.0f} GB of free device memory"}
    a, b, t, lr = synth.trigram_entries(w)
    ngram = P.Ngram3Table.from_entries(a, b, t, lr, w.table_log2_cap, w.miss_logrho, device=dev)
    logits = synth.drafter_logits(w).to(dev)
    ctx = synth.ctx_tokens(w).to(dev)
    layers, kv = [], None
    for j in range(w.layers):
        att = synth.attention_inputs(w, layer=j, device=dev)
        kv = att.pop("kv_len").to(torch.int32)
        layers.append(att)
    step = P.DraftVerifyStep(w.B, w.L, w.V, w.k, w.N, w.Hq, w.Hkv, w.D, w.T,
                             logits_dtype=logits.dtype, b=w.branching, lam=w.lam, ngram=ngram,
                             device=dev)
    target = torch.zeros(w.B, w.N, dtype=torch.int32, device=dev)
    g = step.capture(logits, ctx, layers, kv, target)
    for _ in range(2):
        g.replay()
    ea = torch.cuda.Event(enable_timing=True)
    eb = torch.cuda.Event(enable_timing=True)
    reps = 5
    ea.record()
    for _ in range(reps):
        g.replay()
    eb.record()
    torch.cuda.synchronize()
    ms = ea.elapsed_time(eb) / reps
    n_nodes = step.tree["n_nodes"].cpu().numpy()
    mask = step.mask.cpu().numpy().view(np.uint32)
    anc = sum(int(np.unpackbits(mask[q, : int(n_nodes[q])].view(np.uint8)).sum())
              for q in range(w.B))
    kvh = kv.cpu().numpy()
    flops = 4.0 * w.Hq * w.D * (sum(int(kvh[q]) * int(n_nodes[q]) for q in range(w.B)) + anc)
    launches = step.kernels_per_round(w.layers)
    del layers, step, g
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return {"workload": "long_ctx: B=8 L=16 k=10 N=256 T=32768, 36 attention layers",
            "ms_per_round": ms, "rounds_per_s": 1e3 / ms, "gpu_launches_per_round": launches,
            "attention_tflops": flops * w.layers / (ms * 1e-3) / 1e12,
            "kv_cache_gb": kv_bytes / 1e9}


def _graph_time(args, fn, per_replay):
    """Per-launch time of fn's launches captured in one CUDA graph (replayed after
    three warm-up replays), by CUDA events on the launching stream."""
    import torch
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        fn(side)
    side.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        fn(side)
    reps = max(3, args.kernel_steps // 2)
    with torch.cuda.stream(side):
        for _ in range(3):
            g.replay()
        ea = torch.cuda.Event(enable_timing=True)
        eb = torch.cuda.Event(enable_timing=True)
        ea.record(side)
        for _ in range(reps):
            g.replay()
        eb.record(side)
    side.synchronize()
    return ea.elapsed_time(eb) * 1e3 / (reps * per_replay)


def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    import paper_2607_22634_gb300 as P
    import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    P.load()
    w = synth.WORKLOADS[args.workload]

    # ---- resident state: trigram table, step buffers
    ngram = None
    if w.use_table:
        a, b, t, lr = synth.trigram_entries(w)
        ngram = P.Ngram3Table.from_entries(a, b, t, lr, w.table_log2_cap, w.miss_logrho,
                                           device=dev)
    logits_dtype = torch.bfloat16 if w.logits_dtype == "bf16" else torch.float32
    step = P.DraftVerifyStep(w.B, w.L, w.V, w.k, w.N, w.Hq, w.Hkv, w.D, w.T,
                             logits_dtype=logits_dtype, b=w.branching, lam=w.lam, ngram=ngram,
                             device=dev)

    # ---- rotating input sets, together larger than 2 x L2
    esz = 2 if logits_dtype == torch.bfloat16 else 4
    kv_bytes = 2 * w.B * w.Hkv * w.T * w.D * 2 * w.layers
    set_bytes = w.B * w.L * w.V * esz + kv_bytes + 3 * w.B * w.N * w.Hq * w.D * 2 * w.layers
    n_sets = max(2, math.ceil(2.2 * L2_BYTES / set_bytes))
    sets = []
    for s in range(n_sets):
        ws = w.scaled(seed=w.seed * 1000 + s + 1) if s else w
        logits = synth.drafter_logits(ws).to(dev)
        ctx = synth.ctx_tokens(w).to(dev)
        layers = []
        kv_len = None
        for layer in range(w.layers):
            att = synth.attention_inputs(ws, layer=layer, device=dev)
            kv_len = att.pop("kv_len").to(torch.int32)
            layers.append(att)
        sets.append({"logits": logits, "ctx": ctx, "layers": layers, "kv_len": kv_len,
                     "target": torch.empty(w.B, w.N, dtype=torch.int32, device=dev)})
    # target tokens: the synthetic target model applied to each set's tree (not timed)
    for st in sets:
        step.run(st["logits"], st["ctx"], st["layers"], st["kv_len"], st["target"])
        tree = {k: v.cpu().numpy() for k, v in step.tree.items()}
        st["target"].copy_(synth.target_tokens(w, st["logits"], tree["token"], tree["parent"],
                                               tree["n_nodes"], device=dev).to(dev))
    torch.cuda.synchronize()
    if int(step.dev_status.item()) != 0:
        raise RuntimeError(f"device status: {P.dev_status_names(int(step.dev_status.item()))}")

    use_graph = not args.no_graph
    graphs = []
    if use_graph:
        for st in sets:
            graphs.append(step.capture(st["logits"], st["ctx"], st["layers"], st["kv_len"],
                                       st["target"]))
    stream = torch.cuda.current_stream(dev)

    # the timed rounds replay graphs of many rounds each (the input sets in turn), so
    # that a round pays no per-graph launch gap; the end-to-end loop below keeps one
    # graph per round, as a host loop that reads every round's result must
    def capture_chain(count):
        s2 = torch.cuda.Stream(device=dev)
        s2.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s2):
            for i in range(count):
                st = sets[i % n_sets]
                step.run(st["logits"], st["ctx"], st["layers"], st["kv_len"], st["target"],
                         stream=s2)
        stream.wait_stream(s2)
        return g

    chain = capture_chain(n_sets) if use_graph else None
    rem_n = args.steps % n_sets
    rem = capture_chain(rem_n) if use_graph and rem_n else None

    def timed_rounds():
        if use_graph:
            for _ in range(args.steps // n_sets):
                chain.replay()
            if rem is not None:
                rem.replay()
        else:
            for i in range(args.steps):
                one(i)

    def one(i):
        if use_graph:
            graphs[i % n_sets].replay()
        else:
            st = sets[i % n_sets]
            step.run(st["logits"], st["ctx"], st["layers"], st["kv_len"], st["target"])

    for i in range(args.warmup):
        one(i)
    if chain is not None:
        chain.replay()
    torch.cuda.synchronize()

    # ---- timed region: K rounds, repeated (each repeat between its own pair of CUDA
    # events on the launch stream) at least --repeats times and for at least
    # --repeat-seconds, so that the clock sampler sees the load; value = the median
    # repeat (max over ranks), with its spread
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    evs = []
    with ClockSampler(gpu_smi_id(dev)) as clk:
        t_wall0 = time.time()
        while len(evs) < max(1, args.repeats) or (time.time() - t_wall0 < args.repeat_seconds
                                                  and len(evs) < 5000):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            timed_rounds()
            e1.record(stream)
            evs.append((e0, e1))
            if len(evs) % 64 == 0:
                e1.synchronize()
        torch.cuda.synchronize()
        t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    rep_ms = [a.elapsed_time(b) for a, b in evs]
    ms = max_over_ranks(statistics.median(rep_ms), dev)
    clocks = clk.summary(t_wall0, t_wall1)
    value = job_throughput(world, args.steps, ms / 1e3)
    repeats = {"n": len(rep_ms), "ms_per_step_median": ms / args.steps,
               "ms_per_step_min": min(rep_ms) / args.steps,
               "ms_per_step_max": max(rep_ms) / args.steps,
               "value_min": job_throughput(world, args.steps, max(rep_ms) / 1e3),
               "value_max": job_throughput(world, args.steps, min(rep_ms) / 1e3)}

    # ---- per-call durations: each call alone, captured n_sets times in a row
    # (rotating over the input sets, so the big inputs come from HBM) into a CUDA
    # graph whose replays are timed with CUDA events on the launching stream.
    # Per launch = kernel time + the graph's launch gap.
    us = {}
    side = torch.cuda.Stream(device=dev)
    side.wait_stream(stream)
    for c in step.CALLS:
        def calls(s, c=c):
            for st in sets:
                step.run(st["logits"], st["ctx"], st["layers"], st["kv_len"], st["target"],
                         stream=s, only=(c,))
        with torch.cuda.stream(side):
            calls(side)
        side.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            calls(side)
        with torch.cuda.stream(side):
            for _ in range(3):
                g.replay()
            ea = torch.cuda.Event(enable_timing=True)
            eb = torch.cuda.Event(enable_timing=True)
            ea.record(side)
            for _ in range(args.kernel_steps):
                g.replay()
            eb.record(side)
        side.synchronize()
        us[c] = ea.elapsed_time(eb) * 1e3 / (args.kernel_steps * n_sets)
        del g
    torch.cuda.synchronize()

    # ---- the paper's variants of the same calls, timed the same way: beam search
    # (W = 10), Alg. 2 as printed, a per-row lambda, top-k with entropy-adaptive
    # lambda, and the self-speculative top-k over the accepted node's mask slots
    variant_us = None
    if not args.no_variants:
        variant_us = time_variants(args, P, w, step, sets, side, ngram)

    # ---- end to end through the public API with host buffers: every round's inputs
    # (logits, context, target tokens, each layer's q and tree K/V; the KV cache is
    # resident) sit packed in one pinned host buffer and go to the device in one copy;
    # the round's results come back in one copy that the host waits for.  StagedRounds
    # double-buffers the staging and keeps one round queued ahead of the host; with the
    # pool of pinned buffers fixed, each round step is one graph (the round, its results
    # out, and beside them the next round's inputs in), one replay and one wait
    def tensors_of(st):
        out = [st["logits"], st["ctx"], st["target"]]
        for lay in st["layers"]:
            out += [lay["q"], lay["k_tree"], lay["v_tree"]]
        return out

    def bind(v):
        layers_s = [{"q": v[3 + 3 * j], "k_tree": v[4 + 3 * j], "v_tree": v[5 + 3 * j],
                     "k_cache": sets[0]["layers"][j]["k_cache"],
                     "v_cache": sets[0]["layers"][j]["v_cache"]} for j in range(w.layers)]
        return v[0], v[1], layers_s, sets[0]["kv_len"], v[2]

    staged = P.StagedRounds(step, tensors_of(sets[0]), bind)
    host = [staged.pack(tensors_of(st)) for st in sets]  # the fixed pool of pinned buffers
    staged.fuse(host)
    h2d = staged.nbytes
    d2h = step.result.numel() * step.result.element_size()
    n_warm = min(20, args.e2e_steps)
    staged.start_pooled(host[0], host[1 % n_sets])
    for i in range(n_warm):
        staged.run_pooled(i, host[(i + 2) % n_sets])
    n_e2e = args.e2e_steps
    t0 = time.perf_counter()
    for i in range(n_warm, n_warm + n_e2e):
        staged.run_pooled(i, host[(i + 2) % n_sets])
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)
    e2e_value = job_throughput(world, n_e2e, e2e_s)
    torch.cuda.synchronize()

    # ---- roofline of the dominant call (attention work from input set 0's tree)
    peaks, peak_src = load_peaks()
    if use_graph:
        graphs[0].replay()
    else:
        one(0)
    torch.cuda.synchronize()
    tree = {k: v.cpu().numpy() for k, v in step.tree.items()}
    mask = step.mask.cpu().numpy().view(np.uint32)
    kv = sets[0]["kv_len"].cpu().numpy()
    anc = sum(int(np.unpackbits(mask[b, : int(tree["n_nodes"][b])].view(np.uint8)).sum())
              for b in range(w.B))
    n_used = int(tree["n_nodes"].sum())
    attn_flops = 4.0 * w.Hq * w.D * (sum(int(kv[b]) * int(tree["n_nodes"][b])
                                         for b in range(w.B)) + anc) * w.layers
    attn_bytes = (2 * w.Hkv * w.D * 2 * (int(kv.sum()) + n_used)
                  + 2 * w.B * w.N * w.Hq * w.D * 2) * w.layers
    topk_bytes = w.B * w.L * w.V * esz
    dominant = max(us, key=us.get)
    hbm = float(peaks["hbm_gbs"])
    # each call is timed alone (a graph of that call's launches), so a contraction's
    # fraction is taken of the burst tensor peak; the sustained one is reported too
    tc = float(peaks["bf16_tflops"])
    tc_sus = float(peaks.get("bf16_tflops_sustained", tc))
    if dominant == "attention":
        t_us = us["attention"]
        t_tensor = attn_flops / (tc * 1e12) * 1e6
        t_hbm = attn_bytes / (hbm * 1e9) * 1e6
        if t_tensor >= t_hbm:
            ach = attn_flops / (t_us * 1e-6) / 1e12
            roof = {"bound": "tensor", "achieved": ach, "peak": tc, "unit": "TFLOP/s"}
        else:
            ach = attn_bytes / (t_us * 1e-6) / 1e9
            roof = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s"}
        roof["kernel"] = ("presto_tree_attention (attn_kernel" +
                          (" + attn_merge_kernel)" if step.attn_launches > 1 else ")"))
        roof["traffic"] = profiled_traffic("attention")
        roof["tensor_frac"] = attn_flops / (t_us * 1e-6) / 1e12 / tc
        roof["tensor_frac_sustained"] = attn_flops / (t_us * 1e-6) / 1e12 / tc_sus
        roof["hbm_frac"] = attn_bytes / (t_us * 1e-6) / 1e9 / hbm
        roof["algorithmic"] = {"flops": attn_flops, "bytes": attn_bytes}
    else:
        t_us = us[dominant]
        if dominant == "topk":
            ach = topk_bytes / (t_us * 1e-6) / 1e9
            roof = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s",
                    "kernel": "presto_topk (topk_kernel)", "traffic": profiled_traffic("topk"),
                    "algorithmic": {"bytes": topk_bytes}}
        else:
            roof = {"bound": "latency", "achieved": None, "peak": None, "unit": "us",
                    "kernel": dominant, "traffic": None}
    if roof.get("achieved") is not None:
        roof["frac"] = roof["achieved"] / roof["peak"]
    roof["peak_source"] = (f"{peak_src} ({'bf16 burst; tensor_frac of burst, tensor_frac_sustained'
                           f' of sustained' if roof.get('unit') == 'TFLOP/s' else 'copy'}); "
                           f"attention tensor_frac of burst {tc}, tensor_frac_sustained of "
                           f"sustained {tc_sus} TFLOP/s")
    roof["duration_us"] = t_us
    roof["timing"] = (f"CUDA events around {args.kernel_steps} replays of a graph of {n_sets} "
                      f"launches of the call alone (one per input set); per launch")
    topk_frac = topk_bytes / (us["topk"] * 1e-6) / 1e9 / hbm

    by_workload = None
    if not args.no_variants:
        by_workload = time_workload_rooflines(args, P, hbm, tc, tc_sus)
        by_workload["long_ctx_full_depth"] = time_full_depth(args, P)

    # ---- the CPU oracle on the host cores (rank 0, one GPU): one thread, one process
    # per core, and the large workloads on a subset scaled by flops; the one-thread
    # leg also returns input set 0's round, which the GPU round is checked against
    cpu, parity = None, None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu, oracle_file = cpu_baseline(args, w)
        if oracle_file is not None:
            parity = round_parity(w, step, sets[0], graphs[0] if use_graph else None, oracle_file)
            os.unlink(oracle_file)

    if rank == 0:
        print(json.dumps({
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": bench_config(w, world),
            "timing": {"inputs": f"{n_sets} rotating input sets of {set_bytes / 1e6:.1f} MB "
                                 f"({n_sets * set_bytes / 1e6:.0f} MB > 2 x L2), no L2 flush",
                       "cuda_graph": (f"timed rounds replay graphs of {n_sets} rounds (the input "
                                      f"sets in turn); e2e one graph per round") if use_graph
                                     else False,
                       "repeats": repeats},
            "parity": parity,
            "roofline": roof,
            "topk_hbm_frac": topk_frac,
            "call_us": us,
            "variant_us": variant_us,
            "roofline_by_workload": by_workload,
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": "steps/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h,
                    "note": "every round: its inputs (logits, q, tree K/V, ctx, targets) packed "
                            "in one pinned host buffer, one copy in (on a copy stream, into one "
                            "of two staging buffers, overlapping the previous round); the "
                            "round (a CUDA graph); accept_len/path/bonus in one copy out; a "
                            "host wait for it. One round is queued ahead of the host wait, as "
                            "a server alternating two independent request groups does; the "
                            "pinned buffers form a fixed pool, so each round step (round, "
                            "results out, next inputs in beside it) is one captured graph. "
                            "KV cache resident (StagedRounds pooled mode)"},
            "clocks": clocks,
            "gpu_launches": args.steps * step.kernels_per_round(w.layers),
        }), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.oracle_worker:
        oracle_worker(args)
        return
    if args.impl == "reference":
        run_reference(args)
        return
    run_ours(args)


if __name__ == "__main__":
    main()
