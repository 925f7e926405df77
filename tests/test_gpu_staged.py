"""StagedRounds (rounds fed from pinned host memory, one round queued ahead of the
host), both with separate copies and launches and in pooled mode (one captured graph
per round step): every round's returned accept results equal those of the same
inputs run eagerly through DraftVerifyStep, across three rotating input sets."""

import numpy as np
import torch

import synth
import paper_2607_22634_gb300 as P
from gpu_common import GPU

pytestmark = GPU


def test_staged_rounds_return_each_rounds_results():
    w = synth.WORKLOADS["qwen3_8b"]
    dev = "cuda"
    a, b, t, lr = synth.trigram_entries(w)
    ngram = P.Ngram3Table.from_entries(a, b, t, lr, w.table_log2_cap, w.miss_logrho, device=dev)
    step = P.DraftVerifyStep(w.B, w.L, w.V, w.k, w.N, w.Hq, w.Hkv, w.D, w.T,
                             logits_dtype=torch.bfloat16, b=w.branching, lam=w.lam, ngram=ngram,
                             device=dev)
    att = synth.attention_inputs(w, device=dev)
    kv = att.pop("kv_len").to(torch.int32)
    sets, want = [], []
    for s in range(3):
        ws = w.scaled(seed=w.seed * 1000 + s + 1) if s else w
        logits = synth.drafter_logits(ws).to(dev)
        ctx = synth.ctx_tokens(w).to(dev)
        layer = synth.attention_inputs(ws, device=dev)
        layer.pop("kv_len")
        layer["k_cache"], layer["v_cache"] = att["k_cache"], att["v_cache"]
        target = torch.zeros(w.B, w.N, dtype=torch.int32, device=dev)
        step.run(logits, ctx, [layer], kv, target)
        tree = {k: v.cpu().numpy() for k, v in step.tree.items()}
        target.copy_(synth.target_tokens(w, logits.cpu(), tree["token"], tree["parent"],
                                         tree["n_nodes"]).to(dev))
        step.run(logits, ctx, [layer], kv, target)
        torch.cuda.synchronize()
        want.append(step.result.cpu().numpy().copy())
        sets.append([logits, ctx, target, layer["q"], layer["k_tree"], layer["v_tree"]])

    def bind(v):
        return v[0], v[1], [{"q": v[3], "k_tree": v[4], "v_tree": v[5],
                             "k_cache": att["k_cache"], "v_cache": att["v_cache"]}], kv, v[2]

    staged = P.StagedRounds(step, sets[0], bind)
    host = [staged.pack(st) for st in sets]
    n = 7
    staged.start(host[0])
    for i in range(n):
        got = staged.run(i, host[(i + 1) % 3] if i + 1 < n else None).numpy().copy()
        np.testing.assert_array_equal(got, want[i % 3], err_msg=f"round {i}")
    torch.cuda.synchronize()
    assert int(step.dev_status.item()) == 0
    # pooled mode: one graph replay per round step
    staged.fuse(host)
    staged.start_pooled(host[0], host[1])
    for i in range(n):
        if i + 1 < n:
            got = staged.run_pooled(i, host[(i + 2) % 3] if i + 2 < n else None)
        else:
            got = staged.wait_pooled(i)
        np.testing.assert_array_equal(got.numpy().copy(), want[i % 3], err_msg=f"pooled round {i}")
    torch.cuda.synchronize()
    assert int(step.dev_status.item()) == 0
    # the sets really differ, so a round returning another round's results would fail
    assert not all(np.array_equal(want[0], x) for x in want[1:])
