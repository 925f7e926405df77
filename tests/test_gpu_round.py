"""One whole draft-and-verify round (DraftVerifyStep: top-k -> tree with its mask and
position ids -> tree attention -> accept, all through the C ABI) on the workloads'
own synthetic inputs, checked step by step against the oracle:

* top-k against the oracle's top-k of the same logits (ids exact, log q and lse
  within 1e-5 relative);
* the tree against the oracle's best-first search on the GPU's candidates (exact,
  float32 scores bitwise), and against the oracle's own chain up to float32
  near-ties at the budget boundary;
* mask and position ids from the GPU's tree, and the accepted path on the GPU's tree
  with the synthetic target's tokens, exact;
* attention with the GPU's mask within 2e-2 max abs of float64 (every row for the
  Qwen3-8B-shaped round; seeded (sequence, kv head) samples for the larger ones)."""

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import ATTN_TOL, GPU, LOGQ_TOL, assert_tree_close, rel_close

pytestmark = GPU


def _round(name):
    w = synth.WORKLOADS[name]
    dev = "cuda"
    logits = synth.drafter_logits(w)
    ctx = synth.ctx_tokens(w)
    a, b, t, lr = synth.trigram_entries(w)
    ngram = (P.Ngram3Table.from_entries(a, b, t, lr, w.table_log2_cap, w.miss_logrho, device=dev)
             if w.use_table else None)
    table = O.make_table(a, b, t, lr) if w.use_table else None
    att = synth.attention_inputs(w, device="cpu")
    kv = att["kv_len"]
    step = P.DraftVerifyStep(w.B, w.L, w.V, w.k, w.N, w.Hq, w.Hkv, w.D, w.T,
                             logits_dtype=logits.dtype, b=w.branching, lam=w.lam, ngram=ngram,
                             device=dev)
    layer = {k: v.to(dev) for k, v in att.items() if k != "kv_len"}
    # the target's tokens follow the tree, so the round runs once to build it
    target = torch.zeros(w.B, w.N, dtype=torch.int32, device=dev)
    step.run(logits.to(dev), ctx.to(dev), [layer], kv.to(dev), target)
    torch.cuda.synchronize()
    tree = {k: v.cpu().numpy() for k, v in step.tree.items()}
    target.copy_(synth.target_tokens(w, logits, tree["token"], tree["parent"], tree["n_nodes"]))
    step.dev_status.zero_()
    step.run(logits.to(dev), ctx.to(dev), [layer], kv.to(dev), target)
    torch.cuda.synchronize()
    assert int(step.dev_status.item()) == 0
    return w, logits, ctx.numpy(), table, att, kv.numpy(), step, target.cpu().numpy()


@pytest.mark.parametrize("name,pairs", [
    ("qwen3_8b", None),
    ("batched_ragged", [(0, 0), (7, 3), (15, 7)]),
    ("self_spec", [(1, 2), (3, 5)]),
    ("long_ctx", [(2, 1), (6, 6)]),
])
def test_round_matches_oracle_step_by_step(name, pairs):
    w, logits, ctx, table, att, kv, step, target = _round(name)
    R = w.rows
    # top-k
    oids, ologq, olse = O.topk_logsoftmax(logits.reshape(R, w.V).double().numpy(), w.k)
    gids = step.topk_ids.cpu().numpy().reshape(R, w.k)
    glogq = step.topk_logq.cpu().numpy().reshape(R, w.k)
    np.testing.assert_array_equal(gids, oids)
    assert rel_close(glogq, ologq) <= LOGQ_TOL
    assert rel_close(step.lse.cpu().numpy().reshape(R), olse) <= LOGQ_TOL
    # the tree from the GPU's candidates, exactly; and the oracle's own chain up to
    # near-ties
    g = {k: v.cpu().numpy() for k, v in step.tree.items()}
    ids3, logq3 = gids.astype(np.int64).reshape(w.B, w.L, w.k), glogq.astype(np.float64).reshape(w.B, w.L, w.k)
    o = O.best_first_tree(ids3, logq3, ctx, table, w.miss_logrho, w.lam, w.branching, w.N, "fp32")
    for key in ("token", "parent", "depth", "n_nodes"):
        np.testing.assert_array_equal(g[key], o[key], err_msg=key)
    np.testing.assert_array_equal(g["score"].astype(np.float32), o["score"].astype(np.float32))
    assert_tree_close(g, oids.reshape(w.B, w.L, w.k), ologq.reshape(w.B, w.L, w.k), ctx, table,
                      w.miss_logrho, w.lam, w.N)
    # mask, position ids and acceptance on the GPU's tree
    omask, opos = O.tree_mask(g["parent"], g["depth"], g["n_nodes"], kv, w.N)
    gmask = step.mask.cpu().numpy().view(np.uint32)
    np.testing.assert_array_equal(gmask, omask)
    np.testing.assert_array_equal(step.pos_ids.cpu().numpy(), opos)
    oacc, opath, obonus = O.accept(g["token"], g["parent"], g["n_nodes"], target, w.L)
    np.testing.assert_array_equal(step.accept_len.cpu().numpy(), oacc)
    np.testing.assert_array_equal(step.accept_path.cpu().numpy(), opath)
    np.testing.assert_array_equal(step.bonus.cpu().numpy(), obonus)
    # attention with the GPU's mask
    seqs = None if pairs is None else sorted({p[0] for p in pairs})
    gout = step.attn_out.float().cpu().numpy()
    f64 = lambda x: x.double().numpy()
    if pairs is None:
        oout, _ = O.tree_attention(f64(att["q"]), f64(att["k_cache"]), f64(att["v_cache"]), kv,
                                   f64(att["k_tree"]), f64(att["v_tree"]), gmask, g["n_nodes"])
        assert np.abs(gout - oout).max() <= ATTN_TOL
    else:
        G = w.Hq // w.Hkv
        for (bq, hk) in pairs:
            oout, _ = O.tree_attention(f64(att["q"][bq:bq + 1]), f64(att["k_cache"][bq:bq + 1]),
                                       f64(att["v_cache"][bq:bq + 1]), kv[bq:bq + 1],
                                       f64(att["k_tree"][bq:bq + 1]), f64(att["v_tree"][bq:bq + 1]),
                                       gmask[bq:bq + 1], g["n_nodes"][bq:bq + 1], kv_heads=[hk])
            err = np.abs(gout[bq, :, hk * G:(hk + 1) * G] - oout[0, :, hk * G:(hk + 1) * G]).max()
            assert err <= ATTN_TOL, (bq, hk, err)


def test_back_to_back_rounds_on_rotating_inputs():
    """Rounds replayed back to back with no host synchronisation, rotating three input
    sets (so any round's tree and mask differ from those of the two rounds before it):
    the last round of each ordering matches the oracle step by step.  Kernels of a dependent-launch chain
    start while earlier ones still run, so this checks that no kernel reads a
    previous round's tree, mask or candidates."""
    w = synth.WORKLOADS["qwen3_8b"]
    dev = "cuda"
    a, b, t, lr = synth.trigram_entries(w)
    ngram = P.Ngram3Table.from_entries(a, b, t, lr, w.table_log2_cap, w.miss_logrho, device=dev)
    table = O.make_table(a, b, t, lr)
    step = P.DraftVerifyStep(w.B, w.L, w.V, w.k, w.N, w.Hq, w.Hkv, w.D, w.T,
                             logits_dtype=torch.bfloat16, b=w.branching, lam=w.lam, ngram=ngram,
                             device=dev)
    sets = []
    for s in range(3):
        ws = w.scaled(seed=w.seed * 1000 + s + 1) if s else w
        att = synth.attention_inputs(ws, device="cpu")
        kv = att.pop("kv_len").to(torch.int32)
        st = {"logits": synth.drafter_logits(ws), "ctx": synth.ctx_tokens(w), "att": att, "kv": kv,
              "target": torch.zeros(w.B, w.N, dtype=torch.int32, device=dev)}
        st["dev"] = {"logits": st["logits"].to(dev), "ctx": st["ctx"].to(dev),
                     "layer": {k: v.to(dev) for k, v in att.items()}, "kv": kv.to(dev)}
        step.run(st["dev"]["logits"], st["dev"]["ctx"], [st["dev"]["layer"]], st["dev"]["kv"],
                 st["target"])
        torch.cuda.synchronize()
        tree = {k: v.cpu().numpy() for k, v in step.tree.items()}
        st["target"].copy_(synth.target_tokens(w, st["logits"], tree["token"], tree["parent"],
                                               tree["n_nodes"]))
        sets.append(st)
    graphs = [step.capture(st["dev"]["logits"], st["dev"]["ctx"], [st["dev"]["layer"]],
                           st["dev"]["kv"], st["target"]) for st in sets]
    f64 = lambda x: x.double().numpy()
    for order in ((0, 1, 2), (1, 2, 0), (2, 0, 1)):
        step.dev_status.zero_()
        for _ in range(8):
            for i in order:
                graphs[i].replay()
        torch.cuda.synchronize()
        assert int(step.dev_status.item()) == 0
        st = sets[order[-1]]
        R = w.rows
        oids, ologq, _ = O.topk_logsoftmax(st["logits"].reshape(R, w.V).double().numpy(), w.k)
        gids = step.topk_ids.cpu().numpy().reshape(R, w.k)
        np.testing.assert_array_equal(gids, oids)
        g = {k: v.cpu().numpy() for k, v in step.tree.items()}
        glogq = step.topk_logq.cpu().numpy().astype(np.float64).reshape(w.B, w.L, w.k)
        o = O.best_first_tree(gids.astype(np.int64).reshape(w.B, w.L, w.k), glogq,
                              st["ctx"].numpy(), table, w.miss_logrho, w.lam, w.branching, w.N,
                              "fp32")
        for key in ("token", "parent", "depth", "n_nodes"):
            np.testing.assert_array_equal(g[key], o[key], err_msg=key)
        omask, _ = O.tree_mask(g["parent"], g["depth"], g["n_nodes"], st["kv"].numpy(), w.N)
        gmask = step.mask.cpu().numpy().view(np.uint32)
        np.testing.assert_array_equal(gmask, omask)
        oacc, opath, obonus = O.accept(g["token"], g["parent"], g["n_nodes"],
                                       st["target"].cpu().numpy(), w.L)
        np.testing.assert_array_equal(step.accept_len.cpu().numpy(), oacc)
        np.testing.assert_array_equal(step.accept_path.cpu().numpy(), opath)
        oout, _ = O.tree_attention(f64(st["att"]["q"]), f64(st["att"]["k_cache"]),
                                   f64(st["att"]["v_cache"]), st["kv"].numpy(),
                                   f64(st["att"]["k_tree"]), f64(st["att"]["v_tree"]), gmask,
                                   g["n_nodes"])
        assert np.abs(step.attn_out.float().cpu().numpy() - oout).max() <= ATTN_TOL, order
