"""One round of the draft-and-verify hot path with resident buffers.

`DraftVerifyStep` owns every intermediate and workspace of a round for fixed
shapes, so a round is a few library calls with no allocation:

    presto_topk -> presto_score_build_tree_mask (tree, mask and position ids)
      -> presto_tree_attention (x layers) -> presto_accept

(or, with fuse_mask=False, presto_score_build_tree then presto_tree_mask), and can
be captured once into a CUDA graph and replayed.
"""

from __future__ import annotations

import torch

from . import _lib as P


class DraftVerifyStep:
    def __init__(self, B, L, V, k, N, Hq, Hkv, D, Tmax, logits_dtype=torch.bfloat16,
                 b=None, lam=0.2, ngram=None, device="cuda", fuse_mask=True):
        self.B, self.L, self.V, self.k, self.N = B, L, V, k, N
        self.Hq, self.Hkv, self.D, self.Tmax = Hq, Hkv, D, Tmax
        self.b = k if b is None else b
        self.lam = lam
        self.ngram = ngram
        self.device = torch.device(device)
        i32, f32, bf = torch.int32, torch.float32, torch.bfloat16
        dev = self.device
        W = (N + 31) // 32
        self.topk_ids = torch.empty(B, L, k, dtype=i32, device=dev)
        self.topk_logq = torch.empty(B, L, k, dtype=f32, device=dev)
        self.lse = torch.empty(B, L, dtype=f32, device=dev)
        self.tree = {"token": torch.empty(B, N, dtype=i32, device=dev),
                     "parent": torch.empty(B, N, dtype=i32, device=dev),
                     "depth": torch.empty(B, N, dtype=i32, device=dev),
                     "score": torch.empty(B, N, dtype=f32, device=dev),
                     "n_nodes": torch.empty(B, dtype=i32, device=dev)}
        self.mask = torch.empty(B, N, W, dtype=i32, device=dev)
        self.pos_ids = torch.empty(B, N, dtype=i32, device=dev)
        self.attn_out = torch.empty(B, N, Hq, D, dtype=bf, device=dev)
        self.attn_lse = torch.empty(B, N, Hq, dtype=f32, device=dev)
        # the round's results, contiguous so that one copy brings them to the host:
        # accept_len [B], accept_path [B, L + 1], bonus [B]
        self.result = torch.empty(B * (L + 3), dtype=i32, device=dev)
        self.accept_len = self.result[:B]
        self.accept_path = self.result[B:B + B * (L + 1)].view(B, L + 1)
        self.bonus = self.result[B + B * (L + 1):]
        self.dev_status = torch.zeros(1, dtype=i32, device=dev)
        u8 = torch.uint8
        self.ws_topk = torch.empty(max(P.presto_topk_workspace(B, L, V, k), 1), dtype=u8, device=dev)
        self.ws_build = torch.empty(max(P.presto_build_workspace(B, L, k, N), 1), dtype=u8, device=dev)
        self.ws_attn = torch.empty(max(P.presto_attn_workspace(B, N, Hq, Hkv, D, Tmax), 1),
                                   dtype=u8, device=dev)
        self.attn_launches = P.presto_attn_launches(B, N, Hq, Hkv, D, Tmax)
        self.graph = None
        self.fuse_mask = fuse_mask
        self.CALLS = (("topk", "build", "attention", "accept") if fuse_mask
                      else ("topk", "build", "mask", "attention", "accept"))

    def run(self, logits, ctx2, layers, kv_len, target_token, stream=None, marks=None,
            only=None):
        """One round.  `layers` is a list of dicts with q, k_cache, v_cache, k_tree,
        v_tree (one per attention layer).  Results stay in the step's buffers.
        `marks` (optional) maps a call name to a (start, end) pair of CUDA events
        recorded around that call on the launch stream.  `only` (optional) names
        the calls to make; the others are skipped and their results are whatever
        the buffers hold from an earlier round (for timing one call alone)."""
        s = torch.cuda.current_stream(self.device) if stream is None else stream

        def mark(name, i):
            if marks is not None and name in marks:
                marks[name][i].record(s)

        def on(name):
            return only is None or name in only

        if on("topk"):
            mark("topk", 0)
            P.presto_topk(logits, self.k, self.topk_ids, self.topk_logq, self.lse, ws=self.ws_topk,
                          dev_status=self.dev_status, stream=s)
            mark("topk", 1)
        if on("build"):
            mark("build", 0)
            fused = dict(kv_len=kv_len, mask=self.mask, pos_ids=self.pos_ids) if self.fuse_mask else {}
            P.presto_score_build_tree(self.topk_ids, self.topk_logq, ctx2, self.ngram, self.lam,
                                      self.N, b=self.b, out=self.tree, ws=self.ws_build,
                                      dev_status=self.dev_status, stream=s, **fused)
            mark("build", 1)
        if on("mask") and not self.fuse_mask:
            mark("mask", 0)
            P.presto_tree_mask(self.tree["parent"], self.tree["depth"], self.tree["n_nodes"], kv_len,
                               self.mask, self.pos_ids, dev_status=self.dev_status, stream=s)
            mark("mask", 1)
        if on("attention"):
            mark("attention", 0)
            for lay in layers:
                P.presto_tree_attention(lay["q"], lay["k_cache"], lay["v_cache"], kv_len,
                                        lay["k_tree"], lay["v_tree"], self.mask,
                                        self.tree["n_nodes"], out=self.attn_out, lse=self.attn_lse,
                                        ws=self.ws_attn, dev_status=self.dev_status, stream=s)
            mark("attention", 1)
        if on("accept"):
            mark("accept", 0)
            P.presto_accept(self.tree["token"], self.tree["parent"], self.tree["depth"], self.mask,
                            self.tree["n_nodes"], target_token, self.L, self.accept_len,
                            self.accept_path, self.bonus, dev_status=self.dev_status, stream=s)
            mark("accept", 1)

    def kernels_per_round(self, n_layers=1):
        """Library kernels one round launches: top-k, tree build (with the mask when
        fused, else a mask kernel too), accept and, per layer, the attention kernels
        (one, or two when a second kernel merges the KV splits)."""
        return (3 if self.fuse_mask else 4) + n_layers * self.attn_launches

    def capture(self, logits, ctx2, layers, kv_len, target_token):
        """Capture one round on these exact input tensors into a CUDA graph."""
        s = torch.cuda.Stream(device=self.device)
        s.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(s):
            self.run(logits, ctx2, layers, kv_len, target_token, stream=s)  # warm, outside graph
        torch.cuda.current_stream(self.device).wait_stream(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            self.run(logits, ctx2, layers, kv_len, target_token, stream=s)
        return g


class StagedRounds:
    """Rounds fed from pinned host memory, one round in flight ahead of the host.

    One round's inputs (the tensors of `example`, e.g. logits, context, target
    tokens and each layer's q and tree K/V; the KV cache stays resident) are packed
    into one contiguous 256-byte-aligned layout.  Two device staging buffers hold
    that layout, and one CUDA graph of the round is captured per buffer.  `run(i)`
    queues round i + 1 (its inputs copied in on a copy stream while round i
    computes, its graph queued behind round i, its results queued for a copy back)
    and then waits for round i's results, so that the GPU never idles while the
    host wakes up and launches: this is the schedule of a server that alternates
    two independent groups of requests, whose rounds do not wait on each other's
    results.  Every round still moves its own inputs in and its results out.

    With a fixed pool of pinned host buffers (`fuse`), each round's step is one graph
    replay: the round, the copy of its results out and, on a second stream beside it,
    the copy of the next round's inputs in (`start_pooled`, `run_pooled`).

    `bind(views)` maps the staged tensors (a list of device views, in the order of
    `example`) to the arguments of DraftVerifyStep.run:
    (logits, ctx2, layers, kv_len, target_token).
    """

    def __init__(self, step, example, bind):
        self.step = step
        dev = step.device
        self.shapes = [(t.shape, t.dtype) for t in example]
        self.offs, pos = [], 0
        for t in example:
            self.offs.append(pos)
            pos += -(-t.numel() * t.element_size() // 256) * 256
        self.nbytes = pos
        self.staging = [torch.empty(pos, dtype=torch.uint8, device=dev) for _ in range(2)]
        for buf in self.staging:  # the example round, so that the capture warms up on valid inputs
            for v, t in zip(self.views(buf), example):
                v.copy_(t)
        self.graphs = [step.capture(*bind(self.views(s))) for s in self.staging]
        self.bind = bind
        self.pool = None  # pooled mode (fuse): data_ptr of a pool buffer -> its index
        self.fused = {}
        self.copy_stream = torch.cuda.Stream(device=dev)
        self.result_host = [torch.empty(step.result.numel(), dtype=step.result.dtype).pin_memory()
                            for _ in range(2)]
        self.copied = [torch.cuda.Event(), torch.cuda.Event()]  # inputs in staging[s]
        self.done = [torch.cuda.Event(), torch.cuda.Event()]    # round on staging[s] finished
        self.read = [torch.cuda.Event(), torch.cuda.Event()]    # results in result_host[s]
        self.pending = None

    def views(self, buf):
        return [buf[o:o + torch.Size(sh).numel() * torch.empty(0, dtype=dt).element_size()]
                .view(dt).view(sh) for o, (sh, dt) in zip(self.offs, self.shapes)]

    def pack(self, tensors):
        """One round's inputs, packed into a new pinned host buffer."""
        hb = torch.empty(self.nbytes, dtype=torch.uint8).pin_memory()
        for v, t in zip(self.views(hb), tensors):
            v.copy_(t.cpu())
        return hb

    def _upload(self, host_buf, s):
        cs = self.copy_stream
        cs.wait_event(self.done[s])  # the round that last read staging[s] has finished
        with torch.cuda.stream(cs):
            self.staging[s].copy_(host_buf, non_blocking=True)
        self.copied[s].record(cs)

    def _launch(self, s):
        main = torch.cuda.current_stream(self.step.device)
        main.wait_event(self.copied[s])
        self.graphs[s].replay()
        self.done[s].record(main)
        self.result_host[s].copy_(self.step.result, non_blocking=True)
        self.read[s].record(main)

    def start(self, host_buf):
        """Queue the first round: its inputs into staging buffer 0, then the round."""
        self._upload(host_buf, 0)
        self._launch(0)

    def run(self, i, next_host_buf=None):
        """Queue round i + 1 from next_host_buf (if given), then wait for round i (queued
        by start() or the previous run()) and return its results on the host.  The
        returned pinned buffer is rewritten by round i + 2: copy it to keep it."""
        s = i % 2
        if next_host_buf is not None:
            self._upload(next_host_buf, s ^ 1)
            self._launch(s ^ 1)
        self.read[s].synchronize()
        return self.result_host[s]

    # ---- pooled mode: the host's inputs come from a fixed pool of pinned buffers
    def fuse(self, host_bufs):
        """Capture one CUDA graph per (pinned buffer j of a fixed pool, staging slot s): the
        round on staging[s] and the copy of its results to result_host[s], and beside
        them, on a second stream, the copy of pool buffer j into staging[s ^ 1] (the
        inputs of the round after).  start_pooled() and run_pooled() then move one round
        per graph replay, so the host's work per round is one replay and one wait."""
        dev = self.step.device
        cap = torch.cuda.Stream(device=dev)
        self.pool = {hb.data_ptr(): j for j, hb in enumerate(host_bufs)}
        cap.wait_stream(torch.cuda.current_stream(dev))
        for j, hb in enumerate(host_bufs):
            for s in (0, 1):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=cap):
                    self.copy_stream.wait_stream(cap)
                    with torch.cuda.stream(self.copy_stream):
                        self.staging[s ^ 1].copy_(hb, non_blocking=True)
                    self.step.run(*self.bind(self.views(self.staging[s])), stream=cap)
                    self.result_host[s].copy_(self.step.result, non_blocking=True)
                    cap.wait_stream(self.copy_stream)
                self.fused[(j, s)] = g
        torch.cuda.current_stream(dev).wait_stream(cap)

    def _launch_pooled(self, s, after_next):
        main = torch.cuda.current_stream(self.step.device)
        if after_next is None:  # no round after this one: the round alone
            self.graphs[s].replay()
            self.result_host[s].copy_(self.step.result, non_blocking=True)
        else:
            self.fused[(self.pool[after_next.data_ptr()], s)].replay()
        self.read[s].record(main)

    def start_pooled(self, first, second=None):
        """Queue round 0 (pool buffer `first`, copied in now) with round 1's inputs
        (pool buffer `second`) copied in beside it."""
        self.staging[0].copy_(first, non_blocking=True)
        self._launch_pooled(0, second)

    def run_pooled(self, i, after_next=None):
        """Queue round i + 1 (its inputs were copied in beside round i) with pool buffer
        `after_next` (round i + 2's inputs; None when round i + 1 is the last) copied in
        beside it, then wait for round i and return its results on the host (rewritten
        by round i + 2: copy them to keep them).  wait_pooled() collects the last round."""
        s = i % 2
        self._launch_pooled(s ^ 1, after_next)
        self.read[s].synchronize()
        return self.result_host[s]

    def wait_pooled(self, i):
        """Wait for round i, the last one queued, and return its results."""
        self.read[i % 2].synchronize()
        return self.result_host[i % 2]
