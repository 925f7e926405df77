"""Plain CPU oracle for one round of PRESTO's tree draft-and-verify step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference leg of ``bench.py`` may import this module.  It shares
no code with the CUDA library (``paper_2607_22634_gb300``) and never calls it.

Each function states the part of the paper it follows.  Arithmetic is float64
unless a function says otherwise.  The paper fixes no precision for the tree
search; its decisions (which nodes enter the tree, in what order) are integers
that floating point decides, so ``best_first_tree`` can take them in float32 with
the same operation order as the CUDA kernel (``precision="fp32"``), or in float64.

Readings taken where the paper is silent (each is also listed in the design notes):

R1  Ties in top-k selection go to the lower token id.
R2  The trigram context of depth d is the last two tokens of
    (committed context ++ path), so depths 1 and 2 reach back into the two
    committed tokens ``ctx[b, 0], ctx[b, 1]`` (ctx[b, 1] is the root token).
R3  A missing trigram gives the table's ``miss_logrho``.  With no table
    (marginal-only scoring) s = log q exactly.
R4  float32 token score: s = fl(fl(lambda * logrho) + logq) (two roundings, no
    fused multiply-add); path score S(child) = fl(S(parent) + s).
R5  Children of a node are the top-b of the next position's k candidates ranked
    by (s desc, token id asc) (§4.2 expansion step 2).
R6  Total order on nodes: S desc, then depth asc, then token id asc, then the
    parent's output index asc.  Output order is this order (so parent index <
    child index and node 0 is the root).
R7  Best-first (Alg. 2) commits a node when it is popped from the frontier
    (lazy), and stops after N commits or an empty frontier.  With s <= 0 this is
    exactly the top-N prefix-closed set of §4.2 ("the optimal tree consists of
    the B prefixes with the largest S").  Alg. 2 as printed adds all b children
    to the tree at expansion time, which can keep a shallow low-score child over
    a deeper high-score one; ``eager_tree`` computes that variant.
R8  Tree attention: softmax(scale * q k^T) v over every committed prefix key plus
    the tree keys that are ancestors-or-self of the query node; scale = 1/sqrt(D)
    unless given; no soft-cap; rows of unused node slots are zero with lse = -inf.
R9  Acceptance (§2.1, App. A alpha_T(P)): the deepest node whose root path is
    the target's greedy continuation; the bonus token is the target's token after
    that node.
R10 Beam search (Alg. 1): TopW and TopB use the total order R6; the loop runs
    while |T| < N, counting every node added to T (root included); a depth whose
    beam is empty ends the search.
"""

from __future__ import annotations

import heapq
import math

import numpy as np

F32 = np.float32


# ---------------------------------------------------------------------------
# Step 1: per-position log-softmax and top-k (§2.3 marginals q_d; §4.3 top-k
# diffusion candidates; §5.1 k = 10).
# ---------------------------------------------------------------------------

def topk_logsoftmax(logits, k: int):
    """Top-k candidates of each row with their log-marginals.

    logits: array [R, V] of finite values (bf16/fp32 inputs convert exactly).
    Returns ids int64 [R, k] (descending value, ties -> lower id, R1),
    logq float64 [R, k] = x - lse, and lse float64 [R] = log sum_v exp(x_v).
    """
    x = np.asarray(logits, dtype=np.float64)
    R, V = x.shape
    if not 1 <= k <= V:
        raise ValueError("need 1 <= k <= V")
    m = x.max(axis=1)
    lse = m + np.log(np.exp(x - m[:, None]).sum(axis=1))
    ids = np.empty((R, k), np.int64)
    for r in range(R):
        ids[r] = np.argsort(-x[r], kind="stable")[:k]
    logq = np.take_along_axis(x, ids, axis=1) - lse[:, None]
    return ids, logq, lse


def drafter_entropy(logits):
    """H_d = -sum_w q_d(w) log q_d(w) of each row (App. F), q_d the softmax of the
    row (§2.3 marginal).  Entries of -inf have q = 0 and add nothing (0 log 0 = 0).

    logits: array [R, V] of finite values or -inf, each row with a finite entry.
    Returns float64 [R] in nats.
    """
    x = np.asarray(logits, dtype=np.float64)
    m = x.max(axis=1, keepdims=True)
    z = x - m
    e = np.exp(z)
    Z = e.sum(axis=1)
    logq = z - np.log(Z)[:, None]
    q = e / Z[:, None]
    with np.errstate(invalid="ignore"):
        terms = np.where(q > 0.0, q * logq, 0.0)
    return -terms.sum(axis=1)


def entropy_adaptive_lambda(H, beta: float, C: float):
    """lambda_d(H_d) = beta * H_d / (H_d + C) (App. F; beta > 0 the largest
    correction strength, C > 0 the stabilising constant).  float64."""
    if not (beta > 0 and C > 0):
        raise ValueError("need beta > 0 and C > 0")
    H = np.asarray(H, dtype=np.float64)
    return beta * H / (H + C)


# ---------------------------------------------------------------------------
# Step 2: prefix-aligned token score (§4.1, Eq. prefix-aligned-conditional and
# Eq. path-score): s_{d,t}(c_d) = log q_d(t) + lambda_d log rho_d(t | c_d).
# ---------------------------------------------------------------------------

def trigram_context(ctx2, path):
    """(t_{d-2}, t_{d-1}) for the child at depth len(path)+1 (R2)."""
    seq = (int(ctx2[0]), int(ctx2[1])) + tuple(int(t) for t in path)
    return seq[-2], seq[-1]


def make_table(a, b, t, logrho):
    """The trigram signal as a plain dict {(a, b, t): log rho}."""
    return {(int(x), int(y), int(z)): float(v) for x, y, z, v in zip(a, b, t, logrho)}


def token_score(logq, logrho, lam, precision: str):
    """s = log q + lambda * log rho (Eq. path-score).  logrho None: s = log q (R3)."""
    if precision == "fp64":
        return float(logq) if logrho is None else float(logq) + float(lam) * float(logrho)
    if logrho is None:
        return F32(logq)
    return F32(F32(F32(lam) * F32(logrho)) + F32(logq))          # R4


def path_add(S_parent, s, precision: str):
    """S(child) = S(parent) + s (Eq. path-score is additive over depth)."""
    if precision == "fp64":
        return float(S_parent) + float(s)
    return F32(F32(S_parent) + F32(s))                            # R4


def _lam_of(lam, b):
    """lambda of sequence b: a scalar for every row, or row b of a [B, L] array
    (App. F: a lambda_d per position)."""
    return lam[b] if np.ndim(lam) == 2 else lam


def _lam_at(lam_b, row):
    """lambda of drafter row `row` (depth row + 1)."""
    return float(lam_b[row]) if np.ndim(lam_b) == 1 else lam_b


def children(ids_b, logq_b, ctx2, table, miss, lam, bfac, path, precision):
    """Top-b children of the node with root path `path` (R5).

    Returns a list of (s, token, rank_in_topk) ordered by (s desc, token asc).
    """
    d = len(path)                         # children live at depth d+1 = drafter row d
    a, bb = trigram_context(ctx2, path)
    out = []
    for j in range(ids_b.shape[1]):
        t = int(ids_b[d, j])
        rho = None if table is None else table.get((a, bb, t), miss)
        out.append((token_score(logq_b[d, j], rho, _lam_at(lam, d), precision), t, j))
    out.sort(key=lambda e: (-float(e[0]), e[1]))
    return out[:bfac]


# ---------------------------------------------------------------------------
# Step 3: best-first tree construction (§4.2, Alg. 2, read as R6/R7).
# ---------------------------------------------------------------------------

def _empty_tree(B, N):
    return {
        "token": np.full((B, N), -1, np.int64),
        "parent": np.full((B, N), -1, np.int64),
        "depth": np.full((B, N), -1, np.int64),
        "score": np.full((B, N), -np.inf, np.float64),
        "score64": np.full((B, N), -np.inf, np.float64),
        "rank": np.full((B, N), -1, np.int64),
        "n_nodes": np.zeros(B, np.int64),
    }


def best_first_tree(ids, logq, ctx, table, miss, lam, bfac, N, precision="fp32"):
    """Best-first search over the candidate tree up to N nodes (root included).

    ids, logq: [B, L, k] top-k candidates of each drafter row (row d-1 feeds depth d).
    ctx: [B, 2] last two committed tokens; ctx[b, 1] is the root token.
    table: dict from make_table, or None for marginal-only scoring.
    precision: "fp32" takes every score and comparison in float32 (R4); "fp64" in
    float64.  ``score`` holds S in that precision; ``score64`` recomputes the same
    tree's S in float64.
    """
    ids = np.asarray(ids)
    logq = np.asarray(logq, dtype=np.float64)
    B, L, _ = ids.shape
    out = _empty_tree(B, N)
    for b in range(B):
        lam_b = _lam_of(lam, b)
        tok = [int(ctx[b][1])]
        par, dep, S, S64, rank, paths = [-1], [0], [0.0], [0.0], [-1], [()]
        frontier = []

        def expand(n):
            if dep[n] >= L:
                return
            for s, t, j in children(ids[b], logq[b], ctx[b], table, miss, lam_b, bfac,
                                    paths[n], precision):
                Sc = path_add(S[n], s, precision)
                # heapq pops the smallest tuple: the key order is R6.
                heapq.heappush(frontier, ((-float(Sc), dep[n] + 1, t, n), (Sc, j)))

        expand(0)
        while len(tok) < N and frontier:
            (negS, d, t, p), (Sc, j) = heapq.heappop(frontier)
            rho = None
            if table is not None:
                rho = table.get(trigram_context(ctx[b], paths[p]) + (t,), miss)
            tok.append(t); par.append(p); dep.append(d); S.append(Sc); rank.append(j)
            S64.append(S64[p] + token_score(logq[b, d - 1, j], rho, _lam_at(lam_b, d - 1), "fp64"))
            paths.append(paths[p] + (t,))
            expand(len(tok) - 1)
        n = len(tok)
        out["token"][b, :n] = tok
        out["parent"][b, :n] = par
        out["depth"][b, :n] = dep
        out["score"][b, :n] = [float(v) for v in S]
        out["score64"][b, :n] = S64
        out["rank"][b, :n] = rank
        out["n_nodes"][b] = n
    return out


class _Nodes:
    """Nodes of one sequence's search tree: node 0 is the root.  Each node keeps
    its root path, S in the search precision, S recomputed in float64, the rank of
    its token among the position's top-k, its depth and its parent."""

    def __init__(self, ctx2):
        self.path, self.S, self.S64, self.rank, self.parent = [()], [0.0], [0.0], [-1], [-1]
        self.root_token = int(ctx2[1])
        self._key = {}

    def add(self, parent, t, S, s64, j):
        self.path.append(self.path[parent] + (t,))
        self.S.append(S)
        self.S64.append(self.S64[parent] + s64)
        self.rank.append(j)
        self.parent.append(parent)
        return len(self.path) - 1

    def key(self, v):
        """The total order R6 without output indices: (-S, depth, token, key(parent)),
        compared lexicographically; the root's key () sorts first."""
        if v not in self._key:
            p = self.path[v]
            self._key[v] = () if not p else (-float(self.S[v]), len(p), p[-1],
                                            self.key(self.parent[v]))
        return self._key[v]

    def expand(self, v, ids_b, logq_b, ctx2, table, miss, lam, bfac, precision):
        """§4.2 expansion: add the top-b children of v (R5); returns their node ids."""
        p = self.path[v]
        if len(p) >= ids_b.shape[0]:
            return []
        a, bb = trigram_context(ctx2, p)
        out = []
        for s, t, j in children(ids_b, logq_b, ctx2, table, miss, lam, bfac, p, precision):
            rho = None if table is None else table.get((a, bb, t), miss)
            s64 = token_score(logq_b[len(p), j], rho, _lam_at(lam, len(p)), "fp64")
            out.append(self.add(v, t, path_add(self.S[v], s, precision), s64, j))
        return out

    def write(self, out, b, chosen):
        """Write the chosen node ids, sorted by the total order, as output rows."""
        order = sorted(chosen, key=self.key)
        index = {v: i for i, v in enumerate(order)}
        for i, v in enumerate(order):
            if v and self.parent[v] not in index:
                raise AssertionError("selected set is not prefix-closed")
            out["token"][b, i] = self.root_token if v == 0 else self.path[v][-1]
            out["parent"][b, i] = -1 if v == 0 else index[self.parent[v]]
            out["depth"][b, i] = len(self.path[v])
            out["score"][b, i] = float(self.S[v])
            out["score64"][b, i] = self.S64[v]
            out["rank"][b, i] = self.rank[v]
        out["n_nodes"][b] = len(order)


def beam_search_tree(ids, logq, ctx, table, miss, lam, bfac, N, W, precision="fp32"):
    """Beam search with global retention (§4.2, Alg. 1).

    P = {root}, T = {root}.  For depth d = 1..L, while |T| < N: every node of the
    beam P is expanded by its top-b children (§4.2 expansion step 2); all of them
    join T, and the W best of them (total order R6) become the next beam.  The
    result is TopB(T, N): the N best nodes of T in the order R6.  Same output arrays
    as best_first_tree.
    """
    ids = np.asarray(ids)
    logq = np.asarray(logq, dtype=np.float64)
    B, L, _ = ids.shape
    out = _empty_tree(B, N)
    for b in range(B):
        T = _Nodes(ctx[b])
        P = [0]
        for d in range(1, L + 1):
            if len(T.path) >= N or not P:
                break
            P_new = []
            for v in P:
                P_new += T.expand(v, ids[b], logq[b], ctx[b], table, miss, _lam_of(lam, b), bfac,
                                  precision)
            P = sorted(P_new, key=T.key)[:W]
        T.write(out, b, sorted(range(len(T.path)), key=T.key)[:N])
    return out


def eager_tree(ids, logq, ctx, table, miss, lam, bfac, N, precision="fp32"):
    """Alg. 2 exactly as printed (the eager variant of R7): P = {root}, T = {root};
    while |T| < N, pop the best node of P (order R6), expand it, and add its
    children to both P and T; return TopB(T, N).  Same output arrays as
    best_first_tree."""
    ids = np.asarray(ids)
    logq = np.asarray(logq, dtype=np.float64)
    B, L, _ = ids.shape
    out = _empty_tree(B, N)
    for b in range(B):
        T = _Nodes(ctx[b])
        P = [(T.key(0), 0)]
        while len(T.path) < N and P:
            _, v = heapq.heappop(P)
            for c in T.expand(v, ids[b], logq[b], ctx[b], table, miss, _lam_of(lam, b), bfac,
                              precision):
                heapq.heappush(P, (T.key(c), c))
        T.write(out, b, sorted(range(len(T.path)), key=T.key)[:N])
    return out


def candidate_tree_nodes(ids_b, logq_b, ctx2, table, miss, lam, bfac, precision):
    """Every node of the full candidate tree by explicit enumeration:
    list of (path tuple, S, ranks tuple).  S is summed from scratch along the path
    (no incremental reuse), in the given precision.  Exponential: tiny inputs only."""
    L = ids_b.shape[0]
    nodes = [((), 0.0 if precision == "fp64" else F32(0.0), ())]
    stack = [((), ())]
    while stack:
        path, ranks = stack.pop()
        if len(path) >= L:
            continue
        for s, t, j in children(ids_b, logq_b, ctx2, table, miss, lam, bfac, path, precision):
            cpath, cranks = path + (t,), ranks + (j,)
            S = 0.0 if precision == "fp64" else F32(0.0)
            for d in range(1, len(cpath) + 1):
                a, bb = trigram_context(ctx2, cpath[: d - 1])
                rho = None if table is None else table.get((a, bb, cpath[d - 1]), miss)
                S = path_add(S, token_score(logq_b[d - 1, cranks[d - 1]], rho, _lam_at(lam, d - 1),
                                            precision),
                             precision)
            nodes.append((cpath, S, cranks))
            stack.append((cpath, cranks))
    return nodes


def brute_force_tree(ids, logq, ctx, table, miss, lam, bfac, N, precision="fp32"):
    """Definition of the target tree (§4.2): the N candidate-tree nodes that come
    first in the total order R6, found by enumerating every node and sorting.

    The order's last tie-break (the parent's output index) is expressed without
    indices: key(u) = (-S(u), depth(u), token(u), key(parent(u))), compared
    lexicographically, ranks parents exactly as their output positions do.
    Same output arrays as best_first_tree.  Tiny inputs only.
    """
    ids = np.asarray(ids)
    logq = np.asarray(logq, dtype=np.float64)
    B = ids.shape[0]
    out = _empty_tree(B, N)
    for b in range(B):
        nodes = candidate_tree_nodes(ids[b], logq[b], ctx[b], table, miss, _lam_of(lam, b), bfac,
                                     precision)
        by_path = {e[0]: e for e in nodes}
        keys = {}

        def key(path):
            if path not in keys:
                S = by_path[path][1]
                keys[path] = () if not path else (-float(S), len(path), path[-1], key(path[:-1]))
            return keys[path]

        chosen = sorted(nodes, key=lambda e: key(e[0]))[:N]
        index = {e[0]: i for i, e in enumerate(chosen)}
        out["n_nodes"][b] = len(chosen)
        for i, (path, S, ranks) in enumerate(chosen):
            if path and path[:-1] not in index:
                raise AssertionError("top-N set is not prefix-closed")
            out["token"][b, i] = int(ctx[b][1]) if i == 0 else path[-1]
            out["parent"][b, i] = -1 if i == 0 else index[path[:-1]]
            out["depth"][b, i] = len(path)
            out["score"][b, i] = float(S)
            out["rank"][b, i] = -1 if i == 0 else ranks[-1]
    return out


def competing_pairs(tree, b, tol=1e-5):
    """Adjacent output positions (i, i+1) whose float64 scores lie within
    tol * max(1, |S|): near-ties whose order float rounding may decide."""
    s = tree["score64"][b]
    n = int(tree["n_nodes"][b])
    return [(i, i + 1) for i in range(1, n - 1)
            if abs(s[i] - s[i + 1]) <= tol * max(1.0, abs(s[i]))]


# ---------------------------------------------------------------------------
# Step 4: tree attention mask and position ids (§4.3 and App. C (I), (IV): each
# draft token attends to its ancestors in the draft tree and to the committed
# prefix; positions continue the committed sequence).
# ---------------------------------------------------------------------------

def tree_mask(node_parent, node_depth, n_nodes, kv_len, N):
    """mask[b, i, w] bit j set iff node j is node i or one of its ancestors
    (found by walking parent pointers); pos[b, i] = kv_len[b] + depth(i).
    Unused slots: mask row 0, pos -1."""
    node_parent = np.asarray(node_parent)
    node_depth = np.asarray(node_depth)
    B = node_parent.shape[0]
    W = (N + 31) // 32
    mask = np.zeros((B, N, W), np.uint32)
    pos = np.full((B, N), -1, np.int64)
    for b in range(B):
        for i in range(int(n_nodes[b])):
            j = i
            while j != -1:
                mask[b, i, j // 32] |= np.uint32(1 << (j % 32))
                j = int(node_parent[b, j])
            pos[b, i] = int(kv_len[b]) + int(node_depth[b, i])
    return mask, pos


def mask_to_dense(mask, N):
    """[B, N, W] bit rows -> bool [B, N, N]."""
    B = mask.shape[0]
    dense = np.zeros((B, N, N), bool)
    for j in range(N):
        dense[:, :, j] = (mask[:, :, j // 32] >> np.uint32(j % 32)) & np.uint32(1)
    return dense


# ---------------------------------------------------------------------------
# Step 5: tree-masked GQA attention (§5.1 verification with a tree-structured
# attention mask; App. C (I)).  Dense definition in float64 (R8).
# ---------------------------------------------------------------------------

def tree_attention(q, k_cache, v_cache, kv_len, k_tree, v_tree, mask, n_nodes,
                   scale=None, seqs=None, kv_heads=None):
    """out[b, i, h] = softmax_j(scale <q_{b,i,h}, k_j>) v_j over the T_b prefix keys
    of kv head g = h // (Hq/Hkv) and the tree keys j with mask bit (i, j).

    Inputs are arrays convertible to float64 (bf16 tensors are converted by the
    caller).  Returns out float64 [B, N, Hq, D] and lse float64 [B, N, Hq]
    (natural log of the softmax denominator).  `seqs` / `kv_heads` restrict the
    computation to a subset (other entries stay zero / -inf).
    """
    q = np.asarray(q, np.float64)
    B, N, Hq, D = q.shape
    Hkv = k_cache.shape[1]
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(D) if scale is None else float(scale)
    dense = mask_to_dense(np.asarray(mask), N)
    out = np.zeros((B, N, Hq, D))
    lse = np.full((B, N, Hq), -np.inf)
    for b in (range(B) if seqs is None else seqs):
        n = int(n_nodes[b])
        T = int(kv_len[b])
        for g in (range(Hkv) if kv_heads is None else kv_heads):
            Kp = np.asarray(k_cache[b, g, :T], np.float64)
            Vp = np.asarray(v_cache[b, g, :T], np.float64)
            Kt = np.asarray(k_tree[b, :n, g], np.float64)
            Vt = np.asarray(v_tree[b, :n, g], np.float64)
            for hh in range(G):
                h = g * G + hh
                Q = q[b, :n, h]                                  # [n, D]
                sp = scale * (Q @ Kp.T)                          # [n, T]
                st = scale * (Q @ Kt.T)                          # [n, n]
                st = np.where(dense[b, :n, :n], st, -np.inf)
                s = np.concatenate([sp, st], axis=1)
                m = s.max(axis=1, keepdims=True)
                p = np.exp(s - m)
                l = p.sum(axis=1, keepdims=True)
                out[b, :n, h] = (p @ np.concatenate([Vp, Vt], axis=0)) / l
                lse[b, :n, h] = (m + np.log(l))[:, 0]
    return out, lse


# ---------------------------------------------------------------------------
# Step 6: longest accepted path (§2.1 prefix acceptance; App. A alpha_T(P);
# App. C (I) bonus token).  Path-set lookup, independent of masks.
# ---------------------------------------------------------------------------

def accept(node_token, node_parent, n_nodes, target_token, L):
    """Greedy verification: follow the target's tokens from the root while the
    token path is a node of the tree.

    Returns accept_len [B], accept_path [B, L+1] (node ids root..deepest, -1
    padded) and bonus [B] (target token after the deepest accepted node).
    """
    node_token = np.asarray(node_token)
    node_parent = np.asarray(node_parent)
    target_token = np.asarray(target_token)
    B = node_token.shape[0]
    acc = np.zeros(B, np.int64)
    path_out = np.full((B, L + 1), -1, np.int64)
    bonus = np.zeros(B, np.int64)
    for b in range(B):
        n = int(n_nodes[b])
        paths = [()]
        lookup = {(): 0}
        for i in range(1, n):
            p = int(node_parent[b, i])
            if not 0 <= p < i:                  # parents precede children
                raise ValueError("parent index must be in [0, child index)")
            paths.append(paths[p] + (int(node_token[b, i]),))
            lookup[paths[-1]] = i
        cur, walk = 0, [0]
        while True:
            nxt = paths[cur] + (int(target_token[b, cur]),)
            if nxt not in lookup:
                break
            cur = lookup[nxt]
            walk.append(cur)
        acc[b] = len(paths[cur])
        path_out[b, : len(walk)] = walk
        bonus[b] = int(target_token[b, cur])
    return acc, path_out, bonus


# ---------------------------------------------------------------------------
# Step 7 (self-speculative rounds, App. C (II)): the next round's drafter rows are
# the mask slots attached to the end of the accepted path; the slots of every
# other node (rejected branches) are discarded.
# ---------------------------------------------------------------------------

def accepted_node(accept_len, accept_path):
    """a*_b = accept_path[b, accept_len[b]]: the deepest accepted node (node 0, the
    root, when nothing was accepted)."""
    accept_len = np.asarray(accept_len)
    accept_path = np.asarray(accept_path)
    out = np.empty(len(accept_len), np.int64)
    for b, n in enumerate(accept_len):
        if not 0 <= int(n) < accept_path.shape[1]:
            raise ValueError("accept_len outside the path")
        out[b] = int(accept_path[b, int(n)])
    return out


def accepted_slot_rows(slot_logits, accept_len, accept_path, slot_offset, L):
    """slot_logits [B, n_prev, n_slots, V]: the logits the self-speculative forward
    produced at the mask slots of each previous-round node.  Returns [B, L, V]:
    row j of sequence b is slot slot_offset + j of a*_b, so the slot that predicts
    the token at depth j + 1 of the next tree feeds drafter row j (slot_offset is
    the model's distance between a node and the slot of the position after the
    bonus token)."""
    x = np.asarray(slot_logits)
    B, n_prev, n_slots, V = x.shape
    if not (0 <= slot_offset and slot_offset + L <= n_slots):
        raise ValueError("slots slot_offset .. slot_offset + L - 1 must exist")
    a = accepted_node(accept_len, accept_path)
    rows = np.empty((B, L, V), x.dtype)
    for b in range(B):
        if not 0 <= a[b] < n_prev:
            raise ValueError("accepted node outside the previous tree")
        for j in range(L):
            rows[b, j] = x[b, a[b], slot_offset + j]
    return rows


def next_context(node_token, accept_len, accept_path, bonus):
    """The last two committed tokens after acceptance, the next round's ctx2: the
    token of a*_b and the bonus token (App. C (I): the position after the last
    accepted token holds the model's own prediction).  [B, 2] int64."""
    node_token = np.asarray(node_token)
    a = accepted_node(accept_len, accept_path)
    return np.array([[int(node_token[b, a[b]]), int(bonus[b])] for b in range(len(a))], np.int64)


def coverage_bound(target_fn, topk_sets, L):
    """Obs. 1 (§3): follow the target's greedy continuation and count the longest
    prefix whose token at each depth d lies in the depth-d candidate set.
    target_fn(path) -> token; topk_sets[d-1] is the candidate set of depth d."""
    path = ()
    while len(path) < L and target_fn(path) in topk_sets[len(path)]:
        path = path + (target_fn(path),)
    return len(path)
