"""presto_topk_slots (GPU, C ABI) vs the oracle: the next round's drafter rows
read from the mask slots of the deepest accepted node (App. C (II)).  Ids exact,
log q and lse within 1e-5 * max(1, |x|), ctx2_next exact; the slots of every
other node never influence the result."""

import numpy as np
import pytest
import torch

import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import (GPU, LOGQ_TOL, assert_tree_close, rel_close, synthetic_candidates,
                        to_dev, tree_host)

pytestmark = GPU


def _random_tree(rng, B, N, V):
    """Parents before children, distinct sibling tokens; token 0..V-1."""
    token = np.full((B, N), -1, np.int64)
    parent = np.full((B, N), -1, np.int64)
    n_nodes = rng.integers(1, N + 1, B)
    for b in range(B):
        token[b, 0] = rng.integers(V)
        used = {}
        for i in range(1, n_nodes[b]):
            p = int(rng.integers(i))
            t = int(rng.integers(V))
            while t in used.setdefault(p, set()):
                t = int(rng.integers(V))
            used[p].add(t)
            parent[b, i], token[b, i] = p, t
    return token, parent, n_nodes


def _depths(parent, n_nodes):
    B, N = parent.shape
    depth = np.full((B, N), -1, np.int64)
    for b in range(B):
        depth[b, 0] = 0
        for i in range(1, n_nodes[b]):
            depth[b, i] = depth[b, parent[b, i]] + 1
    return depth


def _planted_targets(rng, token, parent, n_nodes, V):
    """target_token[b, i]: random, except along the root path of one random node,
    which the target follows."""
    B, N = token.shape
    tgt = rng.integers(V, size=(B, N))
    for b in range(B):
        a = int(rng.integers(n_nodes[b]))
        while a > 0:
            tgt[b, parent[b, a]] = token[b, a]
            a = int(parent[b, a])
    return tgt


def _slot_logits(B, n_prev, S, V, dtype, seed):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(B, n_prev, S, V, generator=g) * 3).to(dtype)


def _oracle(x_cpu, acc, path, off, L, k, token, bonus):
    rows = O.accepted_slot_rows(x_cpu.double().numpy(), acc, path, off, L)
    B, _, _, V = x_cpu.shape
    ids, logq, lse = O.topk_logsoftmax(rows.reshape(B * L, V), k)
    return ids, logq, lse, O.next_context(token, acc, path, bonus)


@pytest.mark.parametrize("B,N,S,V,L,off,k,dtype", [
    (3, 20, 9, 4099, 8, 1, 4, torch.float32),
    (4, 64, 17, 1001, 16, 1, 6, torch.bfloat16),      # unaligned rows: head/tail scalars
    (2, 8, 33, 151936, 32, 1, 6, torch.bfloat16),     # the self-speculative shape, L = 32
    (5, 16, 4, 777, 4, 0, 3, torch.float32),          # slots start at the node itself
    (1, 1, 2, 5000, 1, 1, 1, torch.bfloat16),         # a root-only tree
])
def test_slot_topk_matches_oracle(B, N, S, V, L, off, k, dtype):
    rng = np.random.default_rng(B * 100 + N + S + V)
    token, parent, n_nodes = _random_tree(rng, B, N, V)
    depth = _depths(parent, n_nodes)
    tgt = _planted_targets(rng, token, parent, n_nodes, V)
    Lp = int(depth.max())
    acc, path, bonus = O.accept(token, parent, n_nodes, tgt, Lp)
    x = _slot_logits(B, N, S, V, dtype, seed=V + S)
    xd = x.cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ids, logq, lse, ctx2 = P.presto_topk_slots(xd, to_dev(acc), to_dev(path), off, L, k,
                                               node_token=to_dev(token), bonus=to_dev(bonus),
                                               dev_status=st)
    torch.cuda.synchronize()
    oids, ologq, olse, octx = _oracle(x, acc, path, off, L, k, token, bonus)
    assert int(st.item()) == 0
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(B * L, k), oids)
    assert rel_close(logq.cpu().numpy().reshape(B * L, k), ologq) <= LOGQ_TOL
    assert rel_close(lse.cpu().numpy().reshape(-1), olse) <= LOGQ_TOL
    np.testing.assert_array_equal(ctx2.cpu().numpy(), octx)
    # the other nodes' slots do not matter: overwrite them on the device, same result
    a_star = O.accepted_node(acc, path)
    for b in range(B):
        others = [i for i in range(N) if i != a_star[b]]
        if others:
            xd[b, others] = torch.finfo(dtype).max / 4
    ids2, logq2, lse2, _ = P.presto_topk_slots(xd, to_dev(acc), to_dev(path), off, L, k)
    torch.cuda.synchronize()
    assert torch.equal(ids2, ids) and torch.equal(logq2, logq) and torch.equal(lse2, lse)


def test_accept_then_slot_topk_on_one_stream():
    """build -> mask -> accept -> topk_slots -> build of the next round, all on the
    device with no host sync in between, vs the oracle's chain (decisions in
    float32, marginal-only scoring as in the self-speculative setting)."""
    rng = np.random.default_rng(8)
    B, L, k, N, V, S = 4, 12, 5, 96, 3001, 13
    vocab = rng.choice(V, 400, replace=False)
    ids, logq = synthetic_candidates(rng, B, L, k, V, vocab=vocab)
    ctx = rng.choice(vocab, size=(B, 2))
    out = P.presto_score_build_tree(to_dev(ids), to_dev(logq, torch.float32), to_dev(ctx), None,
                                    0.0, N)
    mask, pos = P.presto_tree_mask(out["parent"], out["depth"], out["n_nodes"],
                                   torch.zeros(B, dtype=torch.int32, device="cuda"))
    o = O.best_first_tree(ids, logq, ctx, None, -12.0, 0.0, k, N, "fp32")
    tgt = _planted_targets(rng, o["token"], o["parent"], o["n_nodes"], V)
    acc_d, path_d, bonus_d = P.presto_accept(out["token"], out["parent"], out["depth"], mask,
                                             out["n_nodes"], to_dev(tgt), L)
    x = _slot_logits(B, N, S, V, torch.bfloat16, seed=4)
    nids, nlogq, _, ctx2 = P.presto_topk_slots(x.cuda(), acc_d, path_d, 1, L, k,
                                               node_token=out["token"], bonus=bonus_d)
    nxt = P.presto_score_build_tree(nids, nlogq, ctx2, None, 0.0, N)
    g = tree_host(nxt)
    acc, path, bonus = O.accept(o["token"], o["parent"], o["n_nodes"], tgt, L)
    oids, ologq, _, octx = _oracle(x, acc, path, 1, L, k, o["token"], bonus)
    np.testing.assert_array_equal(acc_d.cpu().numpy(), acc)
    np.testing.assert_array_equal(ctx2.cpu().numpy(), octx)
    np.testing.assert_array_equal(nids.cpu().numpy().reshape(B * L, k), oids)
    assert rel_close(nlogq.cpu().numpy().reshape(B * L, k), ologq) <= LOGQ_TOL
    # the next tree against the oracle's float64 tree from the oracle's own log q
    assert_tree_close(g, oids.reshape(B, L, k), ologq.reshape(B, L, k), octx, None, -12.0, 0.0, N)


def test_bad_accept_path_is_reported_and_reads_the_root():
    B, N, S, V, L, k = 2, 4, 3, 300, 2, 2
    x = _slot_logits(B, N, S, V, torch.float32, seed=1)
    acc = np.array([5, 1])                     # sequence 0: beyond the path
    path = np.array([[0, 2, -1], [0, 9, -1]])  # sequence 1: node 9 of 4
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ids, _, _, _ = P.presto_topk_slots(x.cuda(), to_dev(acc), to_dev(path), 0, L, k, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x200
    root = O.accepted_slot_rows(x.double().numpy(), [0, 0], [[0, -1, -1], [0, -1, -1]], 0, L)
    oids, _, _ = O.topk_logsoftmax(root.reshape(B * L, V), k)
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(B * L, k), oids)


def test_slot_topk_many_rows_stream():
    """B * L rows beyond one wave of the register-resident kernel: slot rows through
    the streaming kernel."""
    rng = np.random.default_rng(21)
    B, N, S, V, L, k = 12, 4, 33, 151936, 32, 6
    token, parent, n_nodes = _random_tree(rng, B, N, V)
    depth = _depths(parent, n_nodes)
    tgt = _planted_targets(rng, token, parent, n_nodes, V)
    acc, path, bonus = O.accept(token, parent, n_nodes, tgt, int(depth.max()))
    x = _slot_logits(B, N, S, V, torch.bfloat16, seed=99)
    ids, logq, lse, ctx2 = P.presto_topk_slots(x.cuda(), to_dev(acc), to_dev(path), 1, L, k,
                                               node_token=to_dev(token), bonus=to_dev(bonus))
    torch.cuda.synchronize()
    oids, ologq, olse, octx = _oracle(x, acc, path, 1, L, k, token, bonus)
    np.testing.assert_array_equal(ids.cpu().numpy().reshape(B * L, k), oids)
    assert rel_close(logq.cpu().numpy().reshape(B * L, k), ologq) <= LOGQ_TOL
    assert rel_close(lse.cpu().numpy().reshape(-1), olse) <= LOGQ_TOL
    np.testing.assert_array_equal(ctx2.cpu().numpy(), octx)
