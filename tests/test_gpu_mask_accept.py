"""presto_tree_mask and presto_accept (GPU, C ABI) vs the oracle, bit-exact, on
trees the oracle builds; plus the App. C / Fig. 3 worked example and device
status reporting for malformed trees."""

import json
import os

import numpy as np
import pytest
import torch

import synth
import paper_2607_22634_gb300 as P
from oracle import presto_oracle as O
from gpu_common import GPU, path_of, synthetic_candidates, to_dev

pytestmark = GPU
HERE = os.path.dirname(os.path.abspath(__file__))


def _oracle_tree(seed, B, L, k, N, quant=None):
    rng = np.random.default_rng(seed)
    ids, logq = synthetic_candidates(rng, B, L, k, 5000, quant=quant)
    ctx = rng.integers(0, 5000, size=(B, 2))
    return rng, ids, O.best_first_tree(ids, logq, ctx, None, 0.0, 0.0, k, N, "fp64")


def _targets(rng, ids, t, L, p_follow=0.75):
    """Target tokens that follow a random child of each node with probability p."""
    B, N = t["token"].shape
    tgt = np.full((B, N), -1, np.int64)
    for b in range(B):
        n = int(t["n_nodes"][b])
        kids = {}
        for i in range(1, n):
            kids.setdefault(int(t["parent"][b, i]), []).append(int(t["token"][b, i]))
        for i in range(n):
            if i in kids and rng.random() < p_follow:
                tgt[b, i] = rng.choice(kids[i])
            else:
                tgt[b, i] = int(rng.integers(0, 5000))
    return tgt


CASES = [(1, 8, 4, 16), (1, 16, 8, 64), (16, 16, 8, 128), (4, 32, 6, 256), (8, 16, 10, 256),
         (3, 5, 3, 40), (2, 4, 2, 1), (1, 63, 1, 64)]


@pytest.mark.parametrize("B,L,k,N", CASES)
def test_mask_and_accept_match_oracle(B, L, k, N):
    rng, ids, t = _oracle_tree(B * 100 + N, B, L, k, N)
    kv = rng.integers(0, 40000, size=B)
    mask, pos = P.presto_tree_mask(to_dev(t["parent"]), to_dev(t["depth"]), to_dev(t["n_nodes"]),
                                   to_dev(kv))
    omask, opos = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, N)
    np.testing.assert_array_equal(mask.cpu().numpy().view(np.uint32), omask)
    np.testing.assert_array_equal(pos.cpu().numpy(), opos)
    for trial in range(3):
        tgt = _targets(rng, ids, t, L)
        acc, path, bonus = P.presto_accept(to_dev(t["token"]), to_dev(t["parent"]),
                                           to_dev(t["depth"]), mask, to_dev(t["n_nodes"]),
                                           to_dev(tgt), L)
        oacc, opath, obonus = O.accept(t["token"], t["parent"], t["n_nodes"], tgt, L)
        np.testing.assert_array_equal(acc.cpu().numpy(), oacc)
        np.testing.assert_array_equal(path.cpu().numpy(), opath)
        np.testing.assert_array_equal(bonus.cpu().numpy(), obonus)


def test_accept_on_synthetic_target_model():
    w = synth.WORKLOADS["qwen3_8b"]
    x = synth.drafter_logits(w)
    oids, ologq, _ = O.topk_logsoftmax(x.reshape(w.rows, w.V).double().numpy(), w.k)
    ctx = synth.ctx_tokens(w).numpy()
    a, bb, tt, lr = synth.trigram_entries(w)
    t = O.best_first_tree(oids.reshape(w.B, w.L, w.k), ologq.reshape(w.B, w.L, w.k), ctx,
                          O.make_table(a, bb, tt, lr), w.miss_logrho, w.lam, w.k, w.N, "fp32")
    tgt = synth.target_tokens(w, x, t["token"], t["parent"], t["n_nodes"]).numpy()
    kv = synth.kv_lengths(w).numpy()
    omask, _ = O.tree_mask(t["parent"], t["depth"], t["n_nodes"], kv, w.N)
    acc, path, bonus = P.presto_accept(to_dev(t["token"]), to_dev(t["parent"]), to_dev(t["depth"]),
                                       to_dev(omask.view(np.int32)), to_dev(t["n_nodes"]),
                                       to_dev(tgt), w.L)
    oacc, opath, obonus = O.accept(t["token"], t["parent"], t["n_nodes"], tgt, w.L)
    assert acc.cpu().tolist() == oacc.tolist()
    assert path.cpu().tolist() == opath.tolist()
    assert bonus.cpu().tolist() == obonus.tolist()


def test_appc_fig3_worked_example_on_gpu():
    g = json.load(open(os.path.join(HERE, "golden", "appc_fig3_accept.json")))
    tok = np.array([g["node_token"]])
    par = np.array([g["node_parent"]])
    dep = np.array([g["node_depth"]])
    n = np.array([len(g["node_token"])])
    mask, _ = P.presto_tree_mask(to_dev(par), to_dev(dep), to_dev(n), to_dev([0]))
    acc, path, bonus = P.presto_accept(to_dev(tok), to_dev(par), to_dev(dep), mask, to_dev(n),
                                       to_dev(np.array([g["target_token"]])), g["L"])
    assert int(acc[0]) == g["expected"]["accept_len"]
    assert path[0].tolist() == g["expected"]["accept_path"]
    assert int(bonus[0]) == g["expected"]["bonus"]


def test_malformed_tree_is_reported_not_trapped():
    par = np.array([[-1, 0, 3, 1]])          # node 2 names a later parent
    dep = np.array([[0, 1, 2, 2]])
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_tree_mask(to_dev(par), to_dev(dep), to_dev([4]), to_dev([10]), dev_status=st)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.presto_tree_mask(to_dev(par), to_dev(dep), to_dev([9]), to_dev([10]), dev_status=st2)
    torch.cuda.synchronize()
    assert int(st.item()) & 0x1
    assert int(st2.item()) & 0x8
