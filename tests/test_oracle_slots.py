"""Pins of the oracle's self-speculative slot gather (App. C (II)): the next
round's drafter rows come from the mask slots of the deepest accepted node, and
from no other node's slots."""

import numpy as np
import pytest

from oracle import presto_oracle as O


def _figure_tree():
    """The walk-through of App. C (I)-(II) (Fig. 3): root D with children E and F,
    F with child G.  The target continues D -> F -> G' (G' != G), so F is accepted,
    G and E are rejected, and G' is the bonus token."""
    D, E, F, G, Gp, X = 10, 11, 12, 13, 20, 21
    token = np.array([[D, E, F, G]])
    parent = np.array([[-1, 0, 0, 2]])
    target = np.array([[F, X, Gp, X]])      # the target's next token after each node
    return token, parent, target, (D, E, F, G, Gp)


def test_figure_walkthrough_reads_the_slots_after_f():
    token, parent, target, (D, E, F, G, Gp) = _figure_tree()
    acc, path, bonus = O.accept(token, parent, [4], target, 3)
    assert acc[0] == 1 and list(path[0][:2]) == [0, 2] and bonus[0] == Gp
    n_slots, V = 3, 64
    x = np.zeros((1, 4, n_slots, V))
    for i in range(4):
        for j in range(n_slots):
            x[0, i, j, i * n_slots + j] = 5.0          # slot (i, j) peaks at token i*S + j
    rows = O.accepted_slot_rows(x, acc, path, 1, 2)
    ids, _, _ = O.topk_logsoftmax(rows.reshape(2, V), 1)
    assert list(ids[:, 0]) == [2 * n_slots + 1, 2 * n_slots + 2]   # F's slots 1 and 2
    np.testing.assert_array_equal(O.next_context(token, acc, path, bonus), [[F, Gp]])


def test_nothing_accepted_reads_the_root_slots():
    token, parent, target, _ = _figure_tree()
    target = target.copy()
    target[0, 0] = 99                               # no child of D matches
    acc, path, bonus = O.accept(token, parent, [4], target, 3)
    x = np.random.default_rng(0).normal(size=(1, 4, 4, 32))
    rows = O.accepted_slot_rows(x, acc, path, 0, 4)
    np.testing.assert_array_equal(rows[0], x[0, 0])
    np.testing.assert_array_equal(O.next_context(token, acc, path, bonus), [[token[0, 0], 99]])


def test_rejected_branch_slots_do_not_matter():
    rng = np.random.default_rng(1)
    B, n_prev, S, V, L = 3, 9, 5, 40, 3
    acc = np.array([0, 2, 1])
    path = np.full((B, 4), -1)
    path[0, :1] = [0]
    path[1, :3] = [0, 3, 7]
    path[2, :2] = [0, 5]
    x = rng.normal(size=(B, n_prev, S, V))
    base = O.accepted_slot_rows(x, acc, path, 2, L)
    keep = {0: 0, 1: 7, 2: 5}
    y = x.copy()
    for b in range(B):
        for i in range(n_prev):
            if i != keep[b]:
                y[b, i] = rng.normal(size=(S, V))
    np.testing.assert_array_equal(O.accepted_slot_rows(y, acc, path, 2, L), base)
    y = x.copy()
    y[1, 7, 2] += 1.0                               # the accepted node's first used slot
    assert not np.array_equal(O.accepted_slot_rows(y, acc, path, 2, L), base)
    for b in range(B):                              # brute force: the row's source slot
        for j in range(L):
            np.testing.assert_array_equal(base[b, j], x[b, keep[b], 2 + j])


def test_slot_gather_rejects_out_of_range():
    x = np.zeros((1, 2, 3, 4))
    with pytest.raises(ValueError):
        O.accepted_slot_rows(x, [0], [[0, -1]], 2, 2)       # slots 2, 3 of 3
    with pytest.raises(ValueError):
        O.accepted_slot_rows(x, [2], [[0, 1]], 0, 1)        # accept_len beyond the path
    with pytest.raises(ValueError):
        O.accepted_slot_rows(x, [1], [[0, 5]], 0, 1)        # node beyond the tree
