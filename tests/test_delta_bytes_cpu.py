"""Pins of the oracle's touched-byte counters for anti-entropy ops (``OTree.apply_ops_counted`` and
``oracle.delta_touched_bytes``), the algorithmic bytes of the delta kernel's roofline: a hand-worked pair of
ops, and agreement of the counted apply with the plain apply on a generated delta."""
import numpy as np

import oracle
import workload as wl
from gpu_util import seqlist_from_lists


def test_hand_worked_counters():
    t = oracle.OTree()
    t.insert([1, 2, 3])
    ops = np.array([0, 1], np.int32)  # INSERT [1, 2, 4], then DELETE [1, 2, 3]
    sl = seqlist_from_lists([[1, 2, 4], [1, 2, 3]])
    c = np.zeros(8, np.int64)
    assert t.apply_ops_counted(ops, sl, c) == 0
    # INSERT: the root has 1 child (4 B of search), edge [1, 2, 3] is visited, 1 and 2 match and the
    # mismatching 4 is compared too (3 tokens); match 2, so 1 new label token.  DELETE: after the split the
    # root's child [1, 2] matches fully (2 tokens), the node [1, 2] has 2 children (4 * ceil(log2 3) = 8 B),
    # edge [3] matches (1 token); 3 nodes visited with the root.
    assert c.tolist() == [3 + 3, 2 + 3, 4 + 4 + 8, 6, 2, 1, 1, 1]
    # Input 12 B per op + 12 B per run + 4 B per token = 24 + 24 + 24; walk 4*6 + 20*5 + 16 = 140; writes: the
    # INSERT's new token and node (4 + 36), the DELETE's node record (16).
    assert oracle.delta_touched_bytes(c) == 72 + 140 + 56
    assert t.export()["labels"].tolist() == [1, 2, 4]


def test_counted_apply_is_the_plain_apply():
    prm = wl.preset(0)
    prm.update(P=2, n_seq=300, n_prefix=10)
    W = wl.Workload(params=prm, seed=3)
    a, b = oracle.OTree(), oracle.OTree()
    a.insert_seqlist(W.tree(1))
    b.insert_seqlist(W.tree(1))
    W.delta_make(0, 0.1, 0.1)
    d = W.delta()
    lo, hi = int(d.peer_begin[1]), int(d.peer_begin[2])
    c = np.zeros(8, np.int64)
    assert a.apply_ops_counted(d.op, d.seqs, c, lo, hi) == b.apply_ops(d.op, d.seqs, lo, hi)
    ea, eb = a.export(), b.export()
    assert all(np.array_equal(ea[k], eb[k]) for k in ea)
    assert c[5] + c[7] == hi - lo and c[6] <= c[3]
