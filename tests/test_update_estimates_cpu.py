"""Pins of the oracle's UpdateTrieEstimate over a routed batch (``oracle.update_estimates``): afterwards
every routed request is matched in full by the tree it went to, every tree's multiset grew by exactly the
requests routed to it (the canonical export equals a fresh build of the old sequences plus those
requests), and unrouted requests change nothing."""
import numpy as np

import oracle
import workload as wl


def _seqs(sl):
    """The sequences of a segmented list: each is the concatenation of its pool runs."""
    out = []
    for i in range(len(sl.seg_begin) - 1):
        s = []
        for g in range(int(sl.seg_begin[i]), int(sl.seg_begin[i + 1])):
            s += list(sl.pool[int(sl.seg_off[g]):int(sl.seg_off[g]) + int(sl.seg_len[g])])
        out.append(s)
    return out


def test_routed_requests_are_added_to_their_targets():
    prm = wl.preset(0)
    prm.update(P=5, n_seq=150, n_prefix=10, B=400)
    W = wl.Workload(params=prm, seed=31)
    sls = [W.tree(p) for p in range(W.P)]
    trees = oracle.build_trees(sls)
    tok, off = W.requests()
    load = W.load()
    _, peer, _ = oracle.route(trees, tok, off, load, W.alpha)
    peer = peer.copy()
    peer[::7] = -1  # some requests have no target
    oracle.update_estimates(trees, tok, off, peer)
    reqs = [tok[int(off[b]):int(off[b + 1])] for b in range(W.B)]
    for b in range(W.B):
        if peer[b] >= 0:
            assert trees[peer[b]].match(reqs[b]) == len(reqs[b])
    for p in range(W.P):
        fresh = oracle.OTree()
        for s in _seqs(sls[p]):
            fresh.insert(s)
        for b in range(W.B):
            if peer[b] == p:
                fresh.insert(reqs[b])
        a, e = trees[p].export(), fresh.export()
        assert all(np.array_equal(a[k], e[k]) for k in e), p
