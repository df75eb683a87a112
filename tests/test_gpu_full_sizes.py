"""GPU parity at the full sizes of the stale-replica workload (P=64, 262,144 requests) and the scale workload
(P=256 trees of 100,000 sequences, 1,048,576 requests, a 5% + 5% delta per replica per batch), in the launch
configuration the bench times.  Both are compared in full: every match value, every chosen peer, and every
patched tree byte for byte against the oracle.  The scale workload first runs anti-entropy rounds until the
delta call compacts the replicas in one wave (and one round after it), so the compaction path is compared
at full size too."""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl
from gpu_util import assert_same_route, oracle_route, same_snapshot

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    g.build()


def _route_full(router, tok, off, load, alpha):
    import torch
    t = torch.from_numpy(tok).cuda()
    o = torch.from_numpy(off).cuda()
    m, p = router.route(t, o, load, alpha)
    router.sync()
    return m.cpu().numpy(), p.cpu().numpy()


def test_stale_replica_workload_full_size():
    W = wl.Workload(2)
    r = g.Router(W.P)
    for p in range(W.P):
        r.build(p, W.tree(p, 1))  # the exact trees
    d = W.delta()  # exact -> replica for trees 1..63
    assert r.apply_delta(-1, d.op, d.seqs, d.peer_begin) == 0
    replicas = [W.tree(p, 0) for p in range(W.P)]
    trees = oracle.build_trees(replicas, n_threads=16)
    for p in (0, 1, 17, 63):
        assert same_snapshot(r.download(p), trees[p].export()), p
    tok, off = W.requests()
    gm, gp = _route_full(r, tok, off, W.load(), W.alpha)
    om, op, _ = oracle.route(trees, tok, off, W.load(), W.alpha, n_threads=16)
    assert_same_route(gm, gp, om, op, "stale replicas, full size")
    # The host-pointer call pipelines 262,144 requests as two chunks (copies overlapping the routing, groups
    # formed per chunk): its results must be those of the one-pass device call.
    hm, hp = r.route_host(tok, off, W.load(), W.alpha)
    assert_same_route(hm, hp, gm, gp, "host-pointer call in chunks")


def _build_router(W, n_threads):
    """Snapshots built on host threads, uploaded in order (as the bench does)."""
    r = g.Router(W.P)

    def make(p):
        return g.p2p_snapshot_build(W.tree(p))

    with ThreadPoolExecutor(max_workers=n_threads) as ex:
        for p, snap in enumerate(ex.map(make, range(W.P))):
            flat = g.FlatTree()
            g._load().p2p_snapshot_view(snap, flat)
            g._check(g._load().p2p_tree_upload(r.handle, p, flat), r.handle)
            g.p2p_snapshot_free(snap)
    r.sync()
    return r


def test_scale_workload_full_after_a_compaction_wave():
    import torch
    W = wl.Workload(4)
    P, B = W.P, W.B
    nt = os.cpu_count() or 8
    r = _build_router(W, nt)
    otrees = oracle.build_trees([W.tree(p) for p in range(P)], n_threads=nt)
    frac = W.params["delta_frac"]

    def stale_labels():
        return np.array([r.stats(p)["stale_label"] for p in range(P)])

    wave = None
    for s in range(40):
        W.delta_make(s, frac, frac, n_threads=nt)
        d = W.delta(n_threads=nt)
        before = stale_labels()
        if s % 2:  # odd rounds from device arrays (the bench's path), even rounds from host arrays
            dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
            sl = wl.SeqList(dev(d.seqs.seg_begin), dev(d.seqs.seg_off), dev(d.seqs.seg_len), dev(d.seqs.pool))
            assert r.apply_delta(-1, dev(d.op), sl, dev(d.peer_begin), on_device=True) == 0
        else:
            assert r.apply_delta(-1, d.op, d.seqs, d.peer_begin) == 0

        def apply(p):
            return otrees[p].apply_ops(d.op, d.seqs, int(d.peer_begin[p]), int(d.peer_begin[p + 1]))

        with ThreadPoolExecutor(max_workers=nt) as ex:
            assert sum(ex.map(apply, range(P))) == 0
        compacted = int((stale_labels() < before).sum())
        if wave is not None:
            break  # one more round on the compacted trees
        if compacted >= P // 2:
            wave = (s, compacted)
    assert wave is not None, "no compaction wave in 40 anti-entropy rounds"
    # The full batch on the device, and the oracle over all 256 trees.
    tok, off = W.requests(n_threads=nt)
    load = W.load()
    gm, gp = _route_full(r, tok, off, load, W.alpha)
    om, op, _ = oracle.route(otrees, tok, off, load, W.alpha, n_threads=nt)
    assert gm.max() > 1000
    assert_same_route(gm, gp, om, op, f"scale workload, full size, after the compaction wave of round {wave[0]}")
    del gm, om
    # Every patched replica byte for byte.
    for p in range(P):
        assert same_snapshot(r.download(p), otrees[p].export()), p
