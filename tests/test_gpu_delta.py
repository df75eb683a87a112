"""GPU parity of the anti-entropy delta path (device INSERT/DELETE on the flattened trees) against the CPU
oracle, through the C ABI.  After every delta the device tree's canonical export must equal the oracle's
byte for byte, the count of absent DELETEs must agree, and routing on the patched trees must match."""
import random

import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl
from gpu_util import (assert_same_route, csr_from_lists, oracle_route, route_device, router_from_seqlists,
                      same_snapshot, seqlist_from_lists)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    g.build()


def _oracle_tree(seqs):
    t = oracle.OTree()
    for s in seqs:
        t.insert(s)
    return t


def _random_ops(rng, stored, V, n_ops, max_len):
    ops, seqs = [], []
    live = list(stored)
    for _ in range(n_ops):
        k = rng.random()
        if k < 0.45 and live:
            s = live.pop(rng.randrange(len(live)))
            ops.append(1)
        elif k < 0.55:
            s = [rng.randrange(V) for _ in range(rng.randint(0, max_len))]  # usually absent
            ops.append(1)
            if s in live:
                live.remove(s)
        elif k < 0.65 and live:
            s = list(rng.choice(live))  # duplicate insert
            ops.append(0)
            live.append(s)
        else:
            base = list(rng.choice(live)) if live and rng.random() < 0.6 else []
            s = base[: rng.randint(0, len(base))] + [rng.randrange(V) for _ in range(rng.randint(0, max_len))]
            ops.append(0)
            live.append(s)
        seqs.append(s)
    return np.array(ops, np.int32), seqs


@pytest.mark.parametrize("seed", range(10))
def test_random_deltas_single_tree(seed):
    rng = random.Random(100 + seed)
    V = rng.choice([2, 3, 5, 1000])
    max_len = rng.choice([6, 30, 200])
    stored = [[rng.randrange(V) for _ in range(rng.randint(0, max_len))] for _ in range(rng.randint(0, 60))]
    r = router_from_seqlists([seqlist_from_lists(stored)])
    t = _oracle_tree(stored)
    for rnd in range(4):
        op, seqs = _random_ops(rng, stored, V, rng.randint(1, 150), max_len)
        sl = seqlist_from_lists(seqs)
        absent_gpu = r.apply_delta(0, op, sl)
        absent_cpu = t.apply_ops(op, sl)
        assert absent_gpu == absent_cpu
        assert same_snapshot(r.download(0), t.export()), f"seed {seed} round {rnd}"
        # keep the python view of the multiset in step
        for o, s in zip(op, seqs):
            if o == 0:
                stored.append(s)
            elif s in stored:
                stored.remove(s)
    reqs = [[rng.randrange(V) for _ in range(rng.randint(0, max_len + 5))] for _ in range(200)]
    reqs += [list(s) + [rng.randrange(V)] for s in stored[:100]]
    tok, off = csr_from_lists(reqs)
    gm, gp = route_device(r, tok, off, [0], 0)
    om, op_, _ = oracle.route([t], tok, off, [0], 0)
    assert_same_route(gm, gp, om, op_, "after deltas")


def test_growth_from_an_empty_tree():
    """Thousands of INSERTs into an empty tree overflow every arena several times over; the host grows
    them and resumes, and the result equals the oracle's."""
    rng = random.Random(5)
    V = 50
    seqs = [[rng.randrange(V) for _ in range(rng.randint(1, 80))] for _ in range(6000)]
    r = g.Router(1)
    op = np.zeros(len(seqs), np.int32)
    assert r.apply_delta(0, op, seqlist_from_lists(seqs)) == 0
    t = _oracle_tree(seqs)
    assert same_snapshot(r.download(0), t.export())
    st = r.stats(0)
    assert st["cap_label"] > 1024 and st["cap_node"] > 64
    # Delete everything again: back to the empty tree.
    rng.shuffle(seqs)
    assert r.apply_delta(0, np.ones(len(seqs), np.int32), seqlist_from_lists(seqs)) == 0
    assert r.download(0)["label_off"].tolist() == [0] and r.stats(0)["live_nodes"] == 1


def test_multi_tree_delta_host_and_device_arrays():
    import torch
    rng = random.Random(9)
    V = 4
    P = 5
    trees = [[[rng.randrange(V) for _ in range(rng.randint(0, 12))] for _ in range(40)] for _ in range(P)]
    ops, seqs, pb = [], [], [0]
    for p in range(P):
        if p == 2:
            pb.append(pb[-1])  # tree 2 gets no ops
            continue
        o, s = _random_ops(rng, trees[p], V, 60, 12)
        ops.extend(o.tolist())
        seqs.extend(s)
        pb.append(pb[-1] + len(o))
    op = np.array(ops, np.int32)
    sl = seqlist_from_lists(seqs)
    peer_begin = np.array(pb, np.int64)
    oracle_trees = [_oracle_tree(t) for t in trees]
    absent_cpu = sum(oracle_trees[p].apply_ops(op, sl, pb[p], pb[p + 1]) for p in range(P))
    r_host = router_from_seqlists([seqlist_from_lists(t) for t in trees])
    r_dev = router_from_seqlists([seqlist_from_lists(t) for t in trees])
    absent_h = r_host.apply_delta(-1, op, sl, peer_begin)
    dsl = wl.SeqList(*[torch.from_numpy(np.ascontiguousarray(a)).cuda()
                       for a in (sl.seg_begin, sl.seg_off, sl.seg_len, sl.pool)])
    absent_d = r_dev.apply_delta(-1, torch.from_numpy(op).cuda(), dsl, torch.from_numpy(peer_begin).cuda(),
                                 on_device=True)
    assert absent_h == absent_d == absent_cpu
    for p in range(P):
        e = oracle_trees[p].export()
        assert same_snapshot(r_host.download(p), e) and same_snapshot(r_dev.download(p), e), p


def test_invalid_deltas_leave_trees_unchanged():
    r = router_from_seqlists([seqlist_from_lists([[1, 2, 3], [1, 2]]), seqlist_from_lists([[4]])])
    before = [r.download(0), r.download(1)]
    sl = seqlist_from_lists([[1, 2, 3], [5]])
    cases = [
        dict(peer=0, op=np.array([0, 7], np.int32), sl=sl, pb=None),                 # bad op code
        dict(peer=2, op=np.array([0, 1], np.int32), sl=sl, pb=None),                 # peer out of range
        dict(peer=-1, op=np.array([0, 1], np.int32), sl=sl, pb=None),                # peer -1 without ranges
        dict(peer=-1, op=np.array([0, 1], np.int32), sl=sl, pb=np.array([0, 2, 1], np.int64)),  # decreasing
        dict(peer=0, op=np.array([0], np.int32),
             sl=wl.SeqList(np.array([0, 1], np.int64), np.array([2], np.int64), np.array([9], np.int32),
                           np.zeros(4, np.int32)), pb=None),                          # segment outside the pool
    ]
    for c in cases:
        with pytest.raises(g.P2PError) as e:
            r.apply_delta(c["peer"], c["op"], c["sl"], c["pb"])
        assert e.value.code == g.P2P_E_INVAL
    assert same_snapshot(r.download(0), before[0]) and same_snapshot(r.download(1), before[1])


def test_stale_replicas_built_by_device_delta():
    """Stale-replica workload at reduced P: upload the exact peer trees, patch trees 1.. with the
    delta that drops 10% of their sequences and adds 5% new ones, and compare with the oracle."""
    prm = wl.preset(2)
    prm.update(P=8, B=20000)
    W = wl.Workload(params=prm, seed=wl.default_seed(2))
    r = router_from_seqlists([W.tree(p, 1) for p in range(W.P)])
    d = W.delta(0, W.P)
    assert d.peer_begin[1] == 0  # tree 0 is exact
    absent = r.apply_delta(-1, d.op, d.seqs, d.peer_begin)
    assert absent == 0
    replicas = [W.tree(p, 0) for p in range(W.P)]
    for p in (0, 1, 5):
        t = oracle.OTree()
        t.insert_seqlist(replicas[p])
        assert same_snapshot(r.download(p), t.export()), p
    tok, off = W.requests()
    gm, gp = route_device(r, tok, off, W.load(), W.alpha)
    om, op = oracle_route(replicas, tok, off, W.load(), W.alpha)
    assert_same_route(gm, gp, om, op, "stale replicas")


def test_repeated_generator_deltas_and_compaction():
    """Anti-entropy rounds as in the scale workload (5% DELETE + 5% INSERT per round) on a smaller
    configuration; enough rounds that stale arena space triggers compaction."""
    prm = wl.preset(4)
    prm.update(P=3, n_seq=3000, n_prefix=300, pre_lo=16, pre_hi=200, B=3000)
    W = wl.Workload(params=prm, seed=77)
    r = router_from_seqlists([W.tree(p) for p in range(W.P)])
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)])
    for step in range(30):
        W.delta_make(step, 0.05, 0.05)
        d = W.delta()
        assert r.apply_delta(-1, d.op, d.seqs, d.peer_begin) == 0
        for p in range(W.P):
            trees[p].apply_ops(d.op, d.seqs, int(d.peer_begin[p]), int(d.peer_begin[p + 1]))
        if step % 10 == 9:
            for p in range(W.P):
                assert same_snapshot(r.download(p), trees[p].export()), (step, p)
    tok, off = W.requests()
    gm, gp = route_device(r, tok, off, W.load(), W.alpha)
    om, op, _ = oracle.route(trees, tok, off, W.load(), W.alpha)
    assert_same_route(gm, gp, om, op, "after 30 rounds")
    st = r.stats(0)
    assert st["stale_label"] + st["stale_child"] <= st["label_tokens"] + st["child_entries"]


def test_device_compaction_keeps_every_tree_canonical():
    """Deletes of a third of each replica per round make stale own-arena labels pass half of the arena, so
    apply_delta compacts the trees on the device (breadth-first copy, tables rehashed without tombstones).
    After every round the downloads and the routes must equal the oracle's, and the stale counters of a
    compacted tree start again from zero."""
    prm = wl.preset(4)
    prm.update(P=4, n_seq=4000, n_prefix=60, pre_lo=16, pre_hi=100, B=2000)
    W = wl.Workload(params=prm, seed=5)
    r = router_from_seqlists([W.tree(p) for p in range(W.P)])
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)])
    compacted = 0
    for step in range(4):
        W.delta_make(step, 0.33, 0.05)
        d = W.delta()
        before = [r.stats(p)["stale_label"] for p in range(W.P)]
        assert r.apply_delta(-1, d.op, d.seqs, d.peer_begin, on_device=step % 2 == 1) == 0
        for p in range(W.P):
            trees[p].apply_ops(d.op, d.seqs, int(d.peer_begin[p]), int(d.peer_begin[p + 1]))
            st = r.stats(p)
            if st["stale_label"] == 0 and st["stale_child"] == 0 and before[p] > 0:
                compacted += 1
            assert same_snapshot(r.download(p), trees[p].export()), (step, p)
        tok, off = W.requests()
        gm, gp = route_device(r, tok, off, W.load(), W.alpha)
        om, op, _ = oracle.route(trees, tok, off, W.load(), W.alpha)
        assert_same_route(gm, gp, om, op, f"round {step}")
    assert compacted >= W.P


def test_compaction_takes_trees_near_the_threshold_along():
    """Once some tree's stale label tokens pass half of its label arena, apply_delta compacts it on the
    device, and in the same call every tree at least 70% of the way there (replicas that receive deltas at
    the same rate reach the threshold within a few calls of one another).  A tree further away keeps its
    stale space.  Each tree holds 2,000 sequences of 100 tokens with distinct first tokens, one leaf edge
    under the root each, so deleting a sequence leaves exactly its 100 label tokens stale."""
    rng = random.Random(11)
    n, L = 2000, 100
    seqs = [[[1 + i] + [rng.randrange(1, 1 << 20) for _ in range(L - 1)] for i in range(n)] for _ in range(3)]
    r = router_from_seqlists([seqlist_from_lists(s) for s in seqs])
    ots = [_oracle_tree(s) for s in seqs]
    done = [0, 0, 0]

    def delete(counts):
        ops, dl, pb = [], [], [0]
        for p, k in enumerate(counts):
            for s in seqs[p][done[p]:done[p] + k]:
                ops.append(1)
                dl.append(s)
                assert ots[p].remove(s)
            done[p] += k
            pb.append(len(ops))
        assert r.apply_delta(-1, np.array(ops, np.int32), seqlist_from_lists(dl), np.array(pb, np.int64)) == 0

    ratio = lambda p: r.stats(p)["stale_label"] / r.stats(p)["label_tokens"]
    # Tree 1 ends at 42% stale, tree 2 at 20%: neither passes half, nothing is compacted.
    delete([0, 840, 400])
    assert 0.35 < ratio(1) < 0.5 and 0 < ratio(2) < 0.35 and ratio(0) == 0
    stale2 = r.stats(2)["stale_label"]
    assert stale2 == 400 * L
    # Tree 0 passes half: it is compacted, and tree 1 with it although this call gave it no ops.
    delete([1200, 0, 0])
    assert r.stats(0)["stale_label"] == 0 and r.stats(1)["stale_label"] == 0
    assert r.stats(2)["stale_label"] == stale2
    assert r.stats(0)["label_tokens"] == (n - 1200) * L and r.stats(1)["label_tokens"] == (n - 840) * L
    for p in range(3):
        assert same_snapshot(r.download(p), ots[p].export()), p


def test_shared_heads_split_at_upload_then_patched():
    """A long label that starts with another tree's interned run (a prompt held with one suffix here and with
    several there) is uploaded as that run's start plus a node with one child: the trees export canonically,
    route like the oracle, and deltas that delete and re-insert through such nodes stay exact."""
    rng = np.random.default_rng(41)
    prompt = rng.integers(0, 30000, size=300).tolist()
    a = [prompt + [1, 2, 3], prompt + [4, 5]]
    b = [prompt + [7, 8, 9, 10]]
    c = [prompt[:200] + [11] * 50, prompt + [7, 8]]
    trees = [a, b, c]
    r = router_from_seqlists([seqlist_from_lists(t) for t in trees])
    o = oracle.build_trees([seqlist_from_lists(t) for t in trees])
    assert r.stats(1)["live_nodes"] == 3  # root, the shared head's node, the leaf
    for p in range(3):
        assert same_snapshot(r.download(p), o[p].export()), p
    reqs = [prompt + [7, 8, 9], prompt[:250], prompt + [4], prompt[:200] + [11, 11], [5]]
    tok, off = csr_from_lists(reqs)
    gm, gp = route_device(r, tok, off, [0, 0, 0], 0)
    om, op_, _ = oracle.route(o, tok, off, [0, 0, 0], 0)
    assert_same_route(gm, gp, om, op_, "shared heads")
    # Delete the only sequence of tree 1 (its head node goes too), then insert through tree 2's heads.
    for p, ops, seqs in ((1, [1], [b[0]]), (2, [0, 1, 0], [prompt + [7], prompt + [7, 8], prompt[:100]])):
        sl = seqlist_from_lists(seqs)
        opa = np.array(ops, np.int32)
        assert r.apply_delta(p, opa, sl) == 0
        o[p].apply_ops(opa, sl)
        assert same_snapshot(r.download(p), o[p].export()), p
    assert r.stats(1)["live_nodes"] == 1
    gm, gp = route_device(r, tok, off, [0, 0, 0], 0)
    om, op_, _ = oracle.route(o, tok, off, [0, 0, 0], 0)
    assert_same_route(gm, gp, om, op_, "shared heads after deltas")


def test_deleting_through_two_shared_heads_under_one_node():
    """Two prompts with the same first token, each held with one suffix: the node of their common first token
    has two upload-split children.  Deleting both sequences in one delta empties the tree (the node left with
    one such child takes it in, then goes with the last deletion)."""
    rng = np.random.default_rng(43)
    p1 = [7] + rng.integers(0, 30000, size=299).tolist()
    p2 = [7] + rng.integers(0, 30000, size=299).tolist()
    a = [p1 + [1], p1 + [2], p2 + [3], p2 + [4]]
    b = [p1 + [5, 6], p2 + [8, 9]]
    r = router_from_seqlists([seqlist_from_lists(a), seqlist_from_lists(b)])
    assert r.stats(1)["live_nodes"] == 6  # root, the first token's node, two head nodes, two leaves
    for order in ([0, 1], [1, 0]):
        sl = seqlist_from_lists([b[i] for i in order])
        assert r.apply_delta(1, np.array([1, 1], np.int32), sl) == 0
        d = r.download(1)
        assert d["label_off"].tolist() == [0] and d["term_count"].tolist() == [0]
        reqs = [p1 + [5], p2[:10], [7]]
        tok, off = csr_from_lists(reqs)
        gm, _ = route_device(r, tok, off, [0, 0], 0)
        assert (gm[:, 1] == 0).all()
        assert r.apply_delta(1, np.zeros(2, np.int32), seqlist_from_lists(b)) == 0  # back for the next order


@pytest.mark.parametrize("single", [False, True])
def test_heavy_tree_split_among_ctas(single):
    """A tree that takes far more ops than a CTA's share of the call (here ~40,000 against 16,384) is split
    among several CTAs by first-token bucket.  Its ops still apply in order per sequence (inserts, deletes and
    re-inserts of the same sequences, duplicates, empty sequences) and the export equals the oracle's byte for
    byte, through a call on every tree (the other tree takes a few ops) and through a call on that tree alone."""
    rng = random.Random(4242 + single)
    V = 3000
    stored = [[rng.randrange(V) for _ in range(rng.randint(1, 40))] for _ in range(3000)]
    small = [[rng.randrange(V) for _ in range(rng.randint(1, 40))] for _ in range(50)]
    r = router_from_seqlists([seqlist_from_lists(stored), seqlist_from_lists(small)])
    t0, t1 = _oracle_tree(stored), _oracle_tree(small)
    for rnd in range(2):
        op0, seqs0 = _random_ops(rng, stored, V, 40_000, 40)
        # the same sequences again: deletes and re-inserts that must follow their first op
        again = [rng.randrange(len(seqs0)) for _ in range(2_000)]
        op0 = np.concatenate([op0, np.array([1 - int(op0[i]) for i in again], np.int32), np.zeros(3, np.int32)])
        seqs0 = seqs0 + [seqs0[i] for i in again] + [[], [], []]
        if single:
            sl = seqlist_from_lists(seqs0)
            assert r.apply_delta(0, op0, sl) == t0.apply_ops(op0, sl)
        else:
            op1, seqs1 = _random_ops(rng, small, V, 20, 40)
            ops = np.concatenate([op0, op1])
            sl = seqlist_from_lists(seqs0 + seqs1)
            pb = np.array([0, len(op0), len(ops)], np.int64)
            r.apply_delta(-1, ops, sl, pb)
            t0.apply_ops(ops, sl, 0, len(op0))
            t1.apply_ops(ops, sl, len(op0), len(ops))
            assert same_snapshot(r.download(1), t1.export()), f"round {rnd}: small tree"
        assert same_snapshot(r.download(0), t0.export()), f"round {rnd}: heavy tree"
