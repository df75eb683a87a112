"""GPU parity of the route path (lookup kernel + fused route reduction) against the CPU oracle, through
the C ABI.  All outputs are integers: every match value and every chosen peer must be identical."""
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


def _random_case(rng, P, V, n_seq, max_len, n_req, max_req):
    trees = [[[rng.randrange(V) for _ in range(rng.randint(0, max_len))] for _ in range(rng.randint(0, n_seq))]
             for _ in range(P)]
    reqs = []
    for _ in range(n_req):
        if rng.random() < 0.5 and any(trees):
            src = rng.choice([t for t in trees if t])
            s = rng.choice(src)
            cut = rng.randint(0, len(s))
            r = s[:cut] + [rng.randrange(V) for _ in range(rng.randint(0, max_req))]
        else:
            r = [rng.randrange(V) for _ in range(rng.randint(0, max_req))]
        reqs.append(r)
    return trees, reqs


@pytest.mark.parametrize("seed", range(12))
def test_small_random_ties_and_deep_sharing(seed):
    rng = random.Random(seed)
    P = rng.randint(1, 11)
    V = rng.choice([2, 3, 4, 50])
    trees, reqs = _random_case(rng, P, V, n_seq=30, max_len=rng.choice([8, 40, 300]), n_req=300,
                               max_req=rng.choice([10, 60, 400]))
    load = [rng.randrange(3) for _ in range(P)]
    alpha = rng.choice([0, 1, 3])
    sls = [seqlist_from_lists(t) for t in trees]
    tok, off = csr_from_lists(reqs)
    r = router_from_seqlists(sls)
    gm, gp = route_device(r, tok, off, load, alpha)
    om, op = oracle_route(sls, tok, off, load, alpha)
    assert_same_route(gm, gp, om, op, f"seed {seed}")


def test_wide_nodes_and_requests_beyond_shared_memory():
    """Roots with thousands of children (32-ary child search), labels and requests longer than the
    4,096 tokens staged in shared memory (tail read from global memory), splits deep in long labels."""
    rng = random.Random(7)
    V = 100000
    P = 3
    base = [rng.randrange(V) for _ in range(12000)]
    trees = []
    for p in range(P):
        seqs = [[rng.randrange(V) for _ in range(rng.randint(1, 20))] for _ in range(3000)]
        seqs += [base[: rng.randint(4000, 12000)] + [rng.randrange(V) for _ in range(50)] for _ in range(20)]
        trees.append(seqs)
    reqs = []
    for _ in range(400):
        k = rng.random()
        if k < 0.4:
            d = rng.randint(0, 11999)
            reqs.append(base[:d] + [rng.randrange(V) for _ in range(rng.randint(0, 300))])
        elif k < 0.7:
            t = rng.choice(trees)
            reqs.append(list(rng.choice(t)) + [rng.randrange(V)])
        else:
            reqs.append([rng.randrange(V) for _ in range(rng.randint(0, 30))])
    sls = [seqlist_from_lists(t) for t in trees]
    tok, off = csr_from_lists(reqs)
    r = router_from_seqlists(sls)
    load = [5, 0, 9]
    gm, gp = route_device(r, tok, off, load, 1)
    om, op = oracle_route(sls, tok, off, load, 1)
    assert_same_route(gm, gp, om, op, "wide/long")
    assert gm.max() > 4096


@pytest.mark.parametrize("cfg", [0, 1, 3])
def test_full_workload_bit_exact(cfg):
    W = wl.Workload(cfg)
    sls = [W.tree(p) for p in range(W.P)]
    tok, off = W.requests()
    load = W.load()
    r = router_from_seqlists(sls)
    gm, gp = route_device(r, tok, off, load, W.alpha)
    om, op = oracle_route(sls, tok, off, load, W.alpha)
    assert_same_route(gm, gp, om, op, f"workload {cfg}")
    assert gm.max() > 0 and len(np.unique(gp)) > 1


def test_alpha_zero_is_pure_prefix_argmax_and_single_tree():
    W = wl.Workload(0)
    sls = [W.tree(p) for p in range(W.P)]
    tok, off = W.requests(0, 1000)
    r = router_from_seqlists(sls)
    zero = np.zeros(W.P, np.int32)
    gm, gp = route_device(r, tok, off, zero, 0)
    # With alpha = 0 and equal loads the route is the first tree with the largest match (Algorithm 1).
    assert np.array_equal(gp, np.argmax(gm, axis=1))
    r1 = router_from_seqlists(sls[:1])
    gm1, gp1 = route_device(r1, tok, off, [7], 3)
    assert np.all(gp1 == 0) and np.array_equal(gm1[:, 0], gm[:, 0])


def test_host_api_equals_device_api_and_pinned_buffers():
    import torch
    W = wl.Workload(0)
    sls = [W.tree(p) for p in range(W.P)]
    tok, off = W.requests(0, 2000)
    load = W.load()
    r = router_from_seqlists(sls)
    gm, gp = route_device(r, tok, off, load, W.alpha)
    hm, hp = r.route_host(tok, off, load, W.alpha)
    assert np.array_equal(gm, hm) and np.array_equal(gp, hp)
    # Pinned host buffers and a request range that does not start at token 0.
    ptok = torch.from_numpy(tok).pin_memory().numpy()
    sub = off[500:1501].copy()
    m2, p2 = r.route_host(ptok, sub, load, W.alpha)
    assert np.array_equal(m2, gm[500:1500]) and np.array_equal(p2, gp[500:1500])


def test_download_roundtrip_and_idempotent_upload():
    W = wl.Workload(1)
    r = g.Router(2)
    sl = W.tree(3)
    h = g.p2p_snapshot_build(sl)
    snap = g.p2p_snapshot_view(h)
    g.p2p_snapshot_free(h)
    r.upload(0, snap)
    r.upload(1, snap)
    r.upload(1, snap)  # the same broadcast delivered twice
    d0, d1 = r.download(0), r.download(1)
    assert same_snapshot(d0, snap) and same_snapshot(d1, snap)
    t = oracle.OTree()
    t.insert_seqlist(sl)
    assert same_snapshot(d0, t.export())


def test_empty_trees_and_empty_requests():
    r = g.Router(3)  # all trees empty (a node restarted after a crash)
    reqs = [[], [1, 2, 3], [], [9]]
    tok, off = csr_from_lists(reqs)
    gm, gp = route_device(r, tok, off, [4, 1, 1], 2)
    assert np.all(gm == 0)
    assert gp.tolist() == [1, 1, 1, 1]  # equal scores except load: lowest load, then lowest index
    r.build(2, seqlist_from_lists([[1, 2], [9, 9]]))
    gm, gp = route_device(r, tok, off, [0, 0, 0], 1)
    assert gm[:, 2].tolist() == [0, 2, 0, 1] and gp.tolist() == [0, 2, 0, 2]
    # B = 0 is a no-op.
    import torch
    r.route(torch.zeros(0, dtype=torch.int32, device="cuda"), torch.zeros(1, dtype=torch.int64, device="cuda"),
            [0, 0, 0], 1)
    r.sync()


def test_bad_offsets_flag_a_device_error_and_recover():
    import torch
    r = router_from_seqlists([seqlist_from_lists([[1, 2, 3]]), seqlist_from_lists([[1]])])
    tok = torch.tensor([1, 2, 3, 4], dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 3, 2, 9], dtype=torch.int64, device="cuda")  # request 1 decreasing, 2 past the end
    m, p = r.route(tok, off, [0, 0], 1)
    with pytest.raises(g.P2PError) as e:
        r.sync()
    assert e.value.code == g.P2P_E_DEVICE
    assert p.cpu().tolist() == [0, -1, -1]
    assert m.cpu().tolist() == [[3, 1], [0, 0], [0, 0]]
    r.sync()  # the error state was cleared
    off2 = torch.tensor([0, 3, 4], dtype=torch.int64, device="cuda")
    m, p = r.route(tok, off2, [0, 0], 1)
    r.sync()
    assert m.cpu().tolist() == [[3, 1], [0, 0]]


def test_invalid_arguments_are_rejected():
    import torch
    r = g.Router(2)
    tok = torch.zeros(4, dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 4], dtype=torch.int64, device="cuda")
    for load, alpha in (([0, -1], 1), ([0, 70000], 1), ([0, 1], -1), ([40000, 40000], 60000)):
        with pytest.raises(g.P2PError) as e:
            r.route(tok, off, load, alpha)
        assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError):
        r.build(2, seqlist_from_lists([[1]]))
    bad = {k: np.array(v) for k, v in dict(label_off=[0, 0], label_len=[0, 1], child_begin=[0, 1],
                                           child_count=[1, 0], term_count=[0, 0], child_first_tok=[4],
                                           child_idx=[1], labels=[4]).items()}
    with pytest.raises(g.P2PError) as e:
        r.upload(0, bad)
    assert e.value.code == g.P2P_E_FORMAT
    assert np.all(r.download(0)["label_off"] == 0)  # unchanged (still empty)
    # More than 2^30 requests in one call: rejected before any device pointer is read.
    big = (1 << 30) + 1
    with pytest.raises(g.P2PError) as e:
        g.p2p_route_batch(r.handle, tok, 4, off, big, [0, 0], 1, tok, tok)
    assert e.value.code == g.P2P_E_INVAL and "2^30" in str(e.value)


def test_route_on_a_side_stream():
    import torch
    W = wl.Workload(0)
    sls = [W.tree(p) for p in range(W.P)]
    tok, off = W.requests(0, 800)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        r = router_from_seqlists(sls)
        t = torch.from_numpy(tok).cuda()
        o = torch.from_numpy(off).cuda()
        m, p = r.route(t, o, W.load(), W.alpha)
    r.sync()
    om, op = oracle_route(sls, tok, off, W.load(), W.alpha)
    assert_same_route(m.cpu().numpy(), p.cpu().numpy(), om, op, "side stream")


def test_kernel_clock_counts_every_launch():
    import torch
    W = wl.Workload(0)
    sls = [W.tree(p) for p in range(W.P)]
    r = router_from_seqlists(sls)
    tok, off = W.requests(0, 1000)
    t = torch.from_numpy(tok).cuda()
    o = torch.from_numpy(off).cuda()
    assert r.kernel_times() == {}  # off
    r.kernel_clock(True)
    n0 = r.launch_count()
    for _ in range(3):
        r.route(t, o, W.load(), W.alpha)
    W.delta_make(0, 0.05, 0.05)
    d = W.delta()
    r.apply_delta(-1, d.op, d.seqs, d.peer_begin)
    times = r.kernel_times()
    assert sum(n for n, _ in times.values()) == r.launch_count() - n0
    assert times["lane_kernel<false>"][0] == 3 and times["group_hash_kernel"][0] == 3
    assert times["delta_kernel"][0] >= 1 and times["validate_kernel"][0] == 1
    assert all(ms > 0 for _, ms in times.values())
    r.kernel_clock(False)
    assert r.kernel_times() == {}
    with pytest.raises(g.P2PError):
        g.p2p_router_kernel_time(r.handle, g.KERNEL_COUNT)


def test_root_first_tokens_added_and_removed_by_deltas():
    """A first token that a delta adds at the root is found by the next route (the root filter learns it on
    the device); one whose sequences are all deleted matches nothing again (its filter bit stays set)."""
    import torch
    rng = np.random.default_rng(12)
    base = [[int(t)] + rng.integers(0, 50, size=20).tolist() for t in range(0, 4000, 7)]
    r = router_from_seqlists([seqlist_from_lists(base)])
    otree = oracle.build_trees([seqlist_from_lists(base)])[0]
    new = [[int(t)] + rng.integers(0, 50, size=12).tolist() for t in range(3, 4000, 7)]
    gone = base[::3]
    ops = np.array([0] * len(new) + [1] * len(gone), np.int32)
    sl = seqlist_from_lists(new + gone)
    assert r.apply_delta(0, _dev_arr(ops), _dev_seqlist(sl), None, on_device=True) == 0
    otree.apply_ops(ops, sl)
    reqs = [s[:15] for s in new] + [s[:15] for s in base] + [[t, 1, 2] for t in range(1, 4000, 7)]
    tok, off = csr_from_lists(reqs)
    gm, gp = route_device(r, tok, off, [0], 0)
    om, op, _ = oracle.route([otree], tok, off, [0], 0)
    assert_same_route(gm, gp, om, op, "root filter after a delta")
    assert (gm[: len(new), 0] == 13).all()  # each new sequence is 13 tokens long
    del torch


@pytest.mark.parametrize("seed", range(4))
def test_requests_that_leave_after_one_or_two_tokens(seed):
    """Requests that leave a tree after one or two tokens: first tokens small and large (up to 2^30), root
    children whose label is one token, one-token requests, and deltas that remove every sequence of some first
    tokens, bring new ones and bring removed ones back (the root filter keeps stale bits); every match value
    and route against the oracle."""
    rng = np.random.default_rng(300 + seed)
    big = [200_000, 300_000, 1 << 30]
    firsts = list(range(40)) + big

    def seq():
        t0 = int(rng.choice(firsts))
        return [t0] + rng.integers(0, 60, size=int(rng.integers(0, 6))).tolist()

    base = [[seq() for _ in range(300)] for _ in range(2)]
    r = router_from_seqlists([seqlist_from_lists(b) for b in base])
    otrees = oracle.build_trees([seqlist_from_lists(b) for b in base])
    stored = [list(b) for b in base]
    for rnd in range(4):
        reqs = [[int(rng.integers(0, 45))] + rng.integers(0, 60, size=int(rng.integers(0, 4))).tolist()
                for _ in range(1500)]
        reqs += [[int(rng.choice(big))] + rng.integers(0, 60, size=int(rng.integers(0, 3))).tolist() for _ in range(200)]
        reqs += [list(s[: int(rng.integers(1, len(s) + 1))]) for s in stored[0][:200]]
        tok, off = csr_from_lists(reqs)
        load = [int(x) for x in rng.integers(0, 3, size=2)]
        gm, gp = route_device(r, tok, off, load, 1)
        om, op, _ = oracle.route(otrees, tok, off, load, 1)
        assert_same_route(gm, gp, om, op, f"seed {seed} round {rnd}")
        # The next delta: every sequence of a few first tokens goes, new first tokens come, old ones come back.
        gone_t0 = set(int(x) for x in rng.choice(firsts, size=6, replace=False))
        ops, seqs, pb = [], [], [0]
        for p in range(2):
            dels = [s for s in stored[p] if s[0] in gone_t0]
            ins = [[int(rng.integers(40, 44))] + rng.integers(0, 60, size=int(rng.integers(0, 5))).tolist()
                   for _ in range(20)] + [seq() for _ in range(20)]
            ops += [1] * len(dels) + [0] * len(ins)
            seqs += dels + ins
            pb.append(len(ops))
            stored[p] = [s for s in stored[p] if s[0] not in gone_t0] + ins
        op_a = np.array(ops, np.int32)
        sl = seqlist_from_lists(seqs)
        r.apply_delta(-1, op_a, sl, np.array(pb, np.int64))
        for p in range(2):
            otrees[p].apply_ops(op_a, sl, pb[p], pb[p + 1])


def _dev_arr(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _dev_seqlist(sl):
    return wl.SeqList(_dev_arr(sl.seg_begin), _dev_arr(sl.seg_off), _dev_arr(sl.seg_len), _dev_arr(sl.pool))


def test_prepared_grouping_overlapping_a_delta():
    """p2p_route_prepare: the batch's grouping runs alongside the next delta kernel, and the route of the same
    batch uses it; results equal a plain route after the same delta, and a route of another batch (or one
    without a delta in between) groups as usual."""
    import torch
    W = wl.Workload(0)
    sls = [W.tree(p) for p in range(W.P)]
    ra, rb = router_from_seqlists(sls), router_from_seqlists(sls)
    tok, off = W.requests()
    t, o = torch.from_numpy(tok).cuda(), torch.from_numpy(off).cuda()
    t2, o2 = t[: int(off[1000])].clone(), o[:1001].clone()
    load = W.load()
    for step in range(3):
        W.delta_make(step, 0.05, 0.05)
        d = W.delta()
        g.p2p_route_prepare(ra.handle, t, t.numel(), o, W.B)
        assert ra.apply_delta(-1, d.op, d.seqs, d.peer_begin) == 0
        assert rb.apply_delta(-1, d.op, d.seqs, d.peer_begin) == 0
        ma, pa = ra.route(t, o, load, W.alpha)
        mb, pb = rb.route(t, o, load, W.alpha)
        ra.sync()
        rb.sync()
        assert torch.equal(ma, mb) and torch.equal(pa, pb), step
    # Prepared, then another batch routed (and no delta): both group on their own.
    g.p2p_route_prepare(ra.handle, t, t.numel(), o, W.B)
    g.p2p_route_prepare(ra.handle, t, t.numel(), o, W.B)  # twice: the later one stands
    m2a, p2a = ra.route(t2, o2, load, W.alpha)
    m2b, p2b = rb.route(t2, o2, load, W.alpha)
    ma, pa = ra.route(t, o, load, W.alpha)
    ra.sync()
    rb.sync()
    assert torch.equal(m2a, m2b) and torch.equal(p2a, p2b) and torch.equal(ma, mb) and torch.equal(pa, pb)
