"""GPU parity of the LRU cache trie (p2p_lru_enable / insert / access / evict: EvictLRUTrie of Algorithm 1
with device stamps) against the oracle's plain per-token LRUTrie (oracle/lru.py), through the C ABI: random
operation sequences over small vocabularies (deep sharing, partial-edge accesses, equal times, evictions
of a few tokens to all of them), a workload tree made an LRU tree after upload, the calls an LRU tree
rejects, and Section 5's expected hit rate of a routed batch."""
import random

import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl
from gpu_util import csr_from_lists, router_from_seqlists, same_snapshot, seqlist_from_lists
from oracle.lru import LRUTrie, hit_rate

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    g.build()


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _oracle_export(lru: LRUTrie) -> dict:
    t = oracle.OTree()
    for seq, cnt in lru.sequences().items():
        for _ in range(cnt):
            t.insert(list(seq))
    return t.export()


def _batch(reqs):
    tok, off = csr_from_lists(reqs)
    return _dev(tok), _dev(off)


def _insert(r, tree, reqs, time):
    t, o = _batch(reqs)
    g.p2p_lru_insert(r.handle, tree, t, t.numel(), o, len(reqs), time)


def _access(r, tree, reqs, time):
    import torch
    t, o = _batch(reqs)
    m = torch.empty(len(reqs), dtype=torch.int32, device="cuda")
    g.p2p_lru_access(r.handle, tree, t, t.numel(), o, len(reqs), time, m)
    r.sync()
    return m.cpu().numpy()


@pytest.mark.parametrize("seed", range(8))
def test_random_operation_sequences(seed):
    rng = random.Random(seed)
    V = rng.choice([2, 3, 4, 7])
    r = g.Router(2)
    g.p2p_lru_enable(r.handle, 1)
    o = LRUTrie()
    time = 0
    stored = []
    for step in range(45):
        time += rng.choice([0, 0, 1, 2])
        kind = rng.random()
        if kind < 0.4:
            reqs = [[rng.randrange(V) for _ in range(rng.randint(0, 12))] for _ in range(rng.randint(1, 6))]
            _insert(r, 1, reqs, time)
            for s in reqs:
                o.insert(s, time)
            stored += reqs
        elif kind < 0.75:
            reqs = []
            for _ in range(rng.randint(1, 6)):
                if stored and rng.random() < 0.6:  # a prefix of a stored sequence, often with a new tail
                    s = rng.choice(stored)
                    s = s[:rng.randint(0, len(s))] + [rng.randrange(V) for _ in range(rng.randint(0, 3))]
                else:
                    s = [rng.randrange(V) for _ in range(rng.randint(0, 10))]
                reqs.append(s)
            got = _access(r, 1, reqs, time)
            want = [o.access(s, time) for s in reqs]
            assert got.tolist() == want, (step, reqs)
        else:
            n = rng.choice([1, 2, 3, 5, 8, 13, 40])
            evicted = g.p2p_lru_evict(r.handle, 1, n)
            k = 0
            while k < n and o.evict() is not None:
                k += 1
            assert evicted == k, step
        assert same_snapshot(r.download(1), _oracle_export(o)), (seed, step)
        assert r.download(0)["label_off"].tolist() == [0]  # the other tree is untouched
    # Routing sees the LRU tree as it is.
    reqs = [[rng.randrange(V) for _ in range(rng.randint(0, 12))] for _ in range(200)]
    tok, off = csr_from_lists(reqs)
    import torch
    m, _ = r.route(torch.from_numpy(tok).cuda(), torch.from_numpy(off).cuda(), [0, 0], 0)
    r.sync()
    assert m.cpu().numpy()[:, 1].tolist() == [o.match(s) for s in reqs]


@pytest.mark.parametrize("seed", range(3))
def test_wide_nodes_eviction_order(seed):
    """Eviction order among many siblings: a root with ~250 children and a node with ~400, stamped at several
    times (the sibling offsets of the preorder ranks come from a sort of all (parent, first token) pairs, so
    the order must hold at any fan-out, negative first tokens included); every snapshot against the oracle."""
    rng = random.Random(900 + seed)
    r = g.Router(1)
    g.p2p_lru_enable(r.handle, 0)
    o = LRUTrie()
    seqs = [[rng.randrange(-50, 5000)] + [rng.randrange(100) for _ in range(rng.randint(0, 3))] for _ in range(250)]
    seqs += [[7, 7, 7] + [rng.randrange(-30, 2000)] + [rng.randrange(50) for _ in range(rng.randint(0, 2))]
             for _ in range(400)]
    _insert(r, 0, seqs, 1)
    for s in seqs:
        o.insert(s, 1)
    t = 1
    for n in (5, 40, 120, 300):
        t += 1
        reqs = [list(rng.choice(seqs))[: rng.randint(1, 5)] for _ in range(120)]
        got = _access(r, 0, reqs, t)
        assert got.tolist() == [o.access(s, t) for s in reqs]
        evicted = g.p2p_lru_evict(r.handle, 0, n)
        k = 0
        while k < n and o.evict() is not None:
            k += 1
        assert evicted == k
        assert same_snapshot(r.download(0), _oracle_export(o)), (seed, n)


def test_workload_tree_made_lru_after_upload():
    """A generator tree (shared prompt prefixes, Zipf requests) made an LRU tree after its upload: accesses,
    inserts of new prompts, and evictions of a few tokens at a time (the oracle evicts one token per scan of its
    trie, so the evicted amounts stay small); then everything, which leaves every stored sequence empty."""
    prm = wl.preset(0)
    prm.update(P=2, n_seq=60, n_prefix=6, B=160, pre_lo=64, pre_hi=256)
    W = wl.Workload(params=prm, seed=33)
    sl = W.tree(0)
    r = router_from_seqlists([sl, W.tree(1)])
    g.p2p_lru_enable(r.handle, 0)
    o = LRUTrie()
    for i in range(len(sl)):
        o.insert(sl.seq(i).tolist(), 0)
    tok, off = W.requests()
    reqs = [tok[off[b]:off[b + 1]].tolist() for b in range(len(off) - 1)]
    got = _access(r, 0, reqs[:100], 3)
    assert got.tolist() == [o.access(s, 3) for s in reqs[:100]]
    _insert(r, 0, reqs[100:130], 5)
    for s in reqs[100:130]:
        o.insert(s, 5)
    for t, n in ((5, 1), (6, 17), (6, 150), (9, 400)):
        got = _access(r, 0, reqs[130:160], t)
        assert got.tolist() == [o.access(s, t) for s in reqs[130:160]]
        evicted = g.p2p_lru_evict(r.handle, 0, n)
        k = 0
        while k < n and o.evict() is not None:
            k += 1
        assert evicted == k
        assert same_snapshot(r.download(0), _oracle_export(o)), n
    stored = sum(o.sequences().values())
    assert g.p2p_lru_evict(r.handle, 0, 10**12) == o.n_tokens
    d = r.download(0)
    assert d["label_off"].tolist() == [0] and d["term_count"].tolist() == [stored]


def test_lru_tree_rejects_other_changes_and_bad_times():
    import torch
    r = router_from_seqlists([seqlist_from_lists([[1, 2, 3]]), seqlist_from_lists([[4, 5]])])
    g.p2p_lru_enable(r.handle, 0)
    _insert(r, 0, [[1, 2, 9]], 4)
    with pytest.raises(g.P2PError) as e:  # time going back
        _insert(r, 0, [[7]], 3)
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError) as e:
        r.build(0, seqlist_from_lists([[1]]))
    assert e.value.code == g.P2P_E_INVAL
    ops = np.zeros(2, np.int32)
    sl = seqlist_from_lists([[8, 8], [9]])
    with pytest.raises(g.P2PError) as e:  # a delta with ops for the LRU tree (peer = -1 and per tree)
        r.apply_delta(-1, ops, sl, np.array([0, 1, 2], np.int64))
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError) as e:
        r.apply_delta(0, ops, sl)
    assert e.value.code == g.P2P_E_INVAL
    assert r.apply_delta(-1, ops, sl, np.array([0, 0, 2], np.int64)) == 0  # none for it: fine
    t, o = _batch([[1, 2, 3], [4, 5]])
    with pytest.raises(g.P2PError) as e:
        r.update_estimates(t, o, torch.tensor([0, -1], dtype=torch.int32, device="cuda"))
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError) as e:
        g.p2p_lru_evict(r.handle, 1, 3)  # not an LRU tree
    assert e.value.code == g.P2P_E_INVAL
    o2 = LRUTrie()
    o2.insert([1, 2, 3], 0)
    o2.insert([1, 2, 9], 4)
    assert same_snapshot(r.download(0), _oracle_export(o2))


def test_expected_hit_rate_of_a_routed_batch():
    import torch
    prm = wl.preset(0)
    prm.update(P=5, n_seq=300, n_prefix=15, B=900)
    W = wl.Workload(params=prm, seed=8)
    r = router_from_seqlists([W.tree(p) for p in range(W.P)])
    tok, off = W.requests()
    t, o = _dev(tok), _dev(off)
    m, p = r.route(t, o, W.load(), W.alpha)
    p[::11] = -1  # unrouted requests
    out = torch.empty(W.B, dtype=torch.float32, device="cuda")
    g.p2p_hit_rate(r.handle, m, o, W.B, p, out)
    r.sync()
    got = out.cpu().numpy().astype(np.float64)
    mm, pp = m.cpu().numpy(), p.cpu().numpy()
    want = np.array([hit_rate(int(mm[b, pp[b]]), int(off[b + 1] - off[b])) if pp[b] >= 0 else 0.0
                     for b in range(W.B)])
    # Single precision, correctly rounded: within half a unit in the last place of the exact ratio.
    assert np.all(np.abs(got - want) <= want * 2.0**-24)
    assert got.max() > 0.5
