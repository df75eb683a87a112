"""GPU parity of the route decision with excluded peers and a fallback target (p2p_route_decide) against
the oracle's plain tuple ordering, through the C ABI: random match matrices with ties and masks (none,
some, all but one, all), tree counts on and off the warp width, negative entries (read as 0 on both sides),
and a routed batch whose decision with nothing excluded must equal the route's own choice."""
import random

import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl
from gpu_util import route_device, router_from_seqlists

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    g.build()


def _decide(r, match, load, alpha, excluded):
    import torch
    peer, nxt = r.decide(torch.from_numpy(match).cuda(), load, alpha, excluded)
    return peer.cpu().numpy(), nxt.cpu().numpy()


@pytest.mark.parametrize("P", [1, 2, 7, 32, 45, 252, 256, 260, 300])
def test_random_matrices_and_masks(P):
    rng = np.random.default_rng(P)
    B = 600 if P >= 252 else 2000
    r = g.Router(P)
    match = rng.integers(0, 40, size=(B, P), dtype=np.int32)  # many ties
    load = rng.integers(0, 6, size=P).astype(np.int32)
    for alpha in (0, 3):
        masks = [None, (rng.random(P) < 0.3).astype(np.uint8), np.ones(P, np.uint8)]
        if P > 1:
            one = np.ones(P, np.uint8)
            one[rng.integers(P)] = 0
            masks.append(one)
        for ex in masks:
            gp, gn = _decide(r, match, load, alpha, ex)
            op, on = oracle.decide(match, load, alpha, ex)
            assert np.array_equal(gp, op) and np.array_equal(gn, on), (P, alpha, None if ex is None else ex.sum())


@pytest.mark.parametrize("P", [3, 40])
def test_negative_entries_count_as_zero(P):
    rng = np.random.default_rng(100 + P)
    B = 1500
    r = g.Router(P)
    match = rng.integers(-6, 6, size=(B, P), dtype=np.int32)
    match[::7, 0] = np.iinfo(np.int32).min  # the most negative entry too
    load = rng.integers(0, 4, size=P).astype(np.int32)
    for alpha in (0, 1, 5):
        for ex in (None, (rng.random(P) < 0.3).astype(np.uint8)):
            gp, gn = _decide(r, match, load, alpha, ex)
            op, on = oracle.decide(match, load, alpha, ex)
            assert np.array_equal(gp, op) and np.array_equal(gn, on), (P, alpha)


@pytest.mark.parametrize("P", [8, 36])
def test_batch_beyond_the_grid_and_matrix_off_a_16_byte_boundary(P):
    """More rows than the launch has warps (each warp takes several rows, two at a time, with a ragged last
    pair), once from a matrix on a 16-byte boundary and once from one 4 bytes past it."""
    import torch
    rng = np.random.default_rng(200 + P)
    B = 25_001
    r = g.Router(P)
    match = rng.integers(0, 30, size=(B, P), dtype=np.int32)
    load = rng.integers(0, 5, size=P).astype(np.int32)
    ex = (rng.random(P) < 0.25).astype(np.uint8)
    op, on = oracle.decide(match, load, 2, ex)
    flat = torch.zeros(B * P + 4, dtype=torch.int32, device="cuda")
    for shift in (0, 1):
        view = flat[shift:shift + B * P].view(B, P)
        view.copy_(torch.from_numpy(match))
        peer, nxt = r.decide(view, load, 2, ex)
        assert np.array_equal(peer.cpu().numpy(), op) and np.array_equal(nxt.cpu().numpy(), on), (P, shift)


@pytest.mark.parametrize("alpha", [64, 65])
def test_values_and_load_terms_at_the_edge_of_the_short_keys(alpha):
    """Match values just below and at or above 2^22, negative ones, and loads up to 0xFFFF: with alpha = 64
    every load term is below 2^22 (65,535 * 64 = 4,194,240), with alpha = 65 some are not.  Row groups that
    hold an out-of-range value and those that do not share one launch."""
    rng = np.random.default_rng(300 + alpha)
    B, P = 4001, 64
    r = g.Router(P)
    match = rng.integers(0, 50, size=(B, P), dtype=np.int32)
    edge = np.array([(1 << 22) - 1, 1 << 22, (1 << 22) + 1, np.iinfo(np.int32).max, -1], np.int32)
    rows = rng.choice(B, 200, replace=False)
    match[rows, rng.integers(0, P, 200)] = edge[rng.integers(0, len(edge), 200)]
    match[rng.choice(B, 300, replace=False), :] += (1 << 22) - 60   # whole rows just below the bound
    load = rng.integers(0, 4, size=P).astype(np.int32)
    load[rng.choice(P, 8, replace=False)] = 0xFFFF
    load[rng.choice(P, 4, replace=False)] = 0xFFFE
    for ex in (None, (rng.random(P) < 0.2).astype(np.uint8)):
        gp, gn = _decide(r, match, load, alpha, ex)
        op, on = oracle.decide(match, load, alpha, ex)
        assert np.array_equal(gp, op) and np.array_equal(gn, on), (alpha, ex is None)


def test_decision_of_a_routed_batch():
    prm = wl.preset(0)
    prm.update(P=9, n_seq=300, n_prefix=20, B=1500)
    W = wl.Workload(params=prm, seed=21)
    r = router_from_seqlists([W.tree(p) for p in range(W.P)])
    tok, off = W.requests()
    load = W.load()
    gm, gpeer = route_device(r, tok, off, load, W.alpha)
    peer, nxt = _decide(r, gm, load, W.alpha, None)
    assert np.array_equal(peer, gpeer)
    op, on = oracle.decide(gm, load, W.alpha)
    assert np.array_equal(nxt, on)
    # Excluding each request's chosen tree is the same as excluding it for everyone when its decision is
    # recomputed: check on a sample of distinct excluded trees.
    for k in random.Random(2).sample(range(W.P), 4):
        ex = np.zeros(W.P, np.uint8)
        ex[k] = 1
        p2, n2 = _decide(r, gm, load, W.alpha, ex)
        o2, q2 = oracle.decide(gm, load, W.alpha, ex)
        assert np.array_equal(p2, o2) and np.array_equal(n2, q2)
        assert (p2 != k).all() and (n2 != k).all()


def test_invalid_arguments_and_empty_batch():
    import torch
    r = g.Router(3)
    m = torch.zeros((4, 3), dtype=torch.int32, device="cuda")
    out = torch.empty(4, dtype=torch.int32, device="cuda")
    with pytest.raises(g.P2PError) as e:
        g.p2p_route_decide(r.handle, m, 4, [0, 70000, 0], 1, None, out, out.clone())
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError) as e:
        g.p2p_route_decide(r.handle, m, 4, [0, 0, 0], -1, None, out, out.clone())
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(g.P2PError) as e:
        g.p2p_route_decide(r.handle, m, -1, [0, 0, 0], 1, None, out, out.clone())
    assert e.value.code == g.P2P_E_INVAL
    with pytest.raises(ValueError):
        g.p2p_route_decide(r.handle, m, 4, [0, 0, 0], 1, [1, 0], out, out.clone())
    g.p2p_route_decide(r.handle, m, 0, [0, 0, 0], 1, None, out, out.clone())  # B = 0: nothing happens


def _fused(r, tok, off, load, alpha, ex, want_next=True):
    import torch
    m, p, n = r.route_decide(torch.from_numpy(tok).cuda(), torch.from_numpy(off).cuda(), load, alpha, ex, want_next)
    r.sync()
    return m.cpu().numpy(), p.cpu().numpy(), (n.cpu().numpy() if n is not None else None)


@pytest.mark.parametrize("cfg", [0, 3])
def test_decision_fused_into_the_walks_matches_the_oracle(cfg):
    """p2p_route_batch_decide on workload 0 (lane-walk leaders) and workload 3 (staged leaders of long
    requests), with masks none, some, all but one and all: the match matrix is the oracle's and (peer, next)
    is oracle.decide of it."""
    W = wl.Workload(cfg)
    sls = [W.tree(p) for p in range(W.P)]
    r = router_from_seqlists(sls)
    trees = oracle.build_trees(sls, n_threads=16)
    B = 2000 if cfg == 3 else W.B
    tok, off = W.requests(0, B)
    load = W.load()
    om, opeer, _ = oracle.route(trees, tok, off, load, W.alpha, n_threads=16)
    rng = np.random.default_rng(cfg)
    one = np.ones(W.P, np.uint8)
    one[rng.integers(W.P)] = 0
    for ex in (None, (rng.random(W.P) < 0.3).astype(np.uint8), one, np.ones(W.P, np.uint8)):
        gm, gp, gn = _fused(r, tok, off, load, W.alpha, ex)
        assert np.array_equal(gm, om)
        bp, bn = oracle.decide(om, load, W.alpha, ex)
        assert np.array_equal(gp, bp) and np.array_equal(gn, bn), None if ex is None else int(ex.sum())
        if ex is None:
            assert np.array_equal(gp, opeer)
    # Without a mask or a next-best output it is the plain route.
    gm, gp, gn = _fused(r, tok, off, load, W.alpha, None, want_next=False)
    assert gn is None and np.array_equal(gm, om) and np.array_equal(gp, opeer)


@pytest.mark.parametrize("seed", [1, 2])
def test_decision_fused_ties_and_groups(seed):
    """Vocabularies of 2-4 tokens (deep sharing, many equal scores) and tree counts off the warp width."""
    rng = random.Random(seed)
    P = 37 + seed
    V = 2 + seed
    seqlists = []
    for _ in range(P):
        seqs = [[rng.randrange(V) for _ in range(rng.randint(1, 90))] for _ in range(rng.randint(0, 40))]
        from gpu_util import seqlist_from_lists
        seqlists.append(seqlist_from_lists(seqs))
    reqs = [[rng.randrange(V) for _ in range(rng.randint(0, 120))] for _ in range(700)]
    from gpu_util import csr_from_lists
    tok, off = csr_from_lists(reqs)
    load = np.array([rng.randrange(4) for _ in range(P)], np.int32)
    r = router_from_seqlists(seqlists)
    trees = oracle.build_trees(seqlists)
    om, _, _ = oracle.route(trees, tok, off, load, 1)
    ex = np.array([rng.random() < 0.25 for _ in range(P)], np.uint8)
    gm, gp, gn = _fused(r, tok, off, load, 1, ex)
    bp, bn = oracle.decide(om, load, 1, ex)
    assert np.array_equal(gm, om) and np.array_equal(gp, bp) and np.array_equal(gn, bn)
