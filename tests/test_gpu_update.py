"""GPU parity of estimate and own-tree maintenance after routing (p2p_update_estimates: UpdateTrieEstimate and
UpdateTrie of Algorithm 1) against ``oracle.update_estimates`` through the C ABI: a routed batch inserted into
the trees it went to (every tree byte for byte, and the next route of the same batch), unrouted requests
skipped, invalid peers and offsets rejected with nothing changed, and a full workload whose inserts make the
trees grow."""
import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl
from gpu_util import assert_same_route, route_device, router_from_seqlists, same_snapshot

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


def _small(seed=31, P=9, B=1500):
    prm = wl.preset(0)
    prm.update(P=P, n_seq=300, n_prefix=20, B=B)
    return wl.Workload(params=prm, seed=seed)


def _check_trees(r, otrees):
    for p, t in enumerate(otrees):
        assert same_snapshot(r.download(p), t.export()), p


def test_routed_batch_goes_into_the_chosen_trees():
    W = _small()
    sls = [W.tree(p) for p in range(W.P)]
    r = router_from_seqlists(sls)
    otrees = oracle.build_trees(sls)
    tok, off = W.requests()
    load = W.load()
    t, o = _dev(tok), _dev(off)
    gm, gpeer = r.route(t, o, load, W.alpha)
    r.sync()
    om, op, _ = oracle.route(otrees, tok, off, load, W.alpha)
    assert_same_route(gm.cpu().numpy(), gpeer.cpu().numpy(), om, op, "before the update")
    assert r.update_estimates(t, o, gpeer) == W.B
    oracle.update_estimates(otrees, tok, off, op)
    _check_trees(r, otrees)
    # The same batch routed again: every request now matches in full in the tree it went to.
    gm2, gp2 = route_device(r, tok, off, load, W.alpha)
    om2, op2, _ = oracle.route(otrees, tok, off, load, W.alpha)
    assert_same_route(gm2, gp2, om2, op2, "after the update")
    assert np.array_equal(gm2[np.arange(W.B), op], np.diff(off).astype(np.int32))


def test_unrouted_requests_are_skipped_and_bad_input_changes_nothing():
    import torch
    W = _small(seed=32, P=5, B=600)
    sls = [W.tree(p) for p in range(W.P)]
    r = router_from_seqlists(sls)
    otrees = oracle.build_trees(sls)
    tok, off = W.requests()
    rng = np.random.default_rng(3)
    peer = rng.integers(-1, W.P, size=W.B).astype(np.int32)  # about a sixth unrouted
    t, o = _dev(tok), _dev(off)
    before = [r.download(p) for p in range(W.P)]
    bad = peer.copy()
    bad[100] = W.P
    with pytest.raises(g.P2PError) as e:
        r.update_estimates(t, o, _dev(bad))
    assert e.value.code == g.P2P_E_INVAL
    off_bad = off.copy()
    off_bad[7] = off_bad[8] + 1  # request 7 now starts after it ends (request 6 grows by one token)
    routed = peer.copy()
    routed[7] = 0
    with pytest.raises(g.P2PError) as e:
        r.update_estimates(t, _dev(off_bad), _dev(routed))
    assert e.value.code == g.P2P_E_INVAL
    for p in range(W.P):
        assert same_snapshot(r.download(p), before[p]), p
    # An unrouted request with invalid offsets is not looked at.
    unrouted = peer.copy()
    unrouted[7] = -1
    assert g.p2p_update_estimates(r.handle, t, t.numel(), _dev(off_bad), W.B, _dev(unrouted)) == int((unrouted >= 0).sum())
    oracle.update_estimates(otrees, tok, off_bad, unrouted)
    _check_trees(r, otrees)
    # Nothing routed, and B = 0.
    assert r.update_estimates(t, o, _dev(np.full(W.B, -1, np.int32))) == 0
    assert g.p2p_update_estimates(r.handle, t, t.numel(), o, 0, _dev(peer)) == 0
    _check_trees(r, otrees)
    with pytest.raises(g.P2PError):
        g.p2p_update_estimates(r.handle, t, t.numel(), o, -1, _dev(peer))
    del torch


def test_workload_one_batch_grows_the_trees():
    """Workload 1 (P = 16, 65,536 requests): the inserts add about 20% fresh prompts to the lowest-load trees,
    far past their arenas' headroom."""
    W = wl.Workload(1)
    sls = [W.tree(p) for p in range(W.P)]
    r = router_from_seqlists(sls)
    otrees = oracle.build_trees(sls, n_threads=16)
    tok, off = W.requests()
    load = W.load()
    t, o = _dev(tok), _dev(off)
    gm, gpeer = r.route(t, o, load, W.alpha)
    r.sync()
    caps = [r.stats(p)["cap_label"] for p in range(W.P)]
    assert r.update_estimates(t, o, gpeer) == W.B
    oracle.update_estimates(otrees, tok, off, gpeer.cpu().numpy())
    assert any(r.stats(p)["cap_label"] > caps[p] for p in range(W.P))
    _check_trees(r, otrees)
    gm2, gp2 = route_device(r, tok, off, load, W.alpha)
    om2, op2, _ = oracle.route(otrees, tok, off, load, W.alpha, n_threads=16)
    assert_same_route(gm2, gp2, om2, op2, "workload 1 after the update")
