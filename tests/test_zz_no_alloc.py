"""The allocation-free delta call, p2p_tree_apply_delta_static.

Callers such as a serving loop whose device memory is managed by another allocator (no cudaMalloc, no
caching-allocator calls on its hot path), or a process that must keep a fixed device footprint after
start-up, patch their replicas through this variant: the delta is already in device memory and the call
uses the library's static device scratch instead of growing buffers of its own.  Its results must be
exactly those of the ordinary delta call, p2p_tree_apply_delta, call after call.

This file is named so that pytest collects it last; it creates its own routers and data, so it passes
alone in a fresh process (where its first call also sets up the static scratch) and after the others.
"""
import numpy as np
import pytest

import paper_2606_17059_gb300 as g
import workload as wl

pytestmark = pytest.mark.gpu


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _device_delta(d):
    return _dev(d.op), wl.SeqList(_dev(d.seqs.seg_begin), _dev(d.seqs.seg_off), _dev(d.seqs.seg_len),
                                  _dev(d.seqs.pool)), _dev(d.peer_begin)


def _same_trees(ra, rb, P):
    for p in range(P):
        a, b = ra.download(p), rb.download(p)
        for k in a:
            assert np.array_equal(a[k], b[k]), (p, k)


def test_static_delta_matches_the_allocating_call_on_two_calls_in_a_row():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    prm = wl.preset(4)
    prm.update(P=4, n_seq=2000, n_prefix=200, pre_lo=16, pre_hi=300, B=2000)
    W = wl.Workload(params=prm, seed=2024)
    ra, rb = g.Router(W.P), g.Router(W.P)
    for p in range(W.P):
        sl = W.tree(p)
        ra.build(p, sl)
        rb.build(p, sl)
    # One ordinary round on both routers first, so that both start from the same patched trees.
    W.delta_make(0, 0.05, 0.05)
    op, sl, pb = _device_delta(W.delta())
    assert ra.apply_delta(-1, op, sl, pb, on_device=True) == rb.apply_delta(-1, op, sl, pb, on_device=True)
    tok, off = W.requests()
    t_tok, t_off = _dev(tok), _dev(off)
    load = W.load()
    for step in (1, 2):  # two calls in a row through the static variant
        W.delta_make(step, 0.02, 0.02)
        op, sl, pb = _device_delta(W.delta())
        absent_a = g.p2p_tree_apply_delta(ra.handle, -1, op, sl, pb, on_device=True)
        absent_b = g.p2p_tree_apply_delta_static(rb.handle, -1, op, sl, pb)
        assert absent_a == absent_b == 0
        _same_trees(ra, rb, W.P)
        ma, pa = ra.route(t_tok, t_off, load, W.alpha)
        mb, pb_ = rb.route(t_tok, t_off, load, W.alpha)
        ra.sync()
        rb.sync()
        assert torch.equal(ma, mb) and torch.equal(pa, pb_)
    # A single-tree call with a DELETE of a sequence that is not stored (a counted no-op) in between.
    seqs = [W.tree(1).seq(0).tolist(), [7, 7, 7]]
    ops = np.array([1, 1], np.int32)
    pool = np.array(seqs[0] + seqs[1], np.int32)
    one = wl.SeqList(np.array([0, 1, 2], np.int64), np.array([0, len(seqs[0])], np.int64),
                     np.array([len(seqs[0]), 3], np.int32), pool)
    dsl = wl.SeqList(_dev(one.seg_begin), _dev(one.seg_off), _dev(one.seg_len), _dev(one.pool))
    assert g.p2p_tree_apply_delta(ra.handle, 1, _dev(ops), dsl, None, on_device=True) == \
        g.p2p_tree_apply_delta_static(rb.handle, 1, _dev(ops), dsl, None)
    _same_trees(ra, rb, W.P)


def test_static_delta_rejects_host_memory_sizes_beyond_its_scratch_and_full_trees():
    import ctypes
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    r = g.Router(4)
    # A host-memory delta would need device staging buffers, so the static variant rejects it.
    h = wl.SeqList(np.array([0, 1], np.int64), np.array([0], np.int64), np.array([3], np.int32),
                   np.array([1, 2, 3], np.int32))
    h_op = np.zeros(1, np.int32)
    keep = []
    d = g.Delta(h_op.ctypes.data, g._seqs_struct(h, keep), None, g.P2P_MEM_HOST)
    rc = g._load().p2p_tree_apply_delta_static(r.handle, 0, ctypes.byref(d), None)
    assert rc == g.P2P_E_INVAL and "device memory" in g.p2p_last_error(r.handle)
    # An op whose sequence is split into more than two pool runs is gathered into the scratch: 16 warps x
    # a 600,000-token sequence per tree cannot fit in the 8 MiB array.
    n = 600_000
    pool = _dev(np.arange(n, dtype=np.int32))
    three = wl.SeqList(_dev(np.array([0, 3], np.int64)), _dev(np.array([0, 200_000, 400_000], np.int64)),
                       _dev(np.array([200_000] * 3, np.int32)), pool)
    ins = _dev(np.zeros(1, np.int32))
    with pytest.raises(g.P2PError) as e:
        g.p2p_tree_apply_delta_static(r.handle, 0, ins, three, None)
    assert e.value.code == g.P2P_E_INVAL and "exceeds the static scratch" in str(e.value)
    big = wl.SeqList(_dev(np.array([0, 1], np.int64)), _dev(np.array([0], np.int64)),
                     _dev(np.array([n], np.int32)), pool)
    # On one tree the scratch suffices, but an empty tree's label arena cannot hold 600,000 tokens and the
    # static variant never grows a tree: P2P_E_NOMEM, nothing applied.
    with pytest.raises(g.P2PError) as e:
        g.p2p_tree_apply_delta_static(r.handle, 2, ins, big, None)
    assert e.value.code == g.P2P_E_NOMEM
    assert r.stats(2)["label_tokens"] == 0
    # The allocating call grows the tree; afterwards the static variant can delete the sequence again.
    assert g.p2p_tree_apply_delta(r.handle, 2, ins, big, None, on_device=True) == 0
    assert r.stats(2)["label_tokens"] == n
    assert g.p2p_tree_apply_delta_static(r.handle, 2, _dev(np.ones(1, np.int32)), big, None) == 0
    assert r.stats(2)["live_nodes"] == 1 and r.download(2)["label_off"].tolist() == [0]
