"""Helpers shared by the GPU tests: build a router from workload sequence lists, route on the device, and
compute the oracle's answer for the same inputs."""
from __future__ import annotations

import numpy as np

import oracle
import workload as wl


def seqlist_from_lists(seqs) -> wl.SeqList:
    pool = np.array([x for s in seqs for x in s], np.int32)
    lens = np.array([len(s) for s in seqs], np.int32)
    off = np.zeros(len(seqs), np.int64)
    if len(seqs):
        off[1:] = np.cumsum(lens.astype(np.int64))[:-1]
    return wl.SeqList(np.arange(len(seqs) + 1, dtype=np.int64), off, lens, pool)


def csr_from_lists(reqs):
    tokens = np.array([x for r in reqs for x in r], np.int32)
    offsets = np.zeros(len(reqs) + 1, np.int64)
    np.cumsum([len(r) for r in reqs], out=offsets[1:])
    return tokens, offsets


def router_from_seqlists(seqlists):
    import paper_2606_17059_gb300 as g
    r = g.Router(len(seqlists))
    for p, sl in enumerate(seqlists):
        r.build(p, sl)
    return r


def route_device(router, tokens: np.ndarray, offsets: np.ndarray, load, alpha: int):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(tokens, dtype=np.int32)).cuda()
    o = torch.from_numpy(np.ascontiguousarray(offsets, dtype=np.int64)).cuda()
    m, p = router.route(t, o, load, alpha)
    router.sync()
    return m.cpu().numpy(), p.cpu().numpy()


def oracle_route(seqlists, tokens, offsets, load, alpha, n_threads: int = 16):
    trees = oracle.build_trees(seqlists, n_threads=n_threads)
    m, p, _ = oracle.route(trees, tokens, offsets, load, alpha, n_threads=n_threads)
    return m, p


def assert_same_route(gm, gp, om, op, what=""):
    assert gm.shape == om.shape, what
    bad = np.argwhere(gm != om)
    assert len(bad) == 0, f"{what}: {len(bad)} match mismatches, first (b,p)={bad[:5].tolist()} gpu={gm[tuple(bad[0])]} oracle={om[tuple(bad[0])]}"
    badp = np.nonzero(gp != op)[0]
    assert len(badp) == 0, f"{what}: {len(badp)} peer mismatches, first b={badp[:5].tolist()}"


def same_snapshot(a: dict, b: dict) -> bool:
    return all(np.array_equal(np.asarray(a[k]), np.asarray(b[k])) for k in oracle.FLAT_FIELDS)
