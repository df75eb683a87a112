"""Generator tests: the published PRNGs, bounded and Zipf draws, and the workload shapes of the five
presets (sizes, length ranges, skew, determinism, deltas).  No GPU."""
import json
import math
import os

import numpy as np
import pytest

import workload as wl

M64 = (1 << 64) - 1


def test_splitmix64_published_values(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "prng.json")))
    assert wl.splitmix64_sequence(g["splitmix64_seed"], 5) == g["splitmix64_first5"]


def _rotl(x, k):
    return ((x << k) | (x >> (64 - k))) & M64


def _xoshiro_py(state, n):
    s = list(state)
    out = []
    for _ in range(n):
        out.append((_rotl((s[1] * 5) & M64, 7) * 9) & M64)
        t = (s[1] << 17) & M64
        s[2] ^= s[0]
        s[3] ^= s[1]
        s[1] ^= s[2]
        s[0] ^= s[3]
        s[2] ^= t
        s[3] = _rotl(s[3], 45)
    return out


def test_xoshiro256ss_matches_definition():
    state = [0x0123456789ABCDEF, 0xFEDCBA9876543210, 0x0F1E2D3C4B5A6978, 0x1122334455667788]
    assert wl.xoshiro_from_state(state, 64) == _xoshiro_py(state, 64)


def test_xoshiro_seeded_by_splitmix():
    st = wl.splitmix64_sequence(99, 4)
    assert wl.xoshiro_sequence(99, 16) == _xoshiro_py(st, 16)


@pytest.mark.parametrize("rng", [1, 2, 3, 7, 1000, 32000, (1 << 63) + 5])
def test_bounded_in_range_and_multiply_high(rng):
    vals = wl.bounded_sequence(5, rng, 400)
    assert all(0 <= v < rng for v in vals)
    # Without a rejection the draw is the high word of raw * range.
    raw = wl.xoshiro_sequence(5, 1)[0]
    lo = (raw * rng) & M64
    if lo >= ((1 << 64) - rng) % rng:
        assert vals[0] == (raw * rng) >> 64


def test_bounded_uniformity_chi_square():
    vals = np.array(wl.bounded_sequence(11, 10, 20000))
    counts = np.bincount(vals, minlength=10)
    chi2 = ((counts - 2000.0) ** 2 / 2000.0).sum()
    assert chi2 < 30.0  # 9 dof, p ~ 4e-4


def test_zipf_index_inverse_cdf():
    n, s = 57, 1.1
    w = np.arange(1, n + 1, dtype=np.float64) ** -s
    cdf = np.cumsum(w)
    for u in np.linspace(0.0, 0.999999, 200):
        k = wl.zipf_index(n, s, float(u))
        assert cdf[k] > u * cdf[-1]
        assert k == 0 or cdf[k - 1] <= u * cdf[-1]


@pytest.mark.parametrize("cfg", [0, 1, 2, 3, 4])
def test_presets_match_workload_definitions(cfg):
    p = wl.preset(cfg)
    expect = {
        0: dict(P=4, n_seq=1000, n_prefix=57, pre_lo=256, pre_hi=1024, B=4096, load_hi=63, alpha=4),
        1: dict(P=16, n_seq=20000, n_prefix=512, pre_lo=128, pre_hi=2048, B=65536),
        2: dict(P=64, n_seq=20000, n_prefix=2000, B=262144, zipf_s=1.5),
        3: dict(P=32, n_seq=5000, pre_lo=4096, pre_hi=32768, suf_lo=256, suf_hi=1024, B=16384, diverge=1),
        4: dict(P=256, n_seq=100000, n_prefix=10000, pre_lo=128, pre_hi=4096, B=1048576, zipf_s=1.2),
    }[cfg]
    for k, v in expect.items():
        assert p[k] == v, (k, p[k], v)
    assert p["vocab"] == 32000 and p["assign_prob"] == 0.5


def test_cfg0_tree_and_request_shapes():
    W = wl.Workload(0)
    prm = W.params
    assert np.all((W.prefix_len >= 256) & (W.prefix_len <= 1024))
    assert W.prefix_pool.min() >= 0 and W.prefix_pool.max() < 32000
    for p in range(W.P):
        t = W.tree(p)
        assert len(t) == 1000
        tok, off = t.to_csr()
        lens = np.diff(off)
        assert lens.min() >= 256 + 32 and lens.max() <= 1024 + 128
        assert tok.min() >= 0 and tok.max() < prm["vocab"]
    tok, off = W.requests()
    assert len(off) == 4097 and off[0] == 0
    lens = np.diff(off)
    assert lens.min() >= 256 + 32 and lens.max() <= 1024 + 128
    # ~20% of requests carry a fresh prefix: their first 256 tokens match no shared prefix.
    starts = {tuple(W.prefix_pool[o:o + 8]) for o in W.prefix_off}
    fresh = sum(tuple(tok[off[b]:off[b] + 8]) not in starts for b in range(4096))
    assert 0.17 < fresh / 4096 < 0.23
    ld = W.load()
    assert ld.shape == (4,) and ld.min() >= 0 and ld.max() <= 63


def test_request_zipf_skew_cfg1():
    W = wl.Workload(1)
    tok, off = W.requests(0, 20000)
    first = {int(W.prefix_pool[o]) * 100003 + int(W.prefix_pool[o + 1]): k for k, o in enumerate(W.prefix_off)}
    ks = []
    for b in range(20000):
        key = int(tok[off[b]]) * 100003 + int(tok[off[b] + 1])
        if key in first:
            ks.append(first[key])
    ks = np.array(ks)
    share0 = np.mean(ks == 0)
    w = np.arange(1, 513, dtype=np.float64) ** -1.1
    assert abs(share0 - w[0] / w.sum()) < 0.02
    assert np.mean(ks < 10) > np.mean(ks >= 256)


def test_determinism_and_thread_independence():
    a = wl.Workload(1).requests(100, 700, n_threads=1)
    b = wl.Workload(1).requests(100, 700, n_threads=7)
    c, d = wl.Workload(1).requests(0, 1000, n_threads=3)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    # A sub-range equals the same slice of a larger range.
    assert np.array_equal(a[0], c[d[100]:d[700]])
    t1 = wl.Workload(1).tree(5).to_csr()
    t2 = wl.Workload(1).tree(5).to_csr()
    assert np.array_equal(t1[0], t2[0])
    other = wl.Workload(1, seed=123).requests(100, 700)
    assert not np.array_equal(a[0], other[0][: len(a[0])])


def test_long_context_requests_diverge_inside_prefix():
    prm = wl.preset(3)
    prm.update(P=2, n_seq=20, B=300)
    W = wl.Workload(params=prm, seed=3)
    tok, off = W.requests()
    n_div = 0
    for b in range(300):
        r = tok[off[b]:off[b + 1]]
        for k, o in enumerate(W.prefix_off):
            L = int(W.prefix_len[k])
            pre = W.prefix_pool[o:o + L]
            m = min(len(r), L)
            eq = r[:m] == pre[:m]
            d = int(np.argmin(eq)) if not eq.all() else m
            if d >= 64:  # this request follows prefix k for d tokens, then a forced different token
                assert d < L and r[d] != pre[d]
                assert 256 <= len(r) - d - 1 <= 1024
                n_div += 1
                break
    assert n_div > 200


def test_stale_replica_lists_and_delta():
    prm = wl.preset(2)
    prm.update(P=3, n_seq=400, n_prefix=40, B=10)
    W = wl.Workload(params=prm, seed=7)
    n0 = W.tree_size(0)[0]
    assert n0 == 400 and W.tree_size(0, 1)[0] == 400
    for p in (1, 2):
        exact = {tuple(s) for s in W.tree(p, 1).to_lists()}
        rep = W.tree(p, 0).to_lists()
        assert len(rep) == 400 - 40 + 20
        d = W.delta(p, p + 1)
        ops = d.op
        assert (ops == wl.DELETE).sum() == 40 and (ops == wl.INSERT).sum() == 20
        dels = [tuple(d.seqs.seq(i)) for i in range(len(ops)) if ops[i] == wl.DELETE]
        ins = [tuple(d.seqs.seq(i)) for i in range(len(ops)) if ops[i] == wl.INSERT]
        assert all(s in exact for s in dels)
        # exact - deletes + inserts == replica (as multisets)
        from collections import Counter
        ce = Counter(tuple(s) for s in W.tree(p, 1).to_lists())
        ce.subtract(Counter(dels))
        ce.update(Counter(ins))
        assert +ce == Counter(tuple(s) for s in rep)


def test_delta_make_updates_live_list():
    prm = wl.default_params(P=3, n_seq=200, n_prefix=10, pre_lo=4, pre_hi=12, suf_lo=1, suf_hi=4)
    W = wl.Workload(params=prm, seed=5)
    before = [W.tree(p).to_lists() for p in range(3)]
    W.delta_make(step=0, del_frac=0.05, ins_frac=0.05)
    d = W.delta()
    assert list(np.diff(d.peer_begin)) == [20, 20, 20]
    from collections import Counter
    for p in range(3):
        lo, hi = d.peer_begin[p], d.peer_begin[p + 1]
        c = Counter(tuple(s) for s in before[p])
        for i in range(lo, hi):
            s = tuple(d.seqs.seq(i))
            if d.op[i] == wl.DELETE:
                assert c[s] > 0
                c[s] -= 1
            else:
                c[s] += 1
        assert +c == Counter(tuple(s) for s in W.tree(p).to_lists())
    # The next step draws a different delta.
    W.delta_make(step=1, del_frac=0.05, ins_frac=0.05)
    d2 = W.delta()
    assert not np.array_equal(d.seqs.to_csr()[0][:50], d2.seqs.to_csr()[0][:50])


def test_cfg4_sizes_are_as_modelled():
    W = wl.Workload(4)
    n, segs, suf = W.tree_size(0)
    assert n == 100000 and segs <= 2 * n
    assert 70 < suf / n < 90  # suffix 32-128
    assert math.isclose(W.prefix_len.mean(), (128 + 4096) / 2, rel_tol=0.03)
