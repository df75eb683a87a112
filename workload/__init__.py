"""Seeded synthetic workload generator (ctypes binding of ``wl.cpp``).

This is the single input source shared by the CPU oracle and the CUDA path.  It holds no radix-tree
or routing arithmetic: it draws token sequences, request batches, peer loads and INSERT/DELETE deltas
and hands them out as numpy arrays.  The workload model and the five presets are described in
``wl.h``; they stand in for the paper's few-shot-prompt workloads (Section 4: shared few-shot prefixes
per topic, skewed topic popularity), with no dataset items used.

Sequences come in segmented form (``SeqList``): sequence i is the concatenation of the pool runs
``pool[seg_off[s]: seg_off[s] + seg_len[s]]`` for s in ``[seg_begin[i], seg_begin[i+1])``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "libwl.so")

INSERT = 0
DELETE = 1


def build(force: bool = False) -> str:
    """Compiles ``libwl.so`` next to this file (plain g++, no GPU needed)."""
    src = os.path.join(_HERE, "wl.cpp")
    hdr = os.path.join(_HERE, "wl.h")
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= max(os.path.getmtime(src), os.path.getmtime(hdr))):
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    subprocess.check_call(["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread", "-o", tmp, src])
    os.replace(tmp, _SO)
    return _SO


class _Params(ctypes.Structure):
    _fields_ = [
        ("P", ctypes.c_int32), ("vocab", ctypes.c_int32), ("n_seq", ctypes.c_int64),
        ("n_prefix", ctypes.c_int32), ("pre_lo", ctypes.c_int32), ("pre_hi", ctypes.c_int32),
        ("suf_lo", ctypes.c_int32), ("suf_hi", ctypes.c_int32), ("zipf_s", ctypes.c_double),
        ("assign_prob", ctypes.c_double), ("B", ctypes.c_int64), ("fresh_frac", ctypes.c_double),
        ("req_suf_lo", ctypes.c_int32), ("req_suf_hi", ctypes.c_int32), ("diverge", ctypes.c_int32),
        ("load_hi", ctypes.c_int32), ("alpha", ctypes.c_int32), ("stale_del_frac", ctypes.c_double),
        ("stale_ins_frac", ctypes.c_double), ("delta_frac", ctypes.c_double),
    ]


PARAM_NAMES = [f[0] for f in _Params._fields_]

_lib = None


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_SO)
        P = ctypes.POINTER
        i32, i64, u64, dbl, vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double, ctypes.c_void_p
        sig = {
            "wl_preset": (ctypes.c_int, [i32, P(_Params)]),
            "wl_default_seed": (u64, [i32]),
            "wl_create": (vp, [P(_Params), u64]),
            "wl_free": (None, [vp]),
            "wl_prefix_pool_size": (i64, [vp]),
            "wl_prefix_pool": (None, [vp, vp, vp, vp]),
            "wl_tree_size": (ctypes.c_int, [vp, i32, i32, P(i64), P(i64), P(i64)]),
            "wl_tree_fill": (ctypes.c_int, [vp, i32, i32, vp, vp, vp, vp, i64]),
            "wl_requests_size": (i64, [vp, i64, i64, i32]),
            "wl_requests_fill": (ctypes.c_int, [vp, i64, i64, vp, vp, i32]),
            "wl_load_fill": (ctypes.c_int, [vp, i64, i32, vp]),
            "wl_delta_make": (ctypes.c_int, [vp, i32, i32, i64, dbl, dbl, i32]),
            "wl_delta_size": (ctypes.c_int, [vp, i32, i32, P(i64), P(i64), P(i64)]),
            "wl_delta_fill": (ctypes.c_int, [vp, i32, i32, vp, vp, vp, vp, vp, i64, vp, i32]),
            "wl_splitmix64": (u64, [P(u64)]),
            "wl_xoshiro_seed": (None, [u64, P(u64 * 4)]),
            "wl_xoshiro_next": (u64, [P(u64 * 4)]),
            "wl_bounded": (u64, [P(u64 * 4), u64]),
            "wl_zipf_index": (i32, [i32, dbl, dbl]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def preset(cfg_id: int) -> dict:
    p = _Params()
    if _load().wl_preset(cfg_id, ctypes.byref(p)) != 0:
        raise ValueError(f"unknown workload id {cfg_id}")
    return {n: getattr(p, n) for n in PARAM_NAMES}


def default_seed(cfg_id: int) -> int:
    return int(_load().wl_default_seed(cfg_id))


def default_params(**kw) -> dict:
    """A small parameter set (for tests); keyword arguments override fields."""
    d = preset(0)
    d.update(kw)
    return d


@dataclass
class SeqList:
    """Segmented sequence list over a token pool (see module docstring)."""
    seg_begin: np.ndarray  # int64 [n+1]
    seg_off: np.ndarray    # int64 [n_segs]
    seg_len: np.ndarray    # int32 [n_segs]
    pool: np.ndarray       # int32 [n_pool]

    def __len__(self) -> int:
        return len(self.seg_begin) - 1

    def seq(self, i: int) -> np.ndarray:
        parts = [self.pool[self.seg_off[s]: self.seg_off[s] + self.seg_len[s]]
                 for s in range(self.seg_begin[i], self.seg_begin[i + 1])]
        return np.concatenate(parts) if parts else np.zeros(0, np.int32)

    def to_csr(self) -> tuple[np.ndarray, np.ndarray]:
        n = len(self)
        lens = np.zeros(n, np.int64)
        np.add.at(lens, np.repeat(np.arange(n), np.diff(self.seg_begin)), self.seg_len.astype(np.int64))
        offsets = np.zeros(n + 1, np.int64)
        np.cumsum(lens, out=offsets[1:])
        tokens = np.empty(int(offsets[-1]), np.int32)
        pos = 0
        for s in range(len(self.seg_off)):
            L = int(self.seg_len[s])
            tokens[pos:pos + L] = self.pool[self.seg_off[s]: self.seg_off[s] + L]
            pos += L
        return tokens, offsets

    def to_lists(self) -> list[list[int]]:
        return [self.seq(i).tolist() for i in range(len(self))]


@dataclass
class Delta:
    """Ordered INSERT(0)/DELETE(1) ops over segmented sequences; ``peer_begin`` marks each tree's ops."""
    op: np.ndarray          # int32 [n_ops]
    seqs: SeqList
    peer_begin: np.ndarray  # int64 [n_trees+1]


class Workload:
    """One seeded workload: a preset id (0..4) or an explicit parameter dict."""

    def __init__(self, cfg_id: int | None = None, params: dict | None = None, seed: int | None = None):
        lib = _load()
        if params is None:
            if cfg_id is None:
                raise ValueError("give cfg_id or params")
            params = preset(cfg_id)
        if seed is None:
            seed = default_seed(cfg_id if cfg_id is not None else 0)
        self.params = dict(params)
        self.seed = seed
        p = _Params(**{k: self.params[k] for k in PARAM_NAMES})
        h = lib.wl_create(ctypes.byref(p), ctypes.c_uint64(seed))
        if not h:
            raise ValueError(f"bad workload parameters: {params}")
        self._h = ctypes.c_void_p(h)
        self._lib = lib
        n_pool = lib.wl_prefix_pool_size(self._h)
        self.prefix_pool = np.empty(n_pool, np.int32)
        self.prefix_off = np.empty(self.params["n_prefix"], np.int64)
        self.prefix_len = np.empty(self.params["n_prefix"], np.int32)
        lib.wl_prefix_pool(self._h, _ptr(self.prefix_pool), _ptr(self.prefix_off), _ptr(self.prefix_len))

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and self._lib is not None:
            self._lib.wl_free(h)
            self._h = None

    @property
    def P(self) -> int:
        return self.params["P"]

    @property
    def B(self) -> int:
        return self.params["B"]

    @property
    def alpha(self) -> int:
        return self.params["alpha"]

    def _pool_with(self, n_suffix: int) -> np.ndarray:
        pool = np.empty(len(self.prefix_pool) + n_suffix, np.int32)
        pool[: len(self.prefix_pool)] = self.prefix_pool
        return pool

    def tree_size(self, p: int, which: int = 0) -> tuple[int, int, int]:
        a, b, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        if self._lib.wl_tree_size(self._h, p, which, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)) != 0:
            raise ValueError("bad tree index")
        return a.value, b.value, c.value

    def tree(self, p: int, which: int = 0) -> SeqList:
        """Sequences stored in tree p: which=0 the replica, which=1 the exact tree (stale case)."""
        n, ns, nt = self.tree_size(p, which)
        sb = np.empty(n + 1, np.int64)
        so = np.empty(ns, np.int64)
        sl = np.empty(ns, np.int32)
        pool = self._pool_with(nt)
        base = len(self.prefix_pool)
        self._lib.wl_tree_fill(self._h, p, which, _ptr(sb), _ptr(so), _ptr(sl), _ptr(pool[base:]), base)
        return SeqList(sb, so, sl, pool)

    def requests(self, b0: int = 0, b1: int | None = None, n_threads: int = 8,
                 out_tokens: np.ndarray | None = None) -> tuple[np.ndarray, np.ndarray]:
        """Requests [b0, b1) as (tokens int32, offsets int64[n+1]); out_tokens may supply (pinned) storage."""
        if b1 is None:
            b1 = self.B
        n_tok = self._lib.wl_requests_size(self._h, b0, b1, n_threads)
        if n_tok < 0:
            raise ValueError("bad request range")
        tokens = out_tokens[:n_tok] if out_tokens is not None else np.empty(n_tok, np.int32)
        offsets = np.empty(b1 - b0 + 1, np.int64)
        self._lib.wl_requests_fill(self._h, b0, b1, _ptr(tokens), _ptr(offsets), n_threads)
        return tokens, offsets

    def load(self, step: int = 0, vary_per_step: bool = False) -> np.ndarray:
        out = np.empty(self.P, np.int32)
        self._lib.wl_load_fill(self._h, step, int(vary_per_step), _ptr(out))
        return out

    def delta_make(self, step: int, del_frac: float, ins_frac: float, p0: int = 0, p1: int | None = None,
                   n_threads: int = 8) -> None:
        if p1 is None:
            p1 = self.P
        if self._lib.wl_delta_make(self._h, p0, p1, step, del_frac, ins_frac, n_threads) != 0:
            raise ValueError("bad delta arguments")

    def delta(self, p0: int = 0, p1: int | None = None, n_threads: int = 8) -> Delta:
        """The pending deltas of trees [p0, p1), concatenated."""
        if p1 is None:
            p1 = self.P
        a, b, c = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        if self._lib.wl_delta_size(self._h, p0, p1, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)) != 0:
            raise ValueError("bad tree range")
        n_ops, n_segs, n_tok = a.value, b.value, c.value
        op = np.empty(n_ops, np.int32)
        sb = np.empty(n_ops + 1, np.int64)
        so = np.empty(n_segs, np.int64)
        sl = np.empty(n_segs, np.int32)
        pool = self._pool_with(n_tok)
        pb = np.empty(p1 - p0 + 1, np.int64)
        base = len(self.prefix_pool)
        self._lib.wl_delta_fill(self._h, p0, p1, _ptr(op), _ptr(sb), _ptr(so), _ptr(sl), _ptr(pool[base:]), base,
                                _ptr(pb), n_threads)
        return Delta(op, SeqList(sb, so, sl, pool), pb)


# Raw PRNG access (tests of the published generators).
def splitmix64_sequence(seed: int, n: int) -> list[int]:
    st = ctypes.c_uint64(seed)
    return [int(_load().wl_splitmix64(ctypes.byref(st))) for _ in range(n)]


def xoshiro_sequence(seed: int, n: int) -> list[int]:
    s = (ctypes.c_uint64 * 4)()
    lib = _load()
    lib.wl_xoshiro_seed(ctypes.c_uint64(seed), ctypes.byref(s))
    return [int(lib.wl_xoshiro_next(ctypes.byref(s))) for _ in range(n)]


def xoshiro_from_state(state: list[int], n: int) -> list[int]:
    s = (ctypes.c_uint64 * 4)(*state)
    lib = _load()
    return [int(lib.wl_xoshiro_next(ctypes.byref(s))) for _ in range(n)]


def bounded_sequence(seed: int, rng: int, n: int) -> list[int]:
    s = (ctypes.c_uint64 * 4)()
    lib = _load()
    lib.wl_xoshiro_seed(ctypes.c_uint64(seed), ctypes.byref(s))
    return [int(lib.wl_bounded(ctypes.byref(s), ctypes.c_uint64(rng))) for _ in range(n)]


def zipf_index(n: int, s: float, u: float) -> int:
    return int(_load().wl_zipf_index(n, s, u))
