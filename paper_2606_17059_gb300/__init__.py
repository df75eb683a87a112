"""GB300 batched routing engine for decentralized, prefix-cache-aware LLM routing.

Thin ctypes binding of ``libp2prouter.so`` (C ABI in ``include/p2p_router.h``).  The functions below
carry the C names and only marshal arguments: every step of routing, matching and tree patching runs in
the library's CUDA kernels.  Device buffers are passed as torch CUDA tensors (or raw integer addresses);
host buffers as numpy arrays.  There is no CPU fallback: importing works without a GPU, but every call
needs the built library and a CUDA device, and raises otherwise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

__all__ = [
    "P2PError", "Router", "build", "library_path",
    "p2p_router_create", "p2p_router_destroy", "p2p_router_set_stream", "p2p_router_sync", "p2p_last_error",
    "p2p_router_num_trees", "p2p_router_launch_count", "p2p_snapshot_build", "p2p_snapshot_view", "p2p_snapshot_free",
    "p2p_flat_tree_validate", "p2p_tree_upload", "p2p_tree_build", "p2p_tree_download", "p2p_tree_apply_delta",
    "p2p_tree_apply_delta_static", "p2p_tree_stats", "p2p_route_batch", "p2p_route_batch_host", "p2p_route_decide",
    "p2p_router_kernel_clock", "p2p_router_kernel_time", "p2p_update_estimates", "p2p_route_batch_decide",
    "p2p_lru_enable", "p2p_lru_insert", "p2p_lru_access", "p2p_lru_evict", "p2p_hit_rate", "p2p_route_prepare",
]

P2P_OK, P2P_E_INVAL, P2P_E_NOMEM, P2P_E_FORMAT, P2P_E_CUDA, P2P_E_DEVICE = 0, -1, -2, -3, -4, -5
P2P_OP_INSERT, P2P_OP_DELETE = 0, 1
P2P_MEM_HOST, P2P_MEM_DEVICE = 0, 1
ERROR_NAMES = {-1: "P2P_E_INVAL", -2: "P2P_E_NOMEM", -3: "P2P_E_FORMAT", -4: "P2P_E_CUDA", -5: "P2P_E_DEVICE"}
FLAT_FIELDS = ("label_off", "label_len", "child_begin", "child_count", "term_count",
               "child_first_tok", "child_idx", "labels")

library_path = _build.LIB


def build(force: bool = False) -> str:
    return _build.build(force=force)


class P2PError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{ERROR_NAMES.get(code, code)}: {msg}")
        self.code = code


_vp = ctypes.c_void_p
_i32, _i64 = ctypes.c_int32, ctypes.c_int64


class FlatTree(ctypes.Structure):
    _fields_ = [("n_nodes", _i32), ("n_labels", _i32)] + [(f, _vp) for f in FLAT_FIELDS]


class Seqs(ctypes.Structure):
    _fields_ = [("n", _i64), ("seg_begin", _vp), ("seg_off", _vp), ("seg_len", _vp), ("pool", _vp),
                ("n_segs", _i64), ("n_pool", _i64)]


class Delta(ctypes.Structure):
    _fields_ = [("op", _vp), ("seqs", Seqs), ("peer_begin", _vp), ("mem", _i32)]


_lib = None


def _load():
    """Loads the CUDA library (building it first when a source is newer).  Raises if it cannot."""
    global _lib
    if _lib is None:
        path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"CUDA library missing: {path}")
        lib = ctypes.CDLL(path)
        P = ctypes.POINTER
        sig = {
            "p2p_router_create": (ctypes.c_int, [_i32, P(_vp)]),
            "p2p_router_destroy": (None, [_vp]),
            "p2p_router_set_stream": (ctypes.c_int, [_vp, _vp]),
            "p2p_router_sync": (ctypes.c_int, [_vp]),
            "p2p_last_error": (ctypes.c_char_p, [_vp]),
            "p2p_router_num_trees": (_i32, [_vp]),
            "p2p_router_launch_count": (_i64, [_vp]),
            "p2p_snapshot_build": (ctypes.c_int, [P(Seqs), P(_vp)]),
            "p2p_snapshot_view": (None, [_vp, P(FlatTree)]),
            "p2p_snapshot_free": (None, [_vp]),
            "p2p_flat_tree_validate": (ctypes.c_int, [P(FlatTree)]),
            "p2p_tree_upload": (ctypes.c_int, [_vp, _i32, P(FlatTree)]),
            "p2p_tree_build": (ctypes.c_int, [_vp, _i32, P(Seqs)]),
            "p2p_tree_download": (ctypes.c_int, [_vp, _i32, P(_vp)]),
            "p2p_tree_apply_delta": (ctypes.c_int, [_vp, _i32, P(Delta), P(_i64)]),
            "p2p_tree_apply_delta_static": (ctypes.c_int, [_vp, _i32, P(Delta), P(_i64)]),
            "p2p_tree_stats": (ctypes.c_int, [_vp, _i32, P(_i64 * 9)]),
            "p2p_route_batch": (ctypes.c_int, [_vp, _vp, _i64, _vp, _i64, _vp, _i32, _vp, _vp]),
            "p2p_route_batch_host": (ctypes.c_int, [_vp, _vp, _vp, _i64, _vp, _i32, _vp, _vp]),
            "p2p_route_decide": (ctypes.c_int, [_vp, _vp, _i64, _vp, _i32, _vp, _vp, _vp]),
            "p2p_router_kernel_clock": (ctypes.c_int, [_vp, _i32]),
            "p2p_update_estimates": (ctypes.c_int, [_vp, _vp, _i64, _vp, _i64, _vp, P(_i64)]),
            "p2p_route_batch_decide": (ctypes.c_int, [_vp, _vp, _i64, _vp, _i64, _vp, _i32, _vp, _vp, _vp, _vp]),
            "p2p_lru_enable": (ctypes.c_int, [_vp, _i32]),
            "p2p_lru_insert": (ctypes.c_int, [_vp, _i32, _vp, _i64, _vp, _i64, _i64]),
            "p2p_lru_access": (ctypes.c_int, [_vp, _i32, _vp, _i64, _vp, _i64, _i64, _vp]),
            "p2p_lru_evict": (ctypes.c_int, [_vp, _i32, _i64, P(_i64)]),
            "p2p_hit_rate": (ctypes.c_int, [_vp, _vp, _vp, _i64, _vp, _vp]),
            "p2p_route_prepare": (ctypes.c_int, [_vp, _vp, _i64, _vp, _i64]),
            "p2p_router_kernel_time": (ctypes.c_int, [_vp, _i32, P(ctypes.c_char_p), P(_i64), P(ctypes.c_double)]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def exported_symbols() -> list[str]:
    """Names of the C entry points this binding declares (all must be exported by the library)."""
    return [n for n in __all__ if n.startswith("p2p_")]


def _check(rc: int, r=None):
    if rc != P2P_OK:
        msg = _load().p2p_last_error(r)
        raise P2PError(rc, msg.decode() if msg else "")


def _addr(x) -> int | None:
    """Address of a torch tensor / numpy array / integer (None stays NULL)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("array must be C-contiguous")
        return x.ctypes.data
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensor must be contiguous")
        return x.data_ptr()
    raise TypeError(f"cannot take the address of {type(x)}")


def _host_i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _load_vec(r, load) -> np.ndarray:
    """The per-tree load as a host int32 array; the library reads one entry per tree."""
    ld = _host_i32(load)
    n = p2p_router_num_trees(r)
    if ld.ndim != 1 or ld.size != n:
        raise ValueError(f"load must have one entry per tree ({n}), got shape {ld.shape}")
    return ld


def _seqs_struct(sl, keep: list) -> Seqs:
    """Seqs struct from an object with seg_begin/seg_off/seg_len/pool (numpy arrays or CUDA tensors)."""
    arrs = []
    for name, dt in (("seg_begin", np.int64), ("seg_off", np.int64), ("seg_len", np.int32), ("pool", np.int32)):
        a = getattr(sl, name)
        if isinstance(a, np.ndarray):
            a = np.ascontiguousarray(a, dtype=dt)
        arrs.append(a)
    keep.extend(arrs)
    sb, so, slen, pool = arrs
    return Seqs(len(sb) - 1, _addr(sb), _addr(so), _addr(slen), _addr(pool), len(so), len(pool))


# ---- the C entry points ---------------------------------------------------------------------------------

def p2p_router_create(P: int):
    h = _vp()
    _check(_load().p2p_router_create(P, ctypes.byref(h)))
    return h


def p2p_router_destroy(r) -> None:
    _load().p2p_router_destroy(r)


def p2p_router_set_stream(r, stream=None) -> None:
    s = None
    if stream is not None:
        s = stream if isinstance(stream, int) else stream.cuda_stream
    _check(_load().p2p_router_set_stream(r, s), r)


def p2p_router_sync(r) -> None:
    _check(_load().p2p_router_sync(r), r)


def p2p_last_error(r=None) -> str:
    m = _load().p2p_last_error(r)
    return m.decode() if m else ""


def p2p_router_num_trees(r) -> int:
    return int(_load().p2p_router_num_trees(r))


def p2p_router_launch_count(r) -> int:
    return int(_load().p2p_router_launch_count(r))


KERNEL_COUNT = 27  # P2P_KERNEL_COUNT: kernels the kernel clock keeps totals for (indices 0 .. 26)


def p2p_router_kernel_clock(r, on: bool) -> None:
    _check(_load().p2p_router_kernel_clock(r, 1 if on else 0), r)


def p2p_router_kernel_time(r, i: int) -> tuple[str, int, float]:
    """(kernel name, timed launches, summed device ms) of kernel i since the clock was switched on."""
    name = ctypes.c_char_p()
    n = _i64()
    ms = ctypes.c_double()
    _check(_load().p2p_router_kernel_time(r, i, ctypes.byref(name), ctypes.byref(n), ctypes.byref(ms)), r)
    return (name.value.decode() if name.value else ""), int(n.value), float(ms.value)


def p2p_snapshot_build(seqlist):
    keep = []
    s = _seqs_struct(seqlist, keep)
    h = _vp()
    _check(_load().p2p_snapshot_build(ctypes.byref(s), ctypes.byref(h)))
    return h


def p2p_snapshot_view(snap) -> dict:
    """Copies a snapshot's arrays into numpy (dict keyed like ``FLAT_FIELDS``)."""
    v = FlatTree()
    _load().p2p_snapshot_view(snap, ctypes.byref(v))
    n, nl = v.n_nodes, v.n_labels
    sizes = {f: n for f in FLAT_FIELDS[:5]}
    sizes.update(child_first_tok=n - 1, child_idx=n - 1, labels=nl)
    out = {}
    for f in FLAT_FIELDS:
        cnt = sizes[f]
        addr = getattr(v, f)
        if cnt == 0 or not addr:
            out[f] = np.zeros(0, np.int32)
        else:
            out[f] = np.ctypeslib.as_array((ctypes.c_int32 * cnt).from_address(addr)).copy()
    return out


def p2p_snapshot_free(snap) -> None:
    _load().p2p_snapshot_free(snap)


def _flat_struct(flat: dict, keep: list) -> FlatTree:
    arrs = {f: _host_i32(flat[f]) for f in FLAT_FIELDS}
    keep.append(arrs)
    t = FlatTree()
    t.n_nodes = len(arrs["label_off"])
    t.n_labels = len(arrs["labels"])
    for f in FLAT_FIELDS:
        setattr(t, f, arrs[f].ctypes.data if len(arrs[f]) else None)
    return t


def p2p_flat_tree_validate(flat: dict) -> int:
    keep = []
    t = _flat_struct(flat, keep)
    return int(_load().p2p_flat_tree_validate(ctypes.byref(t)))


def p2p_tree_upload(r, peer: int, flat: dict) -> None:
    keep = []
    t = _flat_struct(flat, keep)
    _check(_load().p2p_tree_upload(r, peer, ctypes.byref(t)), r)


def p2p_tree_build(r, peer: int, seqlist) -> None:
    keep = []
    s = _seqs_struct(seqlist, keep)
    _check(_load().p2p_tree_build(r, peer, ctypes.byref(s)), r)


def p2p_tree_download(r, peer: int) -> dict:
    h = _vp()
    _check(_load().p2p_tree_download(r, peer, ctypes.byref(h)), r)
    try:
        return p2p_snapshot_view(h)
    finally:
        p2p_snapshot_free(h)


def p2p_tree_apply_delta(r, peer: int, op, seqlist, peer_begin=None, on_device: bool = False) -> int:
    """Applies an ordered INSERT/DELETE delta; returns the number of DELETEs of absent sequences.
    With on_device the op/segment/pool arrays are CUDA tensors, else numpy arrays."""
    keep = []
    if isinstance(op, np.ndarray):
        op = np.ascontiguousarray(op, dtype=np.int32)
    if isinstance(peer_begin, np.ndarray):
        peer_begin = np.ascontiguousarray(peer_begin, dtype=np.int64)
    keep += [op, peer_begin]
    d = Delta(_addr(op), _seqs_struct(seqlist, keep), _addr(peer_begin), P2P_MEM_DEVICE if on_device else P2P_MEM_HOST)
    absent = _i64()
    _check(_load().p2p_tree_apply_delta(r, peer, ctypes.byref(d), ctypes.byref(absent)), r)
    return int(absent.value)


def p2p_tree_apply_delta_static(r, peer: int, op, seqlist, peer_begin=None) -> int:
    """The allocation-free delta call: op/segment/pool arrays (and peer_begin) must be CUDA tensors.
    Returns the number of DELETEs of absent sequences."""
    keep = [op, peer_begin]
    d = Delta(_addr(op), _seqs_struct(seqlist, keep), _addr(peer_begin), P2P_MEM_DEVICE)
    absent = _i64()
    _check(_load().p2p_tree_apply_delta_static(r, peer, ctypes.byref(d), ctypes.byref(absent)), r)
    return int(absent.value)


def p2p_update_estimates(r, tokens, n_tokens: int, offsets, B: int, peer) -> int:
    """Inserts request b into tree peer[b] for every routed request (UpdateTrieEstimate / UpdateTrie of
    Algorithm 1); tokens, offsets and peer are CUDA tensors (or addresses).  Returns the requests inserted."""
    n = _i64()
    _check(_load().p2p_update_estimates(r, _addr(tokens), n_tokens, _addr(offsets), B, _addr(peer), ctypes.byref(n)), r)
    return int(n.value)


def p2p_lru_enable(r, tree: int) -> None:
    _check(_load().p2p_lru_enable(r, tree), r)


def p2p_lru_insert(r, tree: int, tokens, n_tokens: int, offsets, B: int, time: int) -> None:
    """UpdateTrie of a batch at `time` (CUDA tensors tokens/offsets)."""
    _check(_load().p2p_lru_insert(r, tree, _addr(tokens), n_tokens, _addr(offsets), B, time), r)


def p2p_lru_access(r, tree: int, tokens, n_tokens: int, offsets, B: int, time: int, out_match=None) -> None:
    """Requests served at `time`: their matched tokens are touched; out_match (CUDA int32 [B] or None)."""
    _check(_load().p2p_lru_access(r, tree, _addr(tokens), n_tokens, _addr(offsets), B, time, _addr(out_match)), r)


def p2p_lru_evict(r, tree: int, n_tokens: int) -> int:
    """Evicts the n_tokens least recently used leaf tokens; returns how many were evicted."""
    n = _i64()
    _check(_load().p2p_lru_evict(r, tree, n_tokens, ctypes.byref(n)), r)
    return int(n.value)


def p2p_hit_rate(r, match, offsets, B: int, peer, out) -> None:
    """Expected hit rate match[b, peer[b]] / len(b) of routed requests (CUDA tensors; out float32 [B])."""
    _check(_load().p2p_hit_rate(r, _addr(match), _addr(offsets), B, _addr(peer), _addr(out)), r)


STAT_NAMES = ("live_nodes", "node_slots", "child_entries", "label_tokens", "stale_child", "stale_label",
              "cap_node", "cap_child", "cap_label")


def p2p_tree_stats(r, peer: int) -> dict:
    out = (_i64 * 9)()
    _check(_load().p2p_tree_stats(r, peer, ctypes.byref(out)), r)
    return dict(zip(STAT_NAMES, [int(x) for x in out]))


def p2p_route_batch(r, tokens, n_tokens: int, offsets, B: int, load, alpha: int, out_match, out_peer) -> None:
    """Device routing: tokens/offsets/out_match/out_peer are CUDA tensors (or addresses), load is host."""
    ld = _load_vec(r, load)
    _check(_load().p2p_route_batch(r, _addr(tokens), n_tokens, _addr(offsets), B, ld.ctypes.data, alpha,
                                   _addr(out_match), _addr(out_peer)), r)


def _mask(r, excluded, n: int):
    if excluded is None:
        return None
    ex = np.ascontiguousarray(np.asarray(excluded), dtype=np.uint8)
    if ex.size != n:
        raise ValueError(f"excluded must have one entry per tree ({n})")
    return ex


def p2p_route_batch_decide(r, tokens, n_tokens: int, offsets, B: int, load, alpha: int, excluded, out_match, out_peer,
                           out_next=None) -> None:
    """Device routing with excluded trees and the next-best target decided in the walk kernels; tokens, offsets,
    out_match, out_peer and out_next (or None) are CUDA tensors, load and excluded (uint8 per tree, or None)
    host arrays."""
    ld = _load_vec(r, load)
    ex = _mask(r, excluded, ld.size)
    _check(_load().p2p_route_batch_decide(r, _addr(tokens), n_tokens, _addr(offsets), B, ld.ctypes.data, alpha,
                                          ex.ctypes.data if ex is not None else None, _addr(out_match),
                                          _addr(out_peer), _addr(out_next)), r)


def p2p_route_prepare(r, tokens, n_tokens: int, offsets, B: int) -> None:
    """Announces the next batch (CUDA tensors): its grouping overlaps the next delta kernel."""
    _check(_load().p2p_route_prepare(r, _addr(tokens), n_tokens, _addr(offsets), B), r)


def p2p_route_decide(r, match, B: int, load, alpha: int, excluded, out_peer, out_next) -> None:
    """Best and next-best non-excluded tree per request from a device match matrix [B, P] (CUDA tensors or
    addresses); load and excluded (uint8 per tree, or None) are host arrays."""
    ld = _load_vec(r, load)
    n = ld.size
    ex = None
    if excluded is not None:
        ex = np.ascontiguousarray(np.asarray(excluded), dtype=np.uint8)
    if ex is not None and ex.size != n:
        raise ValueError(f"excluded must have one entry per tree ({n})")
    _check(_load().p2p_route_decide(r, _addr(match), B, ld.ctypes.data, alpha,
                                    ex.ctypes.data if ex is not None else None, _addr(out_peer), _addr(out_next)), r)


def p2p_route_batch_host(r, tokens: np.ndarray, offsets: np.ndarray, B: int, load, alpha: int,
                         out_match: np.ndarray, out_peer: np.ndarray) -> None:
    """Host routing: every array is a host numpy array (pinned memory copies faster)."""
    ld = _load_vec(r, load)
    for a, dt in ((tokens, np.int32), (offsets, np.int64), (out_match, np.int32), (out_peer, np.int32)):
        if not isinstance(a, np.ndarray) or a.dtype != dt or not a.flags["C_CONTIGUOUS"]:
            raise TypeError("host routing needs C-contiguous numpy arrays (int32 tokens/outputs, int64 offsets)")
    if B > 0 and (offsets.size < B + 1 or out_match.size < B * ld.size or out_peer.size < B
                  or tokens.size < int(offsets[B])):
        raise ValueError("host routing arrays are smaller than B requests need")
    _check(_load().p2p_route_batch_host(r, _addr(tokens), _addr(offsets), B, ld.ctypes.data, alpha,
                                        _addr(out_match), _addr(out_peer)), r)


# ---- convenience wrapper ----------------------------------------------------------------------------------

class Router:
    """Owns one p2p_router.  Device work runs on torch's current CUDA stream at construction."""

    def __init__(self, P: int, stream=None):
        import torch
        self.P = P
        self._h = p2p_router_create(P)
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        p2p_router_set_stream(self._h, self.stream)

    @property
    def handle(self):
        return self._h

    def close(self):
        if getattr(self, "_h", None) is not None:
            p2p_router_destroy(self._h)
            self._h = None

    def __del__(self):
        self.close()

    def build(self, peer: int, seqlist) -> None:
        p2p_tree_build(self._h, peer, seqlist)

    def upload(self, peer: int, flat: dict) -> None:
        p2p_tree_upload(self._h, peer, flat)

    def download(self, peer: int) -> dict:
        return p2p_tree_download(self._h, peer)

    def stats(self, peer: int) -> dict:
        return p2p_tree_stats(self._h, peer)

    def apply_delta(self, peer: int, op, seqlist, peer_begin=None, on_device: bool = False) -> int:
        return p2p_tree_apply_delta(self._h, peer, op, seqlist, peer_begin, on_device)

    def sync(self) -> None:
        p2p_router_sync(self._h)

    def update_estimates(self, tokens, offsets, peer) -> int:
        """After routing: request b (CUDA tensors tokens/offsets) goes into tree peer[b]; returns the count."""
        return p2p_update_estimates(self._h, tokens, tokens.numel(), offsets, offsets.numel() - 1, peer)

    def launch_count(self) -> int:
        return p2p_router_launch_count(self._h)

    def kernel_clock(self, on: bool) -> None:
        p2p_router_kernel_clock(self._h, on)

    def kernel_times(self) -> dict:
        """{kernel name: (launches, summed device ms)} of the kernels launched since the clock was switched on."""
        out = {}
        for i in range(KERNEL_COUNT):
            name, n, ms = p2p_router_kernel_time(self._h, i)
            if n:
                out[name] = (n, ms)
        return out

    def route(self, tokens, offsets, load, alpha: int, out_match=None, out_peer=None):
        """tokens (int32) and offsets (int64) are CUDA tensors; returns (match [B,P], peer [B]) tensors."""
        import torch
        B = offsets.numel() - 1
        if out_match is None:
            out_match = torch.empty((B, self.P), dtype=torch.int32, device=tokens.device)
        if out_peer is None:
            out_peer = torch.empty(B, dtype=torch.int32, device=tokens.device)
        p2p_route_batch(self._h, tokens, tokens.numel(), offsets, B, load, alpha, out_match, out_peer)
        return out_match, out_peer

    def route_decide(self, tokens, offsets, load, alpha: int, excluded=None, want_next: bool = True):
        """Routing with excluded trees and the next-best target in one pass; returns (match [B,P], peer [B],
        next [B] or None) CUDA tensors."""
        import torch
        B = offsets.numel() - 1
        m = torch.empty((B, self.P), dtype=torch.int32, device=tokens.device)
        p = torch.empty(B, dtype=torch.int32, device=tokens.device)
        n = torch.empty(B, dtype=torch.int32, device=tokens.device) if want_next else None
        p2p_route_batch_decide(self._h, tokens, tokens.numel(), offsets, B, load, alpha, excluded, m, p, n)
        return m, p, n

    def decide(self, match, load, alpha: int, excluded=None, out_peer=None, out_next=None):
        """match is a CUDA int32 tensor [B, P]; returns (peer [B], next [B]) CUDA tensors."""
        import torch
        B = match.shape[0]
        if out_peer is None:
            out_peer = torch.empty(B, dtype=torch.int32, device=match.device)
        if out_next is None:
            out_next = torch.empty(B, dtype=torch.int32, device=match.device)
        p2p_route_decide(self._h, match, B, load, alpha, excluded, out_peer, out_next)
        return out_peer, out_next

    def route_host(self, tokens: np.ndarray, offsets: np.ndarray, load, alpha: int, out_match=None, out_peer=None):
        B = len(offsets) - 1
        if out_match is None:
            out_match = np.empty((B, self.P), np.int32)
        if out_peer is None:
            out_peer = np.empty(B, np.int32)
        p2p_route_batch_host(self._h, tokens, offsets, B, load, alpha, out_match, out_peer)
        return out_match, out_peer
