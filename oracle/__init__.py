"""CPU oracle for the prefix-cache-aware router (ctypes binding of ``oracle_tree.cpp``).

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares no code with the CUDA path and is never used as a
fallback for it.

What it computes, and the passages it follows:

* ``OTree`` -- a pointer radix tree over tokens holding a multiset of sequences.  ``insert`` is the
  paper's updateTrie / updateTrieEstimate (Section 2 primitive list, Algorithm 1); ``remove`` drops one
  stored occurrence (the DELETE op of an anti-entropy delta); ``match`` is PrefixMatch of Algorithm 1;
  ``export`` is the canonical full snapshot broadcast by sendTrie (Section 3, "Trie-broadcast loss").
* ``route`` -- Algorithm 1's argmax over all N tries, with the load term: maximise
  ``match - alpha*load``, ties to the lower load, then to the lower tree index.
* ``brute`` (pure Python) -- the same quantities written as their plain definitions, used to pin the
  C++ oracle on tiny inputs.
* ``lru`` (pure Python) -- a node's own trie with EvictLRUTrie (one least-recently-used leaf token at a
  time, Section 2 primitive list and Algorithm 1) and the expected hit rate of Section 5.
* ``update_estimates`` -- UpdateTrieEstimate of Algorithm 1 over a routed batch: request b is inserted
  into the tree it was routed to (the node's estimate of that peer's cache after a successful send).
* ``decide`` (pure Python) -- the route decision with excluded peers and a fallback target: a peer that
  pushes back (Section 3.2, hot specialist push-back) or is suspected to have failed (Section 3.3,
  in-flight forwarded request failure) is not a candidate, and the next-best candidate is where a request
  goes when forwarding to the best one times out.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# ORACLE_SO points the binding at another build of oracle_tree.cpp (used by the mutation test).
_SO = os.environ.get("ORACLE_SO") or os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compiles ``liboracle.so`` next to this file (plain g++)."""
    src = os.path.join(_HERE, "oracle_tree.cpp")
    if os.environ.get("ORACLE_SO"):
        return _SO
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(src):
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    subprocess.check_call(["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread", "-o", tmp, src])
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_SO)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        sig = {
            "otree_new": (vp, []),
            "otree_free": (None, [vp]),
            "otree_insert": (None, [vp, vp, i64]),
            "otree_remove": (ctypes.c_int, [vp, vp, i64]),
            "otree_match": (i64, [vp, vp, i64, vp]),
            "otree_insert_segmented": (None, [vp, vp, vp, vp, vp, i64, i64]),
            "otree_apply_ops": (i64, [vp, vp, vp, vp, vp, vp, i64, i64]),
            "otree_apply_ops_counted": (i64, [vp, vp, vp, vp, vp, vp, i64, i64, vp]),
            "otree_stats": (None, [vp, vp]),
            "otree_export": (ctypes.c_int, [vp] + [vp] * 8),
            "oracle_argmax": (i32, [i32, vp, vp, i32]),
            "oracle_route": (None, [vp, i32, vp, vp, i64, vp, i32, vp, vp, i32, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _p(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _i32(seq) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(seq, dtype=np.int32))


FLAT_FIELDS = ("label_off", "label_len", "child_begin", "child_count", "term_count",
               "child_first_tok", "child_idx", "labels")


class OTree:
    """One radix tree of the oracle."""

    def __init__(self):
        self._lib = _load()
        self._h = ctypes.c_void_p(self._lib.otree_new())

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None:
            self._lib.otree_free(h)
            self._h = None

    @property
    def handle(self):
        return self._h

    def insert(self, seq) -> None:
        a = _i32(seq)
        self._lib.otree_insert(self._h, _p(a), len(a))

    def remove(self, seq) -> bool:
        a = _i32(seq)
        return bool(self._lib.otree_remove(self._h, _p(a), len(a)))

    def match(self, req, counters: np.ndarray | None = None) -> int:
        a = _i32(req)
        return int(self._lib.otree_match(self._h, _p(a), len(a), _p(counters)))

    def insert_seqlist(self, sl, i0: int = 0, i1: int | None = None) -> None:
        """Inserts sequences [i0, i1) of a ``workload.SeqList``."""
        if i1 is None:
            i1 = len(sl)
        self._lib.otree_insert_segmented(self._h, _p(sl.seg_begin), _p(sl.seg_off), _p(sl.seg_len), _p(sl.pool),
                                         i0, i1)

    def apply_ops(self, op: np.ndarray, sl, i0: int = 0, i1: int | None = None) -> int:
        """Applies ops [i0, i1) (0 INSERT, 1 DELETE) in order; returns the number of absent DELETEs."""
        if i1 is None:
            i1 = len(op)
        return int(self._lib.otree_apply_ops(self._h, _p(op), _p(sl.seg_begin), _p(sl.seg_off), _p(sl.seg_len),
                                             _p(sl.pool), i0, i1))

    def apply_ops_counted(self, op: np.ndarray, sl, counters: np.ndarray, i0: int = 0, i1: int | None = None) -> int:
        """As ``apply_ops``, adding each op's touched-byte counters to ``counters`` (int64[8]): the read-only
        PrefixMatch walk of its sequence before the op (tokens compared, nodes visited, child-search bytes),
        then sequence tokens, pool runs, INSERTs, label tokens the INSERTs add, DELETEs."""
        if i1 is None:
            i1 = len(op)
        assert counters.dtype == np.int64 and counters.size >= 8
        return int(self._lib.otree_apply_ops_counted(self._h, _p(op), _p(sl.seg_begin), _p(sl.seg_off),
                                                     _p(sl.seg_len), _p(sl.pool), i0, i1, _p(counters)))

    def stats(self) -> tuple[int, int, int]:
        """(nodes including the root, label tokens, stored sequences)."""
        out = np.zeros(3, np.int64)
        self._lib.otree_stats(self._h, _p(out))
        return int(out[0]), int(out[1]), int(out[2])

    def export(self) -> dict:
        """Canonical flat snapshot: dict of int32 arrays named as in ``FLAT_FIELDS``."""
        n, lab, _ = self.stats()
        d = {f: np.zeros(n, np.int32) for f in FLAT_FIELDS[:5]}
        d["child_first_tok"] = np.zeros(max(n - 1, 0), np.int32)
        d["child_idx"] = np.zeros(max(n - 1, 0), np.int32)
        d["labels"] = np.zeros(lab, np.int32)
        rc = self._lib.otree_export(self._h, *[_p(d[f]) for f in FLAT_FIELDS])
        if rc != 0:
            raise OverflowError("tree too large for the int32 flat format")
        return d


def build_trees(seqlists, n_threads: int = 8) -> list[OTree]:
    """One OTree per ``workload.SeqList`` (built concurrently; ctypes releases the GIL)."""
    trees = [OTree() for _ in seqlists]
    with ThreadPoolExecutor(max_workers=max(1, n_threads)) as ex:
        list(ex.map(lambda ts: ts[0].insert_seqlist(ts[1]), zip(trees, seqlists)))
    return trees


def argmax_peer(match_row, load, alpha: int) -> int:
    m = _i32(match_row)
    ld = _i32(load)
    return int(_load().oracle_argmax(len(m), _p(m), _p(ld), alpha))


def route(trees, tokens: np.ndarray, offsets: np.ndarray, load, alpha: int, n_threads: int = 8):
    """Routes a CSR batch.  Returns (match int32[B,P], peer int32[B], counters int64[4]) where counters are
    (tokens compared, nodes visited, child-search bytes, request tokens)."""
    lib = _load()
    P = len(trees)
    B = len(offsets) - 1
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    offsets = np.ascontiguousarray(offsets, dtype=np.int64)
    ld = _i32(load)
    arr = (ctypes.c_void_p * P)(*[t.handle.value for t in trees])
    match = np.zeros((B, P), np.int32)
    peer = np.zeros(B, np.int32)
    ctr = np.zeros(4, np.int64)
    lib.oracle_route(arr, P, _p(tokens), _p(offsets), B, _p(ld), alpha, _p(match), _p(peer), n_threads, _p(ctr))
    return match, peer, ctr


def update_estimates(trees, tokens: np.ndarray, offsets: np.ndarray, peer) -> None:
    """Algorithm 1, after a request is sent to node k and acknowledged: UpdateTrieEstimate(r, k) inserts r
    into the sender's estimate of k's trie (Section 2 primitive list).  For a routed batch: request b,
    tokens[offsets[b] .. offsets[b+1]), is inserted into trees[peer[b]]; a request with peer[b] < 0 (no
    target) is skipped.  One plain insert per request, in batch order."""
    for b in range(len(offsets) - 1):
        k = int(peer[b])
        if k >= 0:
            trees[k].insert(tokens[int(offsets[b]):int(offsets[b + 1])])


def decide(match, load, alpha: int, excluded=None):
    """Best and next-best target of every request from its match row, skipping excluded peers.

    For row b of ``match`` [B, P], the candidates are the peers p with ``excluded[p]`` false, ordered by
    the tuple (match[b, p] - alpha*load[p], -load[p], -p): Algorithm 1's argmax with the load term and the
    tie-breaks of ``route``.  Returns (best int32[B], next int32[B]), the first and second candidate of that
    order, -1 where there are fewer candidates.  Section 3.2 takes a pushed-back peer out of routing and
    Section 3.3 a suspected-failed one; on a forwarding timeout Section 3.3 falls back to the next-best
    target.  Plain Python over the tuples.

    A match entry below 0 counts as 0: PrefixMatch is a count of tokens, so no route produces one, and a
    negative entry in a caller's matrix is read as "nothing matched" (the reading the device decision
    applies too)."""
    match = np.asarray(match)
    B, P = match.shape
    ex = np.zeros(P, bool) if excluded is None else np.asarray(excluded).astype(bool)
    best = np.full(B, -1, np.int32)
    nxt = np.full(B, -1, np.int32)
    for b in range(B):
        cand = sorted(((max(int(match[b, p]), 0) - alpha * int(load[p]), -int(load[p]), -p)
                       for p in range(P) if not ex[p]), reverse=True)
        if cand:
            best[b] = -cand[0][2]
        if len(cand) > 1:
            nxt[b] = -cand[1][2]
    return best, nxt


def delta_touched_bytes(counters: np.ndarray) -> int:
    """Algorithmic bytes of anti-entropy ops from ``apply_ops_counted``'s counters: per op, its input (4 B op
    code, 8 B sequence start, 12 B per pool run, 4 B per sequence token), its walk (4 B per token compared,
    20 B per node visited, the child-search bytes), and what it writes (an INSERT: 4 B per new label token
    plus 36 B for a new node record and child entry; a DELETE: a 16 B node record)."""
    c = [int(x) for x in counters]
    n_ops = c[5] + c[7]
    return (12 * n_ops + 12 * c[4] + 4 * c[3]) + (4 * c[0] + 20 * c[1] + c[2]) + (4 * c[6] + 36 * c[5] + 16 * c[7])


def touched_bytes(counters: np.ndarray) -> int:
    """Algorithmic bytes of a routed batch from the oracle's counters: 4 B per token compared, 20 B per node
    visited, the child-search bytes, and 4 B per request token."""
    c = [int(x) for x in counters]
    return 4 * c[0] + 20 * c[1] + c[2] + 4 * c[3]
