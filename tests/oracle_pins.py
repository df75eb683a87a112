"""Checks that pin the CPU oracle to things other than itself.

Each check returns a list of failure strings (empty = pass), so that the same checks run as ordinary tests
and, in the mutation test, against deliberately broken builds of the oracle.

Pins used:
* the hand-worked example in ``golden/worked_example.json`` (match, routes, counters, snapshots);
* brute force on tiny inputs: match = max LCP over the stored multiset; route = tuple argmax; the
  canonical snapshot rebuilt from the set of all prefixes (``oracle.brute``);
* invariants: insert r then match r = |r|; match never exceeds |r|; insertion order does not change the
  snapshot; inserting then deleting a sequence restores the snapshot; insert never lowers and delete never
  raises a match; the empty tree matches 0; alpha = 0 is the pure argmax of match; P = 1 routes to 0.
"""
from __future__ import annotations

import json
import os
import random

import numpy as np

import oracle
import oracle.brute as brute

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _snap_eq(a: dict, b: dict) -> bool:
    return all(list(np.asarray(a[k]).tolist()) == list(b[k]) for k in oracle.FLAT_FIELDS)


def check_golden() -> list[str]:
    g = json.load(open(os.path.join(GOLDEN, "worked_example.json")))
    fails = []
    trees = []
    for i, seqs in enumerate(g["trees"]):
        t = oracle.OTree()
        for s in seqs:
            t.insert(s)
        trees.append(t)
        if not _snap_eq(t.export(), g["snapshots"][i]):
            fails.append(f"golden snapshot {i}")
    for b, r in enumerate(g["requests"]):
        for p, t in enumerate(trees):
            if t.match(r) != g["match"][b][p]:
                fails.append(f"golden match b={b} p={p}")
    toks = np.array([x for r in g["requests"] for x in r], np.int32)
    offs = np.cumsum([0] + [len(r) for r in g["requests"]]).astype(np.int64)
    for case in g["routes"]:
        m, peer, _ = oracle.route(trees, toks, offs, case["load"], case["alpha"], n_threads=2)
        if m.tolist() != g["match"]:
            fails.append("golden route match")
        if peer.tolist() != case["peer"]:
            fails.append(f"golden route peer alpha={case['alpha']} load={case['load']}")
    for c in g["counters"]:
        ctr = np.zeros(3, np.int64)
        trees[c["tree"]].match(g["requests"][c["request"]], ctr)
        if ctr.tolist() != [c["compared"], c["visited"], c["search_bytes"]]:
            fails.append(f"golden counters {c} got {ctr.tolist()}")
    return fails


def check_brute(seed: int = 0, trials: int = 150) -> list[str]:
    rng = random.Random(seed)
    fails = []
    for trial in range(trials):
        V = rng.choice([2, 3, 4])
        P = rng.randint(1, 4)
        stored = [[[rng.randrange(V) for _ in range(rng.randint(0, 9))] for _ in range(rng.randint(0, 12))]
                  for _ in range(P)]
        trees = []
        for seqs in stored:
            t = oracle.OTree()
            for s in seqs:
                t.insert(s)
            trees.append(t)
            if not _snap_eq(t.export(), brute.canonical_snapshot(seqs)):
                fails.append(f"snapshot trial={trial}")
        reqs = [[rng.randrange(V) for _ in range(rng.randint(0, 11))] for _ in range(8)]
        load = [rng.randrange(4) for _ in range(P)]
        alpha = rng.randrange(3)
        rows, peers = brute.route(reqs, stored, load, alpha)
        toks = np.array([x for r in reqs for x in r], np.int32)
        offs = np.cumsum([0] + [len(r) for r in reqs]).astype(np.int64)
        m, peer, _ = oracle.route(trees, toks, offs, load, alpha, n_threads=1 + trial % 3)
        if m.tolist() != rows:
            fails.append(f"match trial={trial}")
        if peer.tolist() != peers:
            fails.append(f"route trial={trial}")
        # Deletes: remove a random half (plus some absent sequences) and compare again.
        for p, seqs in enumerate(stored):
            order = list(range(len(seqs)))
            rng.shuffle(order)
            keep = list(seqs)
            for i in order[: len(seqs) // 2]:
                if not trees[p].remove(seqs[i]):
                    fails.append(f"remove stored trial={trial}")
                keep.remove(seqs[i])
            absent = [rng.randrange(V) for _ in range(rng.randint(0, 9))]
            was_there = absent in keep
            if trees[p].remove(absent) != was_there:
                fails.append(f"remove absent trial={trial}")
            if was_there:
                keep.remove(absent)
            if not _snap_eq(trees[p].export(), brute.canonical_snapshot(keep)):
                fails.append(f"snapshot after delete trial={trial}")
            for r in reqs:
                if trees[p].match(r) != brute.match(r, keep):
                    fails.append(f"match after delete trial={trial}")
    return fails


def check_invariants(seed: int = 1, trials: int = 60) -> list[str]:
    rng = random.Random(seed)
    fails = []
    for trial in range(trials):
        V = rng.choice([2, 3, 4, 50])
        seqs = [[rng.randrange(V) for _ in range(rng.randint(0, 12))] for _ in range(rng.randint(1, 15))]
        t = oracle.OTree()
        if t.match(seqs[0]) != 0:
            fails.append("empty tree match")
        for s in seqs:
            t.insert(s)
        for s in seqs:
            if t.match(s) != len(s):
                fails.append("insert-then-match")
        snap = t.export()
        # Insertion order does not matter.
        t2 = oracle.OTree()
        perm = list(seqs)
        rng.shuffle(perm)
        for s in perm:
            t2.insert(s)
        if not _snap_eq(t2.export(), snap):
            fails.append("order dependence")
        # Insert then delete restores the snapshot; insert never lowers a match, delete never raises one.
        extra = [rng.randrange(V) for _ in range(rng.randint(0, 12))]
        probes = [[rng.randrange(V) for _ in range(rng.randint(0, 12))] for _ in range(6)]
        before = [t.match(r) for r in probes]
        t.insert(extra)
        after = [t.match(r) for r in probes]
        if any(a < b for a, b in zip(after, before)):
            fails.append("insert lowered a match")
        if not t.remove(extra):
            fails.append("remove of inserted")
        if not _snap_eq(t.export(), snap):
            fails.append("insert+delete not identity")
        if [t.match(r) for r in probes] != before:
            fails.append("delete changed matches")
        for r in probes:
            if t.match(r) > len(r):
                fails.append("match > |r|")
        # alpha = 0: pure argmax of match, ties to the lower load then the lower index.
        m = [rng.randrange(5) for _ in range(5)]
        ld = [rng.randrange(3) for _ in range(5)]
        best = max(range(5), key=lambda p: (m[p], -ld[p], -p))
        if oracle.argmax_peer(m, ld, 0) != best:
            fails.append("alpha=0 argmax")
        if oracle.argmax_peer([m[0]], [ld[0]], 3) != 0:
            fails.append("P=1")
    return fails


def run_all() -> list[str]:
    return check_golden() + check_brute() + check_invariants()


if __name__ == "__main__":
    f = run_all()
    print("FAILURES", len(f))
    for x in f[:20]:
        print(x)
    raise SystemExit(1 if f else 0)
