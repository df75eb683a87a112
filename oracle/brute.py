"""Brute-force definitions in pure Python, for tiny inputs.

TEST INFRASTRUCTURE (see the package docstring).  These restate what the router computes with no tree
at all, so that they pin the C++ oracle:

* PrefixMatch(r, T) of Algorithm 1, read as the longest prefix of r shared with any cached sequence:
  ``max over s in S(T) of LCP(r, s)``, 0 when S(T) is empty.
* getBestNode / the argmax of Algorithm 1 with the load term: the peer maximising the tuple
  ``(match - alpha*load, -load, -peer)``.
* The canonical snapshot of a multiset, built from the set of all prefixes of stored sequences
  (the uncompressed trie) by keeping only the branching or terminal positions.
"""
from __future__ import annotations

from collections import Counter


def lcp(a, b) -> int:
    n = 0
    for x, y in zip(a, b):
        if x != y:
            break
        n += 1
    return n


def match(req, stored) -> int:
    """Longest common prefix of req with any sequence of the multiset ``stored``."""
    best = 0
    for s in stored:
        best = max(best, lcp(req, s))
    return best


def route_one(match_row, load, alpha: int) -> int:
    keys = [(m - alpha * l, -l, -p) for p, (m, l) in enumerate(zip(match_row, load))]
    return max(range(len(keys)), key=lambda p: keys[p])


def route(requests, trees, load, alpha: int):
    """(match rows, peers) for lists of requests and of stored multisets."""
    rows = [[match(r, t) for t in trees] for r in requests]
    return rows, [route_one(row, load, alpha) for row in rows]


def canonical_snapshot(stored) -> dict:
    """Canonical flat tree of a multiset of sequences, from first principles.

    The trie positions are the distinct prefixes of stored sequences.  A position is kept as a node when it
    is the root, ends a stored sequence, or has at least two distinct continuations; the edge to a kept node
    carries the tokens since its nearest kept ancestor.  Nodes are numbered in preorder with children in
    ascending order of their first token; labels and child lists are packed in node order.
    """
    stored = [tuple(s) for s in stored]
    mult = Counter(stored)
    prefixes = {()}
    for s in stored:
        for i in range(1, len(s) + 1):
            prefixes.add(s[:i])
    cont = {}
    for q in prefixes:
        if q:
            cont.setdefault(q[:-1], set()).add(q[-1])

    def kept(q):
        return q == () or mult.get(q, 0) > 0 or len(cont.get(q, ())) >= 2

    def kept_children(q):
        # Follow each continuation down to the next kept position.
        out = []
        for t in sorted(cont.get(q, ())):
            x = q + (t,)
            while not kept(x):
                (nxt,) = cont[x]
                x = x + (nxt,)
            out.append(x)
        return out

    order = []
    stack = [()]
    while stack:
        q = stack.pop()
        order.append(q)
        stack.extend(reversed(kept_children(q)))
    idx = {q: i for i, q in enumerate(order)}
    parent_len = {(): 0}
    for q in order:
        for c in kept_children(q):
            parent_len[c] = len(q)
    d = {k: [] for k in ("label_off", "label_len", "child_begin", "child_count", "term_count",
                         "child_first_tok", "child_idx", "labels")}
    for q in order:
        lab = list(q[parent_len[q]:])
        d["label_off"].append(len(d["labels"]))
        d["label_len"].append(len(lab))
        d["labels"].extend(lab)
        kids = kept_children(q)
        d["child_begin"].append(len(d["child_idx"]))
        d["child_count"].append(len(kids))
        d["term_count"].append(mult.get(q, 0))
        for c in kids:
            d["child_first_tok"].append(c[len(q)])
            d["child_idx"].append(idx[c])
    return d
