"""LRU eviction of a node's own prefix trie (TEST INFRASTRUCTURE: see oracle/__init__.py for who may use it).

Algorithm 1 evicts, while a request needs more memory than the GPU has free, one least-recently-used leaf
token at a time (EvictLRUTrie in the Section 2 primitive list), together with its KV cache entry.  Section 5
(cache-hit analysis) reports a request's expected cache hit rate, the routing node's prediction at decision
time: the matched share of its tokens.

This module is the plain definition, over an uncompressed trie of tokens:
- the trie holds a multiset of token sequences; every token node records the time of its last access;
- an access (a request served from the cache: PrefixMatch) and an insert (UpdateTrie) both touch every token
  node on the request's path, the matched part for an access and the whole sequence for an insert;
- ``evict`` removes the leaf token whose last access is the oldest, ties to the lexicographically smallest
  token path, and returns that token.  The stored sequences that ended at it now end one token earlier (their
  cached prefix lost its last token).
Readings taken where Section 2 is silent: what counts as an access, the tie rule, and what happens to the
sequences ending at an evicted token.
"""
from __future__ import annotations


class _Node:
    __slots__ = ("children", "count", "last")

    def __init__(self, last: int):
        self.children: dict[int, _Node] = {}
        self.count = 0  # stored sequences that end at this node
        self.last = last


class LRUTrie:
    """A node's own cache trie with LRU token eviction (plain per-token definition)."""

    def __init__(self):
        self.root = _Node(0)
        self.n_tokens = 0

    def insert(self, seq, t: int) -> None:
        """UpdateTrie at time t: store one more occurrence of seq; every token on its path is touched."""
        node = self.root
        for tok in seq:
            tok = int(tok)
            nxt = node.children.get(tok)
            if nxt is None:
                nxt = node.children[tok] = _Node(t)
                self.n_tokens += 1
            nxt.last = t
            node = nxt
        node.count += 1

    def match(self, req) -> int:
        """PrefixMatch: the number of leading tokens of req found along one path."""
        node, m = self.root, 0
        for tok in req:
            node = node.children.get(int(tok))
            if node is None:
                break
            m += 1
        return m

    def access(self, req, t: int) -> int:
        """A request served from the cache at time t: its matched tokens are touched; returns the match."""
        node, m = self.root, 0
        for tok in req:
            node = node.children.get(int(tok))
            if node is None:
                break
            node.last = t
            m += 1
        return m

    def evict(self):
        """EvictLRUTrie: removes the least-recently-used leaf token (ties to the smallest token path) and
        returns it, or None if the trie is empty."""
        best = None  # (last, path, parent, token)
        stack = [(self.root, ())]
        while stack:
            node, path = stack.pop()
            for tok, ch in node.children.items():
                p = path + (tok,)
                if ch.children:
                    stack.append((ch, p))
                elif best is None or (ch.last, p) < (best[0], best[1]):
                    best = (ch.last, p, node, tok)
        if best is None:
            return None
        _, _, parent, tok = best
        leaf = parent.children.pop(tok)
        parent.count += leaf.count  # sequences that ended at the evicted token now end at its parent
        self.n_tokens -= 1
        return tok

    def sequences(self) -> dict[tuple, int]:
        """The stored multiset: sequence -> occurrences."""
        out: dict[tuple, int] = {}
        stack = [(self.root, ())]
        while stack:
            node, path = stack.pop()
            if node.count:
                out[path] = node.count
            for tok, ch in node.children.items():
                stack.append((ch, path + (tok,)))
        return out


def hit_rate(match: int, length: int) -> float:
    """The expected share of a request's prefill served from the cache: matched tokens over its length (0
    for an empty request)."""
    return match / length if length else 0.0
