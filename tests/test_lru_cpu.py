"""Pins of the LRU eviction oracle (``oracle.lru``): a hand-worked example, and agreement on random operation
sequences with an independent brute force that keeps the cache as a prefix-closed set of token paths with
last-access times and a multiset of stored sequences."""
import random

import pytest

from oracle.lru import LRUTrie, hit_rate


class _Brute:
    """The cache as plain sets: every cached token path (all prefixes of stored sequences) -> last access."""

    def __init__(self):
        self.last: dict[tuple, int] = {}
        self.seqs: dict[tuple, int] = {}

    def insert(self, seq, t):
        seq = tuple(seq)
        for i in range(1, len(seq) + 1):
            self.last[seq[:i]] = t
        self.seqs[seq] = self.seqs.get(seq, 0) + 1

    def match(self, req):
        m = 0
        while m < len(req) and tuple(req[:m + 1]) in self.last:
            m += 1
        return m

    def access(self, req, t):
        m = self.match(req)
        for i in range(1, m + 1):
            self.last[tuple(req[:i])] = t
        return m

    def evict(self):
        leaves = [p for p in self.last if not any(len(q) == len(p) + 1 and q[:len(p)] == p for q in self.last)]
        if not leaves:
            return None
        p = min(leaves, key=lambda q: (self.last[q], q))
        del self.last[p]
        if p in self.seqs:
            c = self.seqs.pop(p)
            self.seqs[p[:-1]] = self.seqs.get(p[:-1], 0) + c
        return p[-1]


def test_hand_worked_eviction_order():
    t = LRUTrie()
    t.insert([1, 2, 3], 1)
    t.insert([1, 2, 4], 2)
    t.insert([5], 3)
    assert t.n_tokens == 5
    # Leaves: ...3 (last 1), ...4 (last 2), 5 (last 3).  [1, 2, 3] loses its last token and now ends at [1, 2].
    assert t.evict() == 3
    assert t.sequences() == {(1, 2): 1, (1, 2, 4): 1, (5,): 1}
    assert t.evict() == 4
    assert t.sequences() == {(1, 2): 2, (5,): 1}
    # Serving [1, 2, 9] at time 4 touches [1] and [1, 2]: now [5] is the oldest leaf.
    assert t.access([1, 2, 9], 4) == 2
    assert t.evict() == 5
    assert t.sequences() == {(1, 2): 2, (): 1}
    assert t.evict() == 2 and t.evict() == 1 and t.evict() is None
    assert t.n_tokens == 0 and t.sequences() == {(): 3}
    assert hit_rate(2, 3) == pytest.approx(2 / 3) and hit_rate(0, 0) == 0.0


@pytest.mark.parametrize("seed", range(6))
def test_random_operations_agree_with_the_brute_force(seed):
    rng = random.Random(seed)
    V = rng.choice([2, 3, 5])
    t, b = LRUTrie(), _Brute()
    for time in range(1, 400):
        k = rng.random()
        if k < 0.45:
            s = [rng.randrange(V) for _ in range(rng.randint(0, 8))]
            t.insert(s, time)
            b.insert(s, time)
        elif k < 0.75:
            r = [rng.randrange(V) for _ in range(rng.randint(0, 8))]
            assert t.access(r, time) == b.access(r, time)
        else:
            assert t.evict() == b.evict()
        if time % 25 == 0:
            assert t.sequences() == {s: c for s, c in b.seqs.items() if c}
            assert t.n_tokens == len(b.last)
            for _ in range(5):
                r = [rng.randrange(V) for _ in range(rng.randint(0, 8))]
                assert t.match(r) == b.match(r)
