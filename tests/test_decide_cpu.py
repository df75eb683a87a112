"""Pins of the oracle's route decision with excluded peers and a fallback target (``oracle.decide``):
hand-worked rows, agreement with the C++ oracle's route argmax when nothing is excluded, and the
invariants that excluding the best candidate promotes the next-best one and that the two differ; a negative
match entry counts as 0 (a prefix-match length is never negative)."""
import random

import numpy as np

import oracle
import workload as wl


def test_hand_worked_rows():
    # Scores with alpha = 1: 5-1, 5-0, 3-0 = 4, 5, 3.
    best, nxt = oracle.decide([[5, 5, 3]], [1, 0, 0], 1)
    assert (best[0], nxt[0]) == (1, 0)
    best, nxt = oracle.decide([[5, 5, 3]], [1, 0, 0], 1, excluded=[0, 1, 0])
    assert (best[0], nxt[0]) == (0, 2)
    best, nxt = oracle.decide([[5, 5, 3]], [1, 0, 0], 1, excluded=[1, 1, 0])
    assert (best[0], nxt[0]) == (2, -1)
    best, nxt = oracle.decide([[5, 5, 3]], [1, 0, 0], 1, excluded=[1, 1, 1])
    assert (best[0], nxt[0]) == (-1, -1)
    # Equal scores: the lower load wins (4-1 = 3-0), then the lower index.
    best, nxt = oracle.decide([[4, 3], [3, 3]], [1, 0], 1)
    assert best.tolist() == [1, 1] and nxt.tolist() == [0, 0]
    best, nxt = oracle.decide([[3, 3]], [0, 0], 0)
    assert (best[0], nxt[0]) == (0, 1)


def test_best_is_the_route_argmax_and_exclusion_promotes_the_next():
    prm = wl.preset(0)
    prm.update(P=6, n_seq=200, n_prefix=12, B=300)
    W = wl.Workload(params=prm, seed=9)
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)])
    tok, off = W.requests()
    load = W.load()
    match, peer, _ = oracle.route(trees, tok, off, load, W.alpha)
    best, nxt = oracle.decide(match, load, W.alpha)
    assert np.array_equal(best, peer)
    assert (best != nxt).all() and (nxt >= 0).all()
    rng = random.Random(4)
    for b in rng.sample(range(W.B), 40):
        ex = np.zeros(W.P, np.uint8)
        ex[best[b]] = 1
        b2, n2 = oracle.decide(match[b:b + 1], load, W.alpha, excluded=ex)
        assert b2[0] == nxt[b]
        assert n2[0] not in (best[b], nxt[b])


def test_random_rows_agree_with_the_cpp_argmax():
    """With nothing excluded, the first candidate is the C++ oracle's argmax (oracle_argmax) on random rows
    full of ties (small match values and loads)."""
    rng = np.random.default_rng(17)
    for _ in range(300):
        P = int(rng.integers(1, 40))
        row = rng.integers(0, 6, size=P).astype(np.int32)
        load = rng.integers(0, 4, size=P).astype(np.int32)
        alpha = int(rng.integers(0, 3))
        best, nxt = oracle.decide(row[None, :], load, alpha)
        assert best[0] == oracle.argmax_peer(row, load, alpha)
        assert (nxt[0] == -1) == (P == 1)


def test_negative_match_entries_count_as_zero():
    # Hand-worked: alpha = 1, loads 0 and 3.  Tree 0's entry -5 counts as 0, score 0; tree 1 scores 2 - 3 = -1.
    # Taken literally, -5 would lose to -1.
    best, nxt = oracle.decide([[-5, 2]], [0, 3], 1)
    assert (best[0], nxt[0]) == (0, 1)
    # A row of negative entries decides by load alone, like an empty tree's zeros: lower load, then index.
    best, nxt = oracle.decide([[-1, -7, -2**31]], [2, 1, 1], 3)
    assert (best[0], nxt[0]) == (1, 2)
