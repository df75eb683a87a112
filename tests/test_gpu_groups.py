"""GPU parity of batches whose requests share prefixes: the route path groups requests by their first 64
tokens, routes each group's leader (smallest index) with full walks and every follower from its leader's
matches and their exact common prefix.  Results must equal independent walks (the oracle) whatever the
grouping: these cases put the group boundaries, common-prefix lengths and leader/follower lengths at the
edges of that logic."""
import random

import numpy as np
import pytest

import paper_2606_17059_gb300 as g
from gpu_util import (assert_same_route, csr_from_lists, oracle_route, route_device, router_from_seqlists,
                      seqlist_from_lists)

pytestmark = pytest.mark.gpu

HEAD = 64  # tokens that key a group


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    g.build()


def _check(trees, reqs, load, alpha, what):
    sls = [seqlist_from_lists(t) for t in trees]
    tok, off = csr_from_lists(reqs)
    r = router_from_seqlists(sls)
    gm, gp = route_device(r, tok, off, load, alpha)
    om, op = oracle_route(sls, tok, off, load, alpha)
    assert_same_route(gm, gp, om, op, what)
    return gm


def test_group_boundaries_and_common_prefix_lengths():
    rng = random.Random(11)
    V = 1000
    A = [rng.randrange(V) for _ in range(3000)]
    B = A[:700] + [rng.randrange(V) for _ in range(900)]  # shares 700 tokens with A
    fresh = lambda n: [rng.randrange(V) for _ in range(n)]
    trees = [
        [A, B, fresh(200)],                    # both long sequences
        [A[:64], A[:65], A[:1000] + fresh(5)],  # node boundaries at 64, 65 and 1000
        [B[:650] + fresh(40), fresh(80)],       # diverges from A and B inside their shared part
        [],                                     # empty tree
        [A[:2999], A + fresh(3)],               # paths just short of, and past, A's end
    ]
    reqs = [A[:HEAD]]  # the smallest index leads A's group with a request of exactly 64 tokens
    for L in (HEAD, HEAD + 1, 100, 650, 700, 701, 999, 1000, 1001, 2999, 3000):
        reqs.append(A[:L])                        # followers that are prefixes of each other
        reqs.append(A[:L] + fresh(rng.randint(1, 50)))
        reqs.append(A[:L] + [A[L] if L < len(A) else 0] + fresh(3))
    for d in (HEAD, HEAD + 1, 300, 699, 700, 701):
        x = A[:d] + [(A[d] + 1) % V] + A[d + 1:]  # one token changed at position d
        reqs.append(x)
    reqs += [A] * 20 + [B] * 5                    # exact duplicates
    reqs += [A[:HEAD - 1], A[:HEAD - 1] + [(A[HEAD - 1] + 1) % V] + A[HEAD:200], A[:10], []]  # not grouped
    reqs += [B[:L] for L in (HEAD, 699, 700, 1600)]
    reqs += [fresh(rng.randint(0, 300)) for _ in range(30)]
    tail = reqs[1:]
    rng.shuffle(tail)
    reqs = reqs[:1] + tail
    load = [rng.randrange(8) for _ in trees]
    for alpha in (0, 1, 5):
        _check(trees, reqs, load, alpha, f"alpha {alpha}")


def test_leader_shorter_than_followers_and_long_followers():
    """Leader = first request, 64 tokens; followers run past the shared-memory window of a staged request."""
    rng = random.Random(5)
    V = 50000
    A = [rng.randrange(V) for _ in range(12000)]
    trees = [[A[:9000] + [rng.randrange(V) for _ in range(20)], A[:200]], [A], [A[:5000]]]
    reqs = [A[:HEAD]] + [A[:d] + [rng.randrange(V) for _ in range(rng.randint(0, 400))]
                         for d in [rng.randint(HEAD, 12000) for _ in range(200)]]
    reqs += [A[:4096], A[:4097], A[:8999], A[:9000], A[:9001], A]
    _check(trees, reqs, [0, 0, 0], 0, "long followers")


@pytest.mark.parametrize("seed", range(6))
def test_small_vocabulary_deep_trees_grouped(seed):
    """Vocabulary 2-3: trees branch at almost every token, and many requests share their first 64 tokens."""
    rng = random.Random(100 + seed)
    V = rng.choice([2, 3])
    stems = [[rng.randrange(V) for _ in range(rng.randint(HEAD, 400))] for _ in range(4)]
    P = rng.randint(2, 9)
    trees = []
    for _ in range(P):
        t = []
        for _ in range(rng.randint(0, 40)):
            s = rng.choice(stems)
            t.append(s[:rng.randint(0, len(s))] + [rng.randrange(V) for _ in range(rng.randint(0, 60))])
        trees.append(t)
    reqs = []
    for _ in range(500):
        s = rng.choice(stems)
        reqs.append(s[:rng.randint(0, len(s))] + [rng.randrange(V) for _ in range(rng.randint(0, 80))])
    load = [rng.randrange(4) for _ in range(P)]
    _check(trees, reqs, load, rng.choice([0, 2]), f"seed {seed}")


@pytest.mark.parametrize("P", [45, 97])
def test_followers_with_tree_counts_off_the_lane_groups(P):
    """Followers take trees 64 at a time (two per lane); P = 45 and 97 leave the last pair of 32-tree
    groups partly empty.  Many trees hold the shared stems, so followers resume at checkpoints in most of
    them."""
    rng = random.Random(P)
    V = 500
    stems = [[rng.randrange(V) for _ in range(rng.randint(HEAD, 600))] for _ in range(6)]
    trees = []
    for _ in range(P):
        t = []
        for _ in range(rng.randint(0, 30)):
            s = rng.choice(stems)
            t.append(s[:rng.randint(len(s) // 2, len(s))] + [rng.randrange(V) for _ in range(rng.randint(0, 40))])
        trees.append(t)
    reqs = []
    for _ in range(1500):
        s = rng.choice(stems)
        reqs.append(s[:rng.randint(HEAD, len(s))] + [rng.randrange(V) for _ in range(rng.randint(0, 50))])
    load = [rng.randrange(8) for _ in range(P)]
    _check(trees, reqs, load, 1, f"P={P}")


def test_route_launch_count():
    """A grouped batch of short requests is routed by four grouping kernels (hash, resolve, follower ranges,
    follower placement), a leader pass and a follower pass."""
    rng = random.Random(3)
    trees = [[[rng.randrange(10) for _ in range(100)] for _ in range(5)]]
    r = router_from_seqlists([seqlist_from_lists(t) for t in trees])
    tok, off = csr_from_lists([trees[0][0], trees[0][0][:80], [1, 2, 3]])
    n0 = r.launch_count()
    route_device(r, tok, off, [0], 0)
    assert r.launch_count() - n0 == 6
