"""Pins of the CPU oracle (no GPU): golden hand-worked values, brute force on tiny inputs, invariants,
property tests, a mutation test showing that the pins catch planted mistakes, and a brute-force check of
sampled outputs at a real workload size."""
import os
import subprocess
import sys
import tempfile
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
import oracle.brute as brute
import workload as wl

from oracle_pins import check_brute, check_golden, check_invariants

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


def test_golden_worked_example():
    assert check_golden() == []


def test_brute_force_tiny_inputs():
    assert check_brute(seed=0, trials=200) == []


def test_invariants():
    assert check_invariants(seed=1, trials=80) == []


def test_brute_canonical_snapshot_itself():
    # The brute-force snapshot builder against the hand-worked snapshots.
    import json
    g = json.load(open(os.path.join(HERE, "golden", "worked_example.json")))
    for seqs, snap in zip(g["trees"], g["snapshots"]):
        assert brute.canonical_snapshot(seqs) == snap


def test_duplicates_are_a_multiset():
    t = oracle.OTree()
    for _ in range(3):
        t.insert([5, 6, 7])
    t.insert([5, 6])
    assert t.stats() == (3, 3, 4)
    assert t.remove([5, 6, 7]) and t.remove([5, 6, 7])
    assert t.match([5, 6, 7, 8]) == 3
    assert t.remove([5, 6, 7])
    assert t.match([5, 6, 7, 8]) == 2
    assert not t.remove([5, 6, 7])
    assert t.remove([5, 6])
    assert t.stats() == (1, 0, 0)


def test_empty_sequence_and_root_terminal():
    t = oracle.OTree()
    t.insert([])
    assert t.stats() == (1, 0, 1)
    assert t.match([1, 2]) == 0 and t.match([]) == 0
    assert t.remove([]) and not t.remove([])


def test_negative_and_large_tokens():
    t = oracle.OTree()
    seqs = [[-5, 2**31 - 1, 0], [-5, -6], [2**31 - 1]]
    for s in seqs:
        t.insert(s)
    for r in ([-5, 2**31 - 1, 0, 1], [-5, -6, 7], [2**31 - 1, 3], [-(2**31)]):
        assert t.match(r) == brute.match(r, seqs)
    assert t.export()["child_first_tok"][:2].tolist() == [-5, 2**31 - 1]


def test_route_thread_count_independent():
    W = wl.Workload(0)
    trees = oracle.build_trees([W.tree(p) for p in range(W.P)])
    tok, off = W.requests(0, 600)
    ld = W.load()
    a = oracle.route(trees, tok, off, ld, W.alpha, n_threads=1)
    b = oracle.route(trees, tok, off, ld, W.alpha, n_threads=7)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    m, peer, ctr = a
    assert ctr[3] == len(tok)
    assert ctr[0] >= m.sum()  # every matched token was compared
    assert ctr[0] <= m.sum() + m.size  # at most one extra (mismatching) token per lookup
    assert ctr[1] >= m.size  # the root at least


def _lcp_np(r: np.ndarray, s: np.ndarray) -> int:
    n = min(len(r), len(s))
    neq = np.nonzero(r[:n] != s[:n])[0]
    return int(neq[0]) if len(neq) else n


@pytest.mark.parametrize("cfg", [0, 1])
def test_sampled_outputs_against_definition_real_size(cfg):
    """At the real tree sizes of workloads 0 and 1: sampled match values equal the definition
    max_s LCP(r, s) over the stored sequences, computed sequence by sequence."""
    W = wl.Workload(cfg)
    P = min(W.P, 4)
    lists = [W.tree(p) for p in range(P)]
    trees = oracle.build_trees(lists)
    tok, off = W.requests(0, 40)
    m, _, _ = oracle.route(trees, tok, off, W.load()[:P], W.alpha)
    csr = [sl.to_csr() for sl in lists]
    for b in range(0, 40, 3):
        r = tok[off[b]:off[b + 1]]
        for p in range(P):
            t, o = csr[p]
            best = 0
            for i in range(len(o) - 1):
                if t[o[i]] == r[0]:  # sequences with another first token share nothing with r
                    best = max(best, _lcp_np(r, t[o[i]:o[i + 1]]))
            assert m[b, p] == best, (b, p)


def test_hypothesis_properties():
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    seq = st.lists(st.integers(0, 2), max_size=8)

    @hyp.settings(max_examples=150, deadline=None)
    @hyp.given(st.lists(seq, max_size=10), seq, st.lists(seq, max_size=5))
    def prop(stored, req, more):
        t = oracle.OTree()
        for s in stored:
            t.insert(s)
        assert t.match(req) == brute.match(req, stored)
        before = t.match(req)
        for s in more:
            t.insert(s)
        assert t.match(req) >= before
        assert t.match(req) == brute.match(req, stored + more)
        snap = brute.canonical_snapshot(stored + more)
        e = t.export()
        assert all(e[k].tolist() == snap[k] for k in snap)

    prop()


# Plausible mistakes planted in a copy of the oracle source; each must make at least one pin fail.
MUTANTS = [
    ("drop the mismatching-token count", "if (k < L && i + k < n) compared += 1;", ";"),
    ("keep walking after a partial edge", "    if (k < L) break;\n    cur = c;", "    cur = c;"),
    ("tie to the higher load", "(load[p] < load[best] ||", "(load[p] > load[best] ||"),
    ("ties to the higher index", "if (sp > sb ||", "if (sp >= sb ||"),
    ("wrong sign of the load term", "(int64_t)m[p] - (int64_t)alpha * load[p]", "(int64_t)m[p] + (int64_t)alpha * load[p]"),
    ("split node loses its terminal", "      mid->term = 1;\n      return;", "      return;"),
    ("no merge after delete", "merge_with_only_child(cur);", ";"),
    ("off-by-one child-search bytes", "while (((int64_t)1 << b) < deg + 1) ++b;", "while (((int64_t)1 << b) <= deg + 1) ++b;"),
    ("root not counted as visited", "compared = 0, visited = 1, search = 0;", "compared = 0, visited = 0, search = 0;"),
    ("request end ignored inside an edge", "while (k < L && i + k < n && c->label[(size_t)k] == r[i + k]) ++k;",
     "while (k < L && c->label[(size_t)k] == r[i + k]) ++k;"),
    ("leaf keeps the first token twice", "leaf->label.assign(s + i, s + n);\n      leaf->term = 1;\n      cur->kids",
     "leaf->label.assign(s + i, s + n);\n      leaf->label.push_back(s[i]);\n      leaf->term = 1;\n      cur->kids"),
    ("children not kept sorted", "cur->kids.insert(it, leaf);", "cur->kids.push_back(leaf);"),
]


def test_mutants_are_caught():
    src = open(os.path.join(ROOT, "oracle", "oracle_tree.cpp")).read()
    tmp = tempfile.mkdtemp(prefix="oracle_mut_")

    def run(idx):
        name, old, new = MUTANTS[idx]
        assert src.count(old) == 1, f"mutant anchor not unique: {name}"
        path = os.path.join(tmp, f"m{idx}.cpp")
        so = os.path.join(tmp, f"m{idx}.so")
        open(path, "w").write(src.replace(old, new))
        subprocess.check_call(["g++", "-O1", "-std=c++17", "-fPIC", "-shared", "-pthread", "-o", so, path])
        env = dict(os.environ, ORACLE_SO=so, PYTHONPATH=ROOT + os.pathsep + HERE)
        r = subprocess.run([sys.executable, os.path.join(HERE, "oracle_pins.py")], env=env,
                           capture_output=True, text=True, timeout=300)
        return name, r.returncode

    with ThreadPoolExecutor(max_workers=6) as ex:
        results = list(ex.map(run, range(len(MUTANTS))))
    survivors = [name for name, rc in results if rc == 0]
    assert survivors == [], f"mutants not caught by the pins: {survivors}"
