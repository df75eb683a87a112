"""The C-ABI library without a GPU: it loads, exports every entry point declared in include/p2p_router.h,
and its host-only parts (snapshot builder, snapshot validation, argument checks) behave as specified.
The builder is compared with the oracle's canonical export; the oracle is never called by the library."""
import os
import random
import re
import subprocess

import numpy as np
import pytest

import oracle
import paper_2606_17059_gb300 as g
import workload as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "p2p_router.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(p2p_[a-z_]+)\s*\(", src)))


def test_library_builds_and_exports_every_declared_symbol():
    path = g.build()
    declared = _declared_functions()
    assert len(declared) >= 15
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (p2p_\w+)", out))
    assert set(declared) <= exported, set(declared) - exported
    assert set(g.exported_symbols()) == set(declared)
    lib = g._load()
    for name in declared:
        assert hasattr(lib, name)


def _declared_parameter_counts():
    """Entry point -> number of parameters, from the prototypes in include/p2p_router.h."""
    src = open(os.path.join(ROOT, "include", "p2p_router.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    out = {}
    for name, params in re.findall(r"\b(p2p_[a-z_]+)\s*\(([^;{]*?)\)\s*;", src, flags=re.S):
        params = params.strip()
        out[name] = 0 if params in ("", "void") else len(params.split(","))
    return out


def test_binding_signatures_match_the_header():
    """The ctypes binding passes as many arguments to each entry point as its prototype declares."""
    counts = _declared_parameter_counts()
    assert set(counts) == set(_declared_functions())
    lib = g._load()
    for name, n in counts.items():
        fn = getattr(lib, name)
        assert fn.argtypes is not None and len(fn.argtypes) == n, (name, n, fn.argtypes)


def test_library_has_no_oracle_dependency():
    out = subprocess.run(["nm", "-D", g.build()], capture_output=True, text=True).stdout
    assert "otree" not in out and "oracle" not in out
    ldd = subprocess.run(["ldd", g.build()], capture_output=True, text=True).stdout
    assert "oracle" not in ldd and "libwl" not in ldd


def _seqlist_from_lists(seqs):
    pool = np.array([x for s in seqs for x in s], np.int32)
    lens = np.array([len(s) for s in seqs], np.int32)
    off = np.zeros(len(seqs), np.int64)
    if len(seqs):
        off[1:] = np.cumsum(lens.astype(np.int64))[:-1]
    return wl.SeqList(np.arange(len(seqs) + 1, dtype=np.int64), off, lens, pool)


def _snap(seqlist):
    h = g.p2p_snapshot_build(seqlist)
    try:
        return g.p2p_snapshot_view(h)
    finally:
        g.p2p_snapshot_free(h)


def _oracle_export(seqs):
    t = oracle.OTree()
    for s in seqs:
        t.insert(s)
    return t.export()


def _same(a, b):
    return all(np.array_equal(np.asarray(a[k]), np.asarray(b[k])) for k in oracle.FLAT_FIELDS)


def test_snapshot_builder_matches_oracle_tiny_random():
    rng = random.Random(3)
    for _ in range(300):
        V = rng.choice([2, 3, 4, 1000])
        seqs = [[rng.randrange(V) - (V // 2 if V > 4 else 0) for _ in range(rng.randint(0, 9))]
                for _ in range(rng.randint(0, 14))]
        snap = _snap(_seqlist_from_lists(seqs))
        assert _same(snap, _oracle_export(seqs))
        assert g.p2p_flat_tree_validate(snap) == 0


def test_snapshot_builder_segmented_shared_runs():
    # Sequences referencing the same pool run (a shared prefix) and overlapping runs.
    pool = np.array([5, 6, 7, 8, 9, 1, 2, 3, 7, 7], np.int32)
    seg_begin = np.array([0, 2, 4, 5, 7, 7], np.int64)
    seg_off = np.array([0, 5, 0, 6, 2, 0, 9], np.int64)
    seg_len = np.array([5, 2, 5, 2, 3, 3, 1], np.int32)
    sl = wl.SeqList(seg_begin, seg_off, seg_len, pool)
    seqs = sl.to_lists()
    assert seqs == [[5, 6, 7, 8, 9, 1, 2], [5, 6, 7, 8, 9, 2, 3], [7, 8, 9], [5, 6, 7, 7], []]
    assert _same(_snap(sl), _oracle_export(seqs))


@pytest.mark.parametrize("cfg", [0, 1])
def test_snapshot_builder_matches_oracle_on_workloads(cfg):
    W = wl.Workload(cfg)
    for p in range(min(W.P, 3)):
        sl = W.tree(p)
        t = oracle.OTree()
        t.insert_seqlist(sl)
        assert _same(_snap(sl), t.export())


def test_stale_replica_snapshot_matches_oracle_after_ops():
    prm = wl.preset(2)
    prm.update(P=3, n_seq=300, n_prefix=30, B=10)
    W = wl.Workload(params=prm, seed=11)
    for p in (1, 2):
        t = oracle.OTree()
        t.insert_seqlist(W.tree(p, 1))
        d = W.delta(p, p + 1)
        assert t.apply_ops(d.op, d.seqs) == 0
        assert _same(_snap(W.tree(p, 0)), t.export())


def _valid_flat():
    return _snap(_seqlist_from_lists([[1, 2, 3], [1, 2, 4], [1, 5], [7]]))


@pytest.mark.parametrize("mutate", [
    lambda d: d["label_len"].__setitem__(0, 1),            # root with a label
    lambda d: d["label_len"].__setitem__(2, 0),            # empty edge
    lambda d: d["child_idx"].__setitem__(0, 0),            # root as a child
    lambda d: d["child_idx"].__setitem__(1, d["child_idx"][0]),  # a node with two parents
    lambda d: d["child_first_tok"].__setitem__(0, 99),     # first token differs from the label
    lambda d: d["term_count"].__setitem__(len(d["term_count"]) - 1, 0),  # leaf storing nothing
    lambda d: d["term_count"].__setitem__(1, -1),          # negative multiplicity
    lambda d: d["child_begin"].__setitem__(0, 10),         # child range out of bounds
    lambda d: d["label_off"].__setitem__(1, 1000),         # label out of bounds
])
def test_validate_rejects_malformed_snapshots(mutate):
    d = {k: np.array(v, copy=True) for k, v in _valid_flat().items()}
    assert g.p2p_flat_tree_validate(d) == 0
    mutate(d)
    assert g.p2p_flat_tree_validate(d) == g.P2P_E_FORMAT
    assert g.p2p_last_error()


def test_validate_rejects_unsorted_children_and_truncation():
    d = {k: np.array(v, copy=True) for k, v in _valid_flat().items()}
    b, c = d["child_begin"][0], d["child_count"][0]
    assert c == 2
    d["child_first_tok"][b], d["child_first_tok"][b + 1] = d["child_first_tok"][b + 1], d["child_first_tok"][b]
    d["child_idx"][b], d["child_idx"][b + 1] = d["child_idx"][b + 1], d["child_idx"][b]
    assert g.p2p_flat_tree_validate(d) == g.P2P_E_FORMAT
    t = {k: np.array(v, copy=True) for k, v in _valid_flat().items()}
    t["labels"] = t["labels"][:-1]  # truncated snapshot
    assert g.p2p_flat_tree_validate(t) == g.P2P_E_FORMAT


def test_validate_rejects_single_child_chain_and_cycle():
    # root -> [1] (term 0, one child) -> [2] (term 1): not compressed.
    d = dict(label_off=[0, 0, 1], label_len=[0, 1, 1], child_begin=[0, 1, 2], child_count=[1, 1, 0],
             term_count=[0, 0, 1], child_first_tok=[1, 2], child_idx=[1, 2], labels=[1, 2])
    assert g.p2p_flat_tree_validate(d) == g.P2P_E_FORMAT
    d["term_count"][1] = 1
    assert g.p2p_flat_tree_validate(d) == 0
    # Two nodes pointing at each other, unreachable from the root.
    cyc = dict(label_off=[0, 0, 1], label_len=[0, 1, 1], child_begin=[0, 0, 1], child_count=[0, 1, 1],
               term_count=[0, 1, 1], child_first_tok=[2, 1], child_idx=[2, 1], labels=[1, 2])
    assert g.p2p_flat_tree_validate(cyc) == g.P2P_E_FORMAT


def test_snapshot_build_rejects_bad_segments():
    sl = wl.SeqList(np.array([0, 1], np.int64), np.array([3], np.int64), np.array([4], np.int32),
                    np.zeros(5, np.int32))
    with pytest.raises(g.P2PError) as e:
        g.p2p_snapshot_build(sl)
    assert e.value.code == g.P2P_E_INVAL
    sl = wl.SeqList(np.array([0, 2, 1], np.int64), np.array([0, 0], np.int64), np.array([1, 1], np.int32),
                    np.zeros(5, np.int32))
    with pytest.raises(g.P2PError):
        g.p2p_snapshot_build(sl)


def test_router_create_rejects_bad_P_without_touching_the_gpu():
    for P in (0, -3, 65537):
        with pytest.raises(g.P2PError) as e:
            g.p2p_router_create(P)
        assert e.value.code == g.P2P_E_INVAL
