"""The C-ABI library without a GPU: it builds, loads, exports every entry point
that include/treeverify.h declares, and its pure-host topology code works."""
import ctypes
import os
import re
import subprocess

import networkx as nx
import numpy as np
import pytest

import paper_2606_27550_gb300 as tv
from paper_2606_27550_gb300 import build as tvbuild
from paper_2606_27550_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    tvbuild.build()
    return tv.load()


def _declared():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", h)).read()
            names |= set(re.findall(r"TB_API\s+[\w\s\*]+?\b(\w+)\s*\(", txt))
    return names


def test_every_declared_symbol_is_exported(lib):
    declared = _declared()
    assert {"verify_step", "tree_attention", "lm_head_stats", "greedy_accept", "kv_compact", "tb_create",
            "tb_add_topology", "tb_destroy", "tb_last_error"} <= declared
    out = subprocess.run(["nm", "-D", "--defined-only", tv.LIB_PATH], capture_output=True, text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
    assert declared <= exported, declared - exported
    assert set(tv.API) == declared
    for name in declared:
        assert hasattr(lib, name)


def test_only_the_c_abi_is_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", tv.LIB_PATH], capture_output=True, text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
    assert exported == _declared()


def test_canonicalize_bfs_order_and_bitsets(lib):
    g = synth.rng(0)
    for trial in range(20):
        n = int(g.integers(1, 65))
        parent = synth.random_tree(g, n)
        perm = np.concatenate([[0], 1 + g.permutation(n - 1)])  # relabel non-root nodes
        inv = np.argsort(perm)
        shuffled = np.array([-1 if perm[i] == 0 else inv[parent[perm[i]]] for i in range(n)], np.int32)
        order, bp, depth, anc = tv.tb_canonicalize(shuffled)
        assert sorted(order.tolist()) == list(range(n)) and order[0] == 0
        # canonical parents are the relabelled original parents, parent < child, depth non-decreasing
        for c in range(1, n):
            assert bp[c] < c and order[bp[c]] == shuffled[order[c]]
        assert np.all(np.diff(depth) >= 0)
        gr = nx.DiGraph([(int(bp[c]), c) for c in range(1, n)])
        gr.add_nodes_from(range(n))
        for c in range(n):
            want = sum(1 << a for a in nx.ancestors(gr, c) | {c})
            assert int(anc[c]) == want
            assert depth[c] == nx.shortest_path_length(gr, 0, c)
        # breadth-first: children of each node appear in increasing original index
        for p in range(n):
            kids = [c for c in range(1, n) if bp[c] == p]
            assert [order[c] for c in kids] == sorted(order[c] for c in kids)


def test_canonicalize_keeps_bfs_input(lib):
    for parent in synth.bank_trees() + [synth.shape_c2().parent, synth.chain(64)]:
        order, bp, _, _ = tv.tb_canonicalize(parent)
        assert np.array_equal(order, np.arange(len(parent)))
        assert np.array_equal(bp, parent)


@pytest.mark.parametrize("parent,why", [
    ([], "empty"), ([0], "root parent"), ([-1, 1], "self loop"), ([-1, 2, 1], "cycle"),
    ([-1, 5], "out of range"), ([1, -1], "root not first"), (list(range(-1, 64)), "65 nodes")])
def test_canonicalize_rejects(lib, parent, why):
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tb_canonicalize(np.array(parent, dtype=np.int32))
    assert e.value.status == tv.TB_EINVAL, why


def test_no_device_calls_fail_cleanly(lib):
    import torch

    if torch.cuda.is_available():
        pytest.skip("has a GPU")
    h = ctypes.c_void_p()
    assert lib.tb_create(ctypes.byref(h), 4, 0) != tv.TB_OK
    assert lib.tb_last_error()
    assert lib.tb_workspace_size(64, 32, 32, 32, 128, 32000, 0) == 0


def test_launch_count_is_host_only(lib):
    """tb_launch_count reads a host counter: callable without a device, and
    TB_EINVAL for a NULL pointer."""
    n = ctypes.c_uint64(12345)
    assert lib.tb_launch_count(ctypes.byref(n)) == tv.TB_OK
    before = n.value
    assert lib.tb_launch_count(ctypes.byref(n)) == tv.TB_OK
    assert n.value == before  # nothing launched in between
    assert lib.tb_launch_count(None) == tv.TB_EINVAL
    assert tv.tb_launch_count() == before
