"""Host-side logic of bench.py: the expected accept length of the synthetic
draft model, checked against exhaustive enumeration of match patterns, and
the rule that ties a committed ncu traffic record to the kernel sources."""
import itertools
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
from paper_2606_27550_gb300 import synth  # noqa: E402


def _enumerate(parent, p):
    n = len(parent)
    depth = synth.depth_of(parent)
    total = 0.0
    for bits in itertools.product([0, 1], repeat=n - 1):
        m = (1,) + bits
        prob = np.prod([p if b else 1 - p for b in bits])
        ok = [True] + [False] * (n - 1)
        for i in range(1, n):
            ok[i] = ok[parent[i]] and bool(m[i])
        total += prob * (max(depth[i] for i in range(n) if ok[i]) + 1)
    return total


@pytest.mark.parametrize("parent", [[-1], [-1, 0], [-1, 0, 0], [-1, 0, 1, 2], [-1, 0, 0, 1, 1, 2, 3],
                                    list(synth.full_tree((2, 2))), list(synth.bank_trees()[4]),
                                    list(synth.rank_product_tree((4, 3, 2, 1), 12))])
@pytest.mark.parametrize("p", [0.0, 0.3, 0.7, 1.0])
def test_expected_accept_len_matches_enumeration(parent, p):
    assert bench.expected_accept_len(parent, p) == pytest.approx(_enumerate(parent, p), rel=1e-12, abs=1e-12)


def test_expected_accept_len_limits():
    for t in synth.bank_trees():
        assert bench.expected_accept_len(t, 0.0) == 1.0
        assert bench.expected_accept_len(t, 1.0) == synth.depth_of(t).max() + 1
    # a chain: 1 + p + p^2 + ... + p^D
    assert bench.expected_accept_len(synth.chain(5), 0.5) == pytest.approx(1 + 0.5 + 0.25 + 0.125 + 0.0625)


def _profiles_tree(tmp_path, records):
    """A copy of the kernel sources and a traffic file with the given records."""
    import shutil

    src = os.path.join(bench.ROOT, "paper_2606_27550_gb300", "csrc")
    dst = tmp_path / "paper_2606_27550_gb300" / "csrc"
    shutil.copytree(src, dst)
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.txt").write_text("# kernel files hash bytes [workload]\n" + records)
    return dst


def test_traffic_record_follows_the_kernel_sources(tmp_path, monkeypatch):
    """The bench reports a kernel's DRAM traffic from a committed ncu record only
    while the record's source hash matches the sources; an edit to any of them
    turns it into null, and a record for another workload does not apply."""
    files = "attention_tc.cu,common.cuh,kernels.cuh"
    dst = _profiles_tree(tmp_path, "")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h = bench.kernel_source_hash(files)
    assert len(h) == 16
    (tmp_path / "profiles" / "traffic.txt").write_text(
        f"k1_tree_attention_tc {files} {h} 12345\n"
        f"k2_lm_head lm_head.cu,common.cuh,kernels.cuh {bench.kernel_source_hash('lm_head.cu,common.cuh,kernels.cuh')}"
        " 678 some-workload\n")
    assert bench.traffic_from_profiles("k1_tree_attention_tc") == 12345
    assert bench.traffic_from_profiles("k2_lm_head", "some-workload") == 678
    assert bench.traffic_from_profiles("k2_lm_head", "another-workload") is None
    assert bench.traffic_from_profiles("k3_accept_compact") is None
    with open(dst / "common.cuh", "a") as f:
        f.write("\n// edited\n")
    assert bench.traffic_from_profiles("k1_tree_attention_tc") is None
    assert bench.traffic_from_profiles("k2_lm_head", "some-workload") is None

