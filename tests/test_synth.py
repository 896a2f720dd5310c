"""Input generators: tree shapes of the synthetic workloads and bf16 rounding."""
import numpy as np

from paper_2606_27550_gb300 import synth


def _widths(parent):
    d = synth.depth_of(parent)
    return np.bincount(d).tolist()


def test_tiny_tree_is_binary_depth2():
    assert _widths(synth.shape_c1().parent) == [1, 2, 4]


def test_26_node_tree_from_branching_4321():
    # hand count: rank sums 0 and 1 give 14 nodes; the first 12 of rank sum 2
    # in (depth, lex) order complete the 26 -> widths 1,3,6,9,7 (depth 4)
    assert _widths(synth.shape_c2().parent) == [1, 3, 6, 9, 7]


def test_64_node_tree_depth5_and_bank_nesting():
    p = synth.shape_c4().parent
    assert len(p) == 64 and max(synth.depth_of(p)) == 5
    bank = synth.bank_trees()
    assert [len(t) for t in bank] == list(synth.BANK_SIZES)
    assert [int(max(synth.depth_of(t))) for t in bank] == [0, 1, 3, 5, 5, 5, 5, 5]
    # every bank tree is a breadth-first tree with parent[i] < i
    for t in bank:
        assert t[0] == -1 and all(0 <= t[i] < i for i in range(1, len(t)))
        assert all(t[i] <= t[i + 1] for i in range(1, len(t) - 1))


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, -2.5, 1e-3], dtype=np.float32)
    b = synth.to_bf16_bits(x)
    assert b.tolist()[:4] == [0x3F80, 0x3F80, 0x3F82, 0xC020]
    import torch
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(b, ref)


def test_drafts_follow_match_probability():
    parent = synth.shape_c4().parent
    argmax = np.arange(64, dtype=np.int32) + 7
    hits = 0
    for s in range(200):
        d = synth.gen_drafts(s, parent, argmax, 32000, 0.5)
        hits += int(np.sum(d[1:] == argmax[parent[1:]]))
        assert np.all((d >= 0) & (d < 32000))
    assert abs(hits / (200 * 63) - 0.5) < 0.03
