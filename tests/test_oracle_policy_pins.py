"""Pins for the oracle's per-step tree selection (Sec. 4): the path-value
score against its closed forms, the policies against hand traces and numpy's
searchsorted."""
import numpy as np
import pytest

import oracle
from paper_2606_27550_gb300 import synth


def test_path_value_closed_forms():
    # probabilities <= 1: every g_d <= p0, so s = p0 (the formula as printed)
    g = synth.rng(5)
    for _ in range(200):
        p0 = float(g.random())
        heads = g.random(int(g.integers(0, 6)))
        assert oracle.path_value(p0, heads) == p0
    assert oracle.path_value(0.5, []) == 0.5
    # the cumulative product itself, with factors above 1
    assert oracle.path_value(0.5, [2.0, 0.25]) == 1.0           # g1 = 1.0, g2 = 0.25
    assert oracle.path_value(0.25, [2.0, 3.0, 0.1]) == 1.5      # g = 0.5, 1.5, 0.15
    assert oracle.path_value(0.0, [5.0]) == 0.0


def test_ladder_hand_trace():
    feats = [3.0, 1.0, 1.0, 1.0, 2.0, 2.0, 1.4, 2.6, 2.6, 2.6, 2.6, 0.0]
    rungs, r = [], 0
    for f in feats:
        r = oracle.policy_next("ladder", r, 4, f, 1.5, 2.5)
        rungs.append(r)
    # up below 1.5, down above 2.5, dead band in between, clamped to [0, 3]
    assert rungs == [0, 1, 2, 3, 3, 3, 3, 2, 1, 0, 0, 1]


def test_binary_hysteresis_hand_trace():
    feats = [0.1, 0.8, 0.7, 0.6, 0.5, 0.4, 0.9, 0.45]
    rungs, r = [], 0
    for f in feats:
        r = oracle.policy_next("binary", r, 2, f, 0.7, 0.5)
        rungs.append(r)
    assert rungs == [0, 1, 1, 1, 0, 0, 1, 0]
    # tau_on == tau_off: a single threshold
    assert oracle.policy_next("binary", 0, 2, 0.7, 0.7, 0.7) == 0
    assert oracle.policy_next("binary", 1, 2, 0.70001, 0.7, 0.7) == 1


def test_threshold_ladder_matches_searchsorted():
    g = synth.rng(6)
    for _ in range(300):
        k = int(g.integers(1, 9))
        edges = np.sort(g.random(k - 1))
        f = float(g.random())
        want = int(np.searchsorted(edges, f, side="right"))
        assert oracle.policy_next("threshold", int(g.integers(0, k)), k, f, edges=edges) == want
