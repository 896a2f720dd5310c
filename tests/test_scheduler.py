"""Per-step tree selection (host, C ABI): the hysteretic step ladder over the
bank, the paper's binary hysteretic rule on s and threshold_ladder (Sec. 4)."""
import numpy as np
import pytest

import paper_2606_27550_gb300 as tv
from paper_2606_27550_gb300 import build as tvbuild
from paper_2606_27550_gb300 import synth


@pytest.fixture(scope="module", autouse=True)
def lib():
    tvbuild.build()
    return tv.load()


def test_ladder_moves_one_step_with_dead_band():
    f = tv.tb_schedule_hysteretic_ladder
    assert f(0, 8, 1.0, 1.5, 2.5) == 1          # predictable: bigger tree
    assert f(7, 8, 1.0, 1.5, 2.5) == 7          # clamped at the largest
    assert f(3, 8, 3.0, 1.5, 2.5) == 2          # unpredictable: smaller tree
    assert f(0, 8, 3.0, 1.5, 2.5) == 0          # clamped at the smallest
    for h in (1.5, 2.0, 2.5):                   # dead band [1.5, 2.5]: stay
        assert f(4, 8, h, 1.5, 2.5) == 4
    assert f(9, 8, 2.0, 1.5, 2.5) == 7 and f(-2, 8, 2.0, 1.5, 2.5) == 0


def test_ladder_trace_matches_rule_written_out():
    trace = synth.ar1_entropy_trace(0, 1000, hmax=np.log(32000))
    k, ks = 0, []
    for h in trace:
        k = tv.tb_schedule_hysteretic_ladder(k, 8, float(h), 1.5, 2.5)
        ks.append(k)
    # the rule, step by step
    k2, ks2 = 0, []
    for h in trace:
        if h < 1.5:
            k2 = min(k2 + 1, 7)
        elif h > 2.5:
            k2 = max(k2 - 1, 0)
        ks2.append(k2)
    assert ks == ks2
    assert len(set(ks)) >= 4  # the trace exercises the bank


def test_binary_rule_hysteresis():
    f = tv.tb_schedule_binary
    assert f(0, 0.05, 0.02, 0.01) == 1   # s > tau_on: aggressive
    assert f(1, 0.015, 0.02, 0.01) == 1  # between the thresholds: keep
    assert f(0, 0.015, 0.02, 0.01) == 0
    assert f(1, 0.01, 0.02, 0.01) == 0   # s <= tau_off: conservative
    assert f(1, 0.02, 0.02, 0.02) == 0 and f(0, 0.0201, 0.02, 0.02) == 1  # single threshold


def test_threshold_ladder_bins():
    edges = [0.001, 0.005, 0.01, 0.02, 0.05]
    f = tv.tb_schedule_threshold_ladder
    assert [f(s, edges) for s in (0.0, 0.001, 0.003, 0.0099, 0.01, 0.03, 0.05, 0.9)] == [0, 1, 1, 2, 3, 4, 5, 5]
