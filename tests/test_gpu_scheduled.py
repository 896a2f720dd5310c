"""GPU parity of the device-driven decode loop (verify_step_scheduled): the
tree and the prefix length of every step come from device memory, and the
acceptance kernel's last CTA takes the per-step policy decision (Sec. 4).

Every step is checked against the fp64 oracle: attention of the tree the
device chose at the prefix length it holds, the greedy statistics, acceptance,
the whole compacted cache, and the next state (rung from the oracle's policy
on the step's feature, L + accept_len, step + 1).  A CUDA-graph replay of a
run of steps must reproduce the eager run byte for byte.
"""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, gap_filtered_hidden, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

LAYERS, HQ, HKV, D_HEAD, D_MODEL, V = 2, 4, 2, 128, 256, 1000
TREES = synth.bank_trees()
N_MAX = max(len(t) for t in TREES)


@pytest.fixture(scope="module")
def dev():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda:0")


class Loop:
    """Seeded inputs of a scheduled run: per step, queries and hidden rows for
    N_MAX nodes and one draft row per rung (drafts copy the parent's oracle
    greedy token with probability p_match)."""

    def __init__(self, dev, steps, L0, seed=0, p_match=0.7, rungs=tuple(range(len(TREES))), d_head=D_HEAD):
        self.dev, self.steps, self.L0 = dev, steps, L0
        self.trees = [TREES[i] for i in rungs]  # the tree of each rung; draft rows follow the rungs
        self.L_cap = L0 + steps * 7 + N_MAX + 8
        self.bank = tv.Bank(16, 0)
        self.ids = [self.bank.add(t)[0] for t in self.trees]
        # every slot holds finite random K/V (the tree slots of each step are read where L lands)
        self.k, self.v = synth.gen_kv(seed, LAYERS, HKV, self.L_cap, d_head, self.L_cap)
        self.W = synth.gen_lm_head(seed, V, D_MODEL)
        self.q = [synth.gen_q(seed + 10 + t, LAYERS, N_MAX, HQ, d_head) for t in range(steps)]
        self.h, self.am, self.t1, self.en = [], [], [], []
        self.drafts = []
        for t in range(steps):
            h, am, t1, en = gap_filtered_hidden(seed + 100 + t, N_MAX, self.W)
            self.h.append(h)
            self.am.append(am)
            self.t1.append(t1)
            self.en.append(en)
            rows = np.zeros((len(self.trees), N_MAX), np.int32)
            for r, tr in enumerate(self.trees):
                rows[r, :len(tr)] = synth.gen_drafts(seed + 1000 * t + r, tr, am[:len(tr)], V, p_match)
            self.drafts.append(rows)
        self.kd, self.vd = to_dev(self.k, dev), to_dev(self.v, dev)
        self.Wd = to_dev(self.W, dev)
        self.qd = [to_dev(x, dev) for x in self.q]
        self.hd = [to_dev(x, dev) for x in self.h]
        self.dd = [to_dev(x, dev) for x in self.drafts]
        self.out = torch.empty((LAYERS, N_MAX, HQ, d_head), dtype=torch.bfloat16, device=dev)
        self.g_am = torch.empty(N_MAX, dtype=torch.int32, device=dev)
        self.g_t1 = torch.empty(N_MAX, dtype=torch.float32, device=dev)
        self.g_en = torch.empty(N_MAX, dtype=torch.float32, device=dev)
        self.res = tv.make_result(dev)
        self.ws = tv.make_workspace(tv.tb_workspace_size(N_MAX, LAYERS, HKV, HQ, d_head, V, 0), dev)

    def kv(self):
        return tv.KvCache(self.kd, self.vd, 0)

    def step(self, t, policy, state, flags=0, stream=None):
        tv.verify_step_scheduled(self.bank, policy, state, self.kv(), self.qd[t], self.hd[t], self.Wd, self.dd[t],
                                 self.out, self.g_am, self.g_t1, self.g_en, self.res, self.ws, flags, stream)


def _trace(steps, seed=3):
    # feature trace on a float32 grid so host and device compare the same numbers
    g = synth.rng(seed, 1)
    return np.round(g.uniform(0.5, 3.5, steps) * 64).astype(np.float32) / np.float32(64)


def _run_loop(dev, steps, L0, d_head, trace, seed=0):
    """The loop against the oracle, step by step; returns the rungs visited."""
    lp = Loop(dev, steps, L0=L0, seed=seed, d_head=d_head)
    tr_d = to_dev(trace, dev)
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, lp.ids, a=1.5, b=2.5, trace=tr_d,
                         node_stride=N_MAX)
    state = tv.make_state(3, lp.L0, dev)
    k_ref, v_ref = lp.k.copy(), lp.v.copy()
    rung, L = 3, lp.L0
    seen = set()
    for t in range(steps):
        lp.step(t, pol, state)
        torch.cuda.synchronize()
        tree = TREES[rung]
        n = len(tree)
        seen.add(rung)
        # attention of the device-chosen tree at the device-held prefix length
        got = lp.out.float().cpu().numpy()
        for layer in range(LAYERS):
            ref = oracle.tree_attention(lp.q[t][layer][:n], k_ref[layer], v_ref[layer], L, tree)
            check_attention(got[layer][:n], ref, f"step {t} layer {layer}")
        assert np.array_equal(lp.g_am.cpu().numpy()[:n], lp.am[t][:n])
        assert np.abs(lp.g_t1.cpu().numpy()[:n] - lp.t1[t][:n]).max() <= STAT_TOL
        assert np.abs(lp.g_en.cpu().numpy()[:n] - lp.en[t][:n]).max() <= STAT_TOL
        ka, path, bonus = oracle.accept(tree, lp.drafts[t][rung][:n], lp.am[t][:n])
        r = tv.parse_result(lp.res)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        k_ref = oracle.kv_compact(k_ref, L, path)
        v_ref = oracle.kv_compact(v_ref, L, path)
        assert np.array_equal(bits(lp.kd), k_ref) and np.array_equal(bits(lp.vd), v_ref), f"step {t}"
        nxt = oracle.policy_next("ladder", rung, len(TREES), float(trace[t]), 1.5, 2.5)
        st = tv.parse_state(state)
        assert st == {"rung": nxt, "L": L + ka, "step": t + 1, "feature": float(trace[t]), "accept_len": ka}, t
        rung, L = nxt, L + ka
    lp.bank.close()
    return seen


@pytest.mark.parametrize("d_head", [128, 64])
def test_scheduled_loop_matches_oracle(dev, d_head):
    seen = _run_loop(dev, 24, 100, d_head, _trace(24))
    assert len(seen) >= 3  # the ladder moved across several trees


def test_scheduled_loop_few_tiles_per_step(dev):
    """Steps with far fewer key tiles than CTAs (2 layers x 2 kv heads x 12
    tiles against one CTA per SM) whose tree, and so the split of the tiles,
    changes from step to step: the split merge must combine only partials the
    step itself wrote (stale partials of earlier steps sit in the same
    workspace slots)."""
    g = np.random.default_rng(5)
    trace = (np.round(g.uniform(0.5, 3.5, 12) * 64) / 64).astype(np.float32)
    seen = _run_loop(dev, 12, 1500, 128, trace, seed=2048)
    assert len(seen) >= 4


def test_scheduled_graph_replay_matches_eager(dev):
    steps = 10
    lp = Loop(dev, steps, L0=300, seed=1)
    trace = _trace(steps, seed=4)
    tr_d = to_dev(trace, dev)
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, lp.ids, a=1.5, b=2.5, trace=tr_d,
                         node_stride=N_MAX)
    k0, v0 = lp.kd.clone(), lp.vd.clone()
    # eager
    state = tv.make_state(2, lp.L0, dev)
    for t in range(steps):
        lp.step(t, pol, state)
    torch.cuda.synchronize()
    eager = (tv.parse_state(state), bits(lp.kd), bits(lp.vd), lp.out.clone(), tv.parse_result(lp.res))
    # one CUDA graph of all the steps, replayed from the same initial state
    lp.kd.copy_(k0)
    lp.vd.copy_(v0)
    state.copy_(tv.make_state(2, lp.L0, dev))
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for t in range(steps):
            lp.step(t, pol, state, stream=s)
    for _ in range(2):  # capture records without running: reset, replay, twice
        lp.kd.copy_(k0)
        lp.vd.copy_(v0)
        state.copy_(tv.make_state(2, lp.L0, dev))
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        assert tv.parse_state(state) == eager[0]
        assert np.array_equal(bits(lp.kd), eager[1]) and np.array_equal(bits(lp.vd), eager[2])
        assert torch.equal(lp.out.view(torch.int16), eager[3].view(torch.int16))
        assert tv.parse_result(lp.res) == eager[4]
    assert eager[0]["step"] == steps and eager[0]["L"] > lp.L0
    lp.bank.close()


@pytest.mark.parametrize("feature", ["path_value", "entropy"])
def test_scheduled_features(dev, feature):
    steps = 8
    rungs = (3, 7) if feature == "path_value" else (2, 3, 4, 5)  # the second set tops out at 26 nodes
    lp = Loop(dev, steps, L0=64, seed=2, rungs=rungs)
    g = synth.rng(9)
    if feature == "path_value":
        heads = g.uniform(0.05, 1.0, (steps, 3)).astype(np.float32)
        hd = to_dev(heads, dev)
        # the top-1 probabilities of these V = 1000 rows lie in [0.0020, 0.0045]: thresholds inside
        pol = tv.make_policy(tv.TB_POLICY_BINARY, tv.TB_FEATURE_PATH_VALUE, lp.ids, a=0.0027,
                             b=0.0025, trace=hd, n_heads=3)
    else:
        edges = [6.852, 6.856, 6.860]  # the entropies of these rows lie in [6.840, 6.872]
        # arrays laid out for 64 nodes although the policy's largest tree has 26
        pol = tv.make_policy(tv.TB_POLICY_THRESHOLD_LADDER, tv.TB_FEATURE_ENTROPY, lp.ids, edges=edges,
                             node_stride=N_MAX)
    state = tv.make_state(0, lp.L0, dev)
    rung, L = 0, lp.L0
    for t in range(steps):
        lp.step(t, pol, state, flags=tv.TB_NO_COMPACT)
        torch.cuda.synchronize()
        tree = lp.trees[rung]
        n = len(tree)
        ka, path, bonus = oracle.accept(tree, lp.drafts[t][rung][:n], lp.am[t][:n])
        r = tv.parse_result(lp.res)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["status"]) == (ka, path, bonus, 0), t
        jstar = path[-1]
        st = tv.parse_state(state)
        if feature == "path_value":
            want = oracle.path_value(lp.t1[t][jstar], heads[t].astype(np.float64))
            nxt = oracle.policy_next("binary", rung, 2, st["feature"], np.float32(0.0027), np.float32(0.0025))
        else:
            want = lp.en[t][jstar]
            nxt = oracle.policy_next("threshold", rung, 4, st["feature"], edges=np.float32(edges))
        assert abs(st["feature"] - want) <= STAT_TOL, t
        # the decision is the policy applied to the feature the device computed
        assert (st["rung"], st["L"], st["accept_len"]) == (nxt, L + ka, ka), t
        rung, L = nxt, L + ka
    lp.bank.close()


def test_scheduled_capacity_and_bad_rung(dev):
    lp = Loop(dev, 2, L0=10, seed=5)
    trace = to_dev(np.array([2.0], np.float32), dev)
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, lp.ids, a=1.5, b=2.5, trace=trace,
                         node_stride=N_MAX)
    k0 = bits(lp.kd)
    # L + N beyond the cache: nothing is read past it, the step reports TB_ECAPACITY, the state stays
    state = tv.make_state(7, lp.L_cap - 10, dev)
    lp.step(0, pol, state)
    torch.cuda.synchronize()
    assert tv.parse_result(lp.res)["status"] == tv.TB_ECAPACITY
    assert tv.parse_state(state) == {"rung": 7, "L": lp.L_cap - 10, "step": 0, "feature": 0.0, "accept_len": 0}
    assert np.array_equal(bits(lp.kd), k0)
    # a rung outside the policy: TB_EINVAL, state unchanged
    state = tv.make_state(9, 20, dev)
    lp.step(1, pol, state)
    torch.cuda.synchronize()
    assert tv.parse_result(lp.res)["status"] == tv.TB_EINVAL
    assert tv.parse_state(state)["rung"] == 9 and tv.parse_state(state)["step"] == 0
    # the same workspace still serves a valid step afterwards
    state = tv.make_state(1, 20, dev)
    lp.step(1, pol, state)
    torch.cuda.synchronize()
    assert tv.parse_result(lp.res)["status"] == 0 and tv.parse_state(state)["step"] == 1
    lp.bank.close()


def test_scheduled_argument_errors(dev):
    lp = Loop(dev, 1, L0=10, seed=6)
    state = tv.make_state(0, 10, dev)
    trace = to_dev(np.array([1.0], np.float32), dev)
    bad = [
        tv.make_policy(tv.TB_POLICY_BINARY, tv.TB_FEATURE_TRACE, lp.ids[:3], a=1.0, b=0.5, trace=trace),
        tv.make_policy(tv.TB_POLICY_BINARY, tv.TB_FEATURE_TRACE, lp.ids[:2], a=0.5, b=1.0, trace=trace),
        tv.make_policy(tv.TB_POLICY_THRESHOLD_LADDER, tv.TB_FEATURE_ENTROPY, lp.ids[:3], edges=[2.0, 1.0]),
        tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, lp.ids[:3], a=1.0, b=2.0),
        tv.make_policy(7, tv.TB_FEATURE_TRACE, lp.ids[:3], trace=trace),
        tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_ENTROPY, []),
    ]
    for pol in bad:
        with pytest.raises(tv.TreeVerifyError) as e:
            lp.step(0, pol, state)
        assert e.value.status == tv.TB_EINVAL
    with pytest.raises(tv.TreeVerifyError) as e:  # node stride below the largest tree
        lp.step(0, tv.make_policy(tv.TB_POLICY_THRESHOLD_LADDER, tv.TB_FEATURE_ENTROPY, lp.ids[:8], edges=[1] * 7,
                                  node_stride=40), state)
    assert e.value.status == tv.TB_EINVAL
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_ENTROPY, [lp.ids[0], 99])
    with pytest.raises(tv.TreeVerifyError) as e:
        lp.step(0, pol, state)
    assert e.value.status == tv.TB_ENOTFOUND
    lp.bank.close()
