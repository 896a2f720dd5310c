"""The bank-switching decode loop at the 7B single-layer shapes (32 x 128 heads,
d_model 4096, V 32000): the 8-tree bank, L from 2048 growing by accept_len,
KV compaction every step, and the hysteretic step ladder (one rung up below
1.5 nats, one down above 2.5) over the seeded AR(1) entropy trace (mu 2.0,
phi 0.9, sigma 0.35, seed 0) -- the paper's per-step tree selection (Sec. 4
"Policy") around its verification pass and KV-cache update (Sec. 3.2).

The configured loop runs 1000 steps, host-driven (verify_step, the tree picked
on the host) and device-driven (verify_step_scheduled, the tree picked by the
acceptance kernel).  Hidden rows come from a pool whose oracle argmax is known,
so every step's acceptance (accept_len, path, bonus token, new L) and every
policy decision is checked against the oracle; every 50th step the attention
of all heads, the LM-head statistics and the whole compacted cache are
checked as well.  A short hand-made trace checks the ladder's walk exactly."""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, gap_filtered_hidden, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

STEPS = 1000
CHECK_EVERY = 50
POOL_ROWS = 576   # hidden rows with known oracle argmax (>= 512, more than any step needs)
Q_POOL = 8        # query tensors cycled through the steps (they do not affect acceptance)
UP, DOWN = 1.5, 2.5


@pytest.fixture(scope="module")
def setup():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda:0")
    sh = synth.shape_c3()
    W = synth.gen_lm_head(31, sh.vocab, sh.d_model)
    pool = gap_filtered_hidden(41, POOL_ROWS, W)
    trace = synth.ar1_entropy_trace(0, STEPS, hmax=float(np.log(sh.vocab))).astype(np.float32)
    return dev, sh, W, to_dev(W, dev), pool, trace


class Cache:
    """Device K/V cache of L_cap slots (all finite random values) and its host
    reference, updated with the oracle's compaction of each step's tree window."""

    def __init__(self, dev, sh, seed):
        H, d = sh.n_q_heads, sh.head_dim
        self.k, self.v = synth.gen_kv(seed, 1, H, sh.L_cap, d, sh.L_cap)
        self.kd, self.vd = to_dev(self.k, dev), to_dev(self.v, dev)

    def compact(self, L, n, path):
        # the oracle's compaction, applied to the window [L, L + n) it can touch
        for a in (self.k, self.v):
            a[:, :, L:L + n] = oracle.kv_compact(a[:, :, L:L + n], 0, path)

    def check(self, what):
        assert np.array_equal(bits(self.kd), self.k) and np.array_equal(bits(self.vd), self.v), what


def _rows(t, n, pool):
    g = synth.rng(5000 + t, 11)
    idx = g.choice(POOL_ROWS, n, replace=False)
    return tuple(x[idx] for x in pool)


def _check_full(step, L, tree, q, cache, out, g_am, g_t1, g_en, am, t1, en):
    n = len(tree)
    got = out.float().cpu().numpy()[0][:n]
    ref = oracle.tree_attention(q[0][:n], cache.k[0], cache.v[0], L, tree)
    check_attention(got, ref, f"step {step}")
    assert np.array_equal(g_am.cpu().numpy()[:n], am)
    assert np.abs(g_t1.cpu().numpy()[:n] - t1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy()[:n] - en).max() <= STAT_TOL


def test_bank_loop_configured_host_driven(setup):
    dev, sh, W, Wd, pool, trace = setup
    H, d, V = sh.n_q_heads, sh.head_dim, sh.vocab
    trees = synth.bank_trees()
    bank = tv.Bank(16, 0)
    ids = [bank.add(t)[0] for t in trees]
    cache = Cache(dev, sh, 31)
    qs = [synth.gen_q(300 + i, 1, 64, H, d) for i in range(Q_POOL)]
    qds = [to_dev(x, dev) for x in qs]
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, H, H, d, V, 0), dev)
    out = torch.empty((1, 64, H, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(64, dtype=torch.int32, device=dev)
    g_t1, g_en = (torch.empty(64, dtype=torch.float32, device=dev) for _ in range(2))
    res = tv.make_result(dev)
    L, kix = sh.L, 0
    visits = np.zeros(len(trees), int)
    for t in range(STEPS):
        nxt = tv.tb_schedule_hysteretic_ladder(kix, len(trees), float(trace[t]), UP, DOWN)
        assert nxt == oracle.policy_next("ladder", kix, len(trees), float(trace[t]), UP, DOWN), t
        kix = nxt
        visits[kix] += 1
        tree = trees[kix]
        n = len(tree)
        h, am, t1, en = _rows(t, n, pool)
        drafts = synth.gen_drafts(7000 + t, tree, am, V, sh.p_match)
        q = qs[t % Q_POOL]
        tv.verify_step(bank, ids[kix], tv.KvCache(cache.kd, cache.vd, L), qds[t % Q_POOL][:, :n], to_dev(h, dev), Wd,
                       to_dev(drafts, dev), out[:, :n], g_am[:n], g_t1[:n], g_en[:n], res, ws)
        r = tv.parse_result(res)  # synchronises
        ka, path, bonus = oracle.accept(tree, drafts, am)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0), t
        if t % CHECK_EVERY == 0 or t == STEPS - 1:
            _check_full(t, L, tree, q, cache, out, g_am, g_t1, g_en, am, t1, en)
        cache.compact(L, n, path)
        if t % CHECK_EVERY == 0 or t == STEPS - 1:
            cache.check(f"cache after step {t}")
        L += ka
    assert (visits > 0).all(), visits  # the ladder visits every rung of the bank
    assert L <= sh.L_cap
    bank.close()


def test_bank_loop_configured_device_driven(setup):
    dev, sh, W, Wd, pool, trace = setup
    H, d, V = sh.n_q_heads, sh.head_dim, sh.vocab
    trees = synth.bank_trees()
    n_max = max(len(t) for t in trees)
    bank = tv.Bank(16, 0)
    ids = [bank.add(t)[0] for t in trees]
    cache = Cache(dev, sh, 32)
    qs = [synth.gen_q(400 + i, 1, n_max, H, d) for i in range(Q_POOL)]
    qds = [to_dev(x, dev) for x in qs]
    ws = tv.make_workspace(tv.tb_workspace_size(n_max, 1, H, H, d, V, 0), dev)
    out = torch.empty((1, n_max, H, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(n_max, dtype=torch.int32, device=dev)
    g_t1, g_en = (torch.empty(n_max, dtype=torch.float32, device=dev) for _ in range(2))
    res = tv.make_result(dev)
    tr_d = to_dev(trace, dev)
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, ids, a=UP, b=DOWN, trace=tr_d,
                         node_stride=n_max)
    state = tv.make_state(0, sh.L, dev)
    L, rung = sh.L, 0
    visits = np.zeros(len(trees), int)
    for t in range(STEPS):
        visits[rung] += 1
        tree = trees[rung]
        n = len(tree)
        h, am, t1, en = _rows(t, n_max, pool)
        rows = np.zeros((len(trees), n_max), np.int32)
        for j, tj in enumerate(trees):
            rows[j, :len(tj)] = synth.gen_drafts(9000 + 8 * t + j, tj, am[:len(tj)], V, sh.p_match)
        q = qs[t % Q_POOL]
        tv.verify_step_scheduled(bank, pol, state, tv.KvCache(cache.kd, cache.vd, 0), qds[t % Q_POOL], to_dev(h, dev),
                                 Wd, to_dev(rows, dev), out, g_am, g_t1, g_en, res, ws)
        r = tv.parse_result(res)  # synchronises
        ka, path, bonus = oracle.accept(tree, rows[rung, :n], am[:n])
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0), t
        nxt = oracle.policy_next("ladder", rung, len(trees), float(trace[t]), UP, DOWN)
        st = tv.parse_state(state)
        assert st == {"rung": nxt, "L": L + ka, "step": t + 1, "feature": float(trace[t]), "accept_len": ka}, t
        if t % CHECK_EVERY == 0 or t == STEPS - 1:
            _check_full(t, L, tree, q, cache, out, g_am, g_t1, g_en, am[:n], t1[:n], en[:n])
        cache.compact(L, n, path)
        if t % CHECK_EVERY == 0 or t == STEPS - 1:
            cache.check(f"cache after step {t}")
        L, rung = L + ka, nxt
    assert (visits > 0).all(), visits
    bank.close()


def test_bank_loop_hand_trace(setup):
    """Ten steps on a hand-made trace (six low-entropy steps, then four high):
    the ladder walks up and back down, every step checked in full."""
    dev, sh, W, Wd, pool, _ = setup
    H, d, V = sh.n_q_heads, sh.head_dim, sh.vocab
    steps = 10
    trees = synth.bank_trees()
    bank = tv.Bank(16, 0)
    ids = [bank.add(t)[0] for t in trees]
    cache = Cache(dev, sh, 33)
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, H, H, d, V, 0), dev)
    trace = np.concatenate([np.full(6, 1.0), np.full(4, 3.0)])
    L, kix = sh.L, 0
    seen = []
    for step in range(steps):
        kix = tv.tb_schedule_hysteretic_ladder(kix, len(trees), float(trace[step]), UP, DOWN)
        seen.append(kix)
        tree = trees[kix]
        n = len(tree)
        q = synth.gen_q(200 + step, 1, n, H, d)
        h, am, t1, en = _rows(100000 + step, n, pool)
        drafts = synth.gen_drafts(200 + step, tree, am, V, sh.p_match)
        out = torch.empty((1, n, H, d), dtype=torch.bfloat16, device=dev)
        g_am = torch.empty(n, dtype=torch.int32, device=dev)
        g_t1, g_en = (torch.empty(n, dtype=torch.float32, device=dev) for _ in range(2))
        res = tv.make_result(dev)
        tv.verify_step(bank, ids[kix], tv.KvCache(cache.kd, cache.vd, L), to_dev(q, dev), to_dev(h, dev), Wd,
                       to_dev(drafts, dev), out, g_am, g_t1, g_en, res, ws)
        r = tv.parse_result(res)
        _check_full(step, L, tree, q, cache, out, g_am, g_t1, g_en, am, t1, en)
        ka, path, bonus = oracle.accept(tree, drafts, am)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        cache.compact(L, n, path)
        cache.check(f"step {step}")
        L = r["new_L"]
    assert seen == [1, 2, 3, 4, 5, 6, 5, 4, 3, 2]
    bank.close()
