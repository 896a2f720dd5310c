"""GPU parity of speculative sampling on the draft tree (Sec. 2.1 rule tried
sibling by sibling with the residual; R21) through the C ABI.

Exact: accept_len, path, the drawn token, new_L, status and the compacted
cache.  Every accept / reject decision compares a uniform with a probability
ratio, and the draw compares a uniform with a CDF: both are float decisions,
so the uniforms are redrawn until every decision the oracle takes is at least
1e-4 away from its boundary.  Losslessness is checked on the GPU path itself:
the first emitted token is distributed as the target when the children are
drawn from q.
"""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, draw_decidable_walk as _draw_case, gap_filtered_hidden, \
    softmax_rows as _softmax_rows, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

T = 0.7


@pytest.fixture(scope="module")
def dev():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda:0")


def _walk_on_gpu(dev, bank, parent, draft, z, q, unif, temp, L=0):
    bid, _ = bank.add(parent)
    logz, _ = oracle.tempered_stats(z, temp)
    V = z.shape[1]
    res = tv.make_result(dev)
    scratch = torch.empty(V, dtype=torch.float32, device=dev)
    tv.spec_sample_accept(bank, bid, to_dev(np.asarray(draft, np.int32), dev), to_dev(z.astype(np.float32), dev),
                          to_dev(logz.astype(np.float32), dev), to_dev(q.astype(np.float32), dev),
                          to_dev(unif.astype(np.float32), dev), L, temp, scratch, res)
    torch.cuda.synchronize()
    return tv.parse_result(res)


def test_walk_random_trees_vs_oracle(dev):
    b = tv.Bank(512, 0)
    g = synth.rng(31)
    deep = 0
    for trial in range(200):
        n = int(g.integers(1, 65))
        kind = trial % 3
        parent = (synth.rank_product_tree(synth.BANK_BRANCHING, n) if kind == 0 else
                  synth.chain(n) if kind == 1 else np.sort(synth.random_tree(g, n)))
        parent = np.asarray(parent, np.int32)
        parent[0] = -1
        V = int(g.choice([3, 17, 100, 1000, 4099]))
        # float32-representable logits and draft distributions: both sides see the same numbers
        z = (g.standard_normal((n, V)) * float(g.uniform(0.3, 3.0))).astype(np.float32).astype(np.float64)
        q = _softmax_rows(g.standard_normal((n, V)) * float(g.uniform(0.3, 3.0)), 1.0)
        q = (q / q.sum(axis=1, keepdims=True)).astype(np.float32).astype(np.float64)
        draft, unif, want = _draw_case(g, parent, z, q, T)
        r = _walk_on_gpu(dev, b, parent, draft, z, q, unif, T, L=trial)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
            want[0], want[1], want[2], trial + want[0], 0), trial
        deep += want[0] > 2
    assert deep > 20
    b.close()


def _spiky_rows(g, n, V, spikes, temp):
    """Logits: N(0, 1) plus +U(8, 12) on `spikes` tokens of each row, so most of
    p's mass sits on a few tokens anywhere in the vocabulary (the draw stays
    decidable at any V).  Draft distribution: two of p's spikes and two of its
    own, plus the background, so the residual keeps peaks after a rejection."""
    z = g.standard_normal((n, V))
    q = g.standard_normal((n, V)) * 0.5
    for u in range(n):
        hot = g.choice(V, size=spikes + 2, replace=False)
        z[u, hot[:spikes]] += g.uniform(8.0, 12.0, size=spikes)
        q[u, np.concatenate([hot[:2], hot[spikes:]])] += g.uniform(11.0, 14.0, size=4)
    z = z.astype(np.float32).astype(np.float64)
    q = _softmax_rows(q, 1.0)
    return z, (q / q.sum(axis=1, keepdims=True)).astype(np.float32).astype(np.float64)


@pytest.mark.parametrize("V", [32767, 32768, 32772, 50001, 131072, 131073, 150004])
def test_walk_vocab_paths(dev, V):
    """Vocabularies on both sides of the register-slice limits of the cluster
    walk (8 CTAs x 1024 threads x 4 or 16 entries: 32768 and 131072) and past
    them (the one-CTA walk), with 16-byte and unaligned rows; the spikes fall
    in the slices of every CTA."""
    b = tv.Bank(16, 0)
    g = synth.rng(34 + V % 97)
    trees = [synth.bank_trees()[-1], synth.chain(9), np.sort(synth.random_tree(g, 40)), synth.bank_trees()[5]]
    for trial, parent in enumerate(trees):
        parent = np.asarray(parent, np.int32)
        parent[0] = -1
        z, q = _spiky_rows(g, len(parent), V, 4, T)
        draft, unif, want = _draw_case(g, parent, z, q, T)
        r = _walk_on_gpu(dev, b, parent, draft, z, q, unif, T, L=trial)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
            want[0], want[1], want[2], trial + want[0], 0), (V, trial)
    b.close()


def test_walk_is_lossless_on_the_gpu(dev):
    """Root with three children drawn from q: the first emitted token follows p."""
    b = tv.Bank(4, 0)
    parent = np.array([-1, 0, 0, 0], np.int32)
    bid, _ = b.add(parent)
    g = synth.rng(32)
    V, trials = 8, 4000
    z = (g.standard_normal(V) * 1.5).astype(np.float32).astype(np.float64)
    p = _softmax_rows(z[None], T)[0]
    q = _softmax_rows(g.standard_normal((1, V)) * 1.5, 1.0)[0].astype(np.float32)
    zt = to_dev(np.tile(z, (4, 1)).astype(np.float32), dev)
    logz, _ = oracle.tempered_stats(np.tile(z, (4, 1)), T)
    lz = to_dev(logz.astype(np.float32), dev)
    qt = to_dev(np.tile(q, (4, 1)), dev)
    drafts = np.concatenate([np.zeros((trials, 1), np.int32),
                             g.choice(V, size=(trials, 3), p=q / q.sum()).astype(np.int32)], 1)
    unifs = g.random((trials, 8)).astype(np.float32)
    dd, ud = to_dev(drafts, dev), to_dev(unifs, dev)
    res = torch.empty((trials, tv.RESULT_INTS), dtype=torch.int32, device=dev)
    scratch = torch.empty(V, dtype=torch.float32, device=dev)
    for i in range(trials):
        tv.spec_sample_accept(b, bid, dd[i], zt, lz, qt, ud[i], 0, T, scratch, res[i])
    torch.cuda.synchronize()
    rh = res.cpu().numpy()
    first = np.where(rh[:, 0] > 1, drafts[np.arange(trials), rh[:, 4 + 1]], rh[:, 1])
    freq = np.bincount(first, minlength=V) / trials
    # binomial standard error <= 0.008: 5 sigma
    assert np.abs(freq - p).max() < 0.04, (freq, p)
    b.close()


@pytest.mark.parametrize("cfg", ["c1", "c2"])
def test_verify_step_sampled_parity(dev, cfg):
    sh = synth.SHAPES[cfg]()
    parent = np.asarray(sh.parent, np.int32)
    N, L, H, Hkv, d, D, V = sh.N, sh.L, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model, sh.vocab
    b = tv.Bank(4, 0)
    bid, _ = b.add(parent)
    g = synth.rng(33)
    k, v = synth.gen_kv(33, 1, Hkv, L + N + 3, d, L + N)
    qv = synth.gen_q(33, 1, N, H, d)
    W = synth.gen_lm_head(33, V, D)
    hidden, am, t1, en, logits = gap_filtered_hidden(33, N, W, want_logits=True)
    # the draft distributions: the target sharpened and mixed with noise (a head that mostly agrees)
    qd = _softmax_rows(logits / T * 1.3 + g.standard_normal((N, V)) * 0.5, 1.0)
    qd = (qd / qd.sum(axis=1, keepdims=True)).astype(np.float32).astype(np.float64)
    draft, unif, want = _draw_case(g, parent, logits, qd, T)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    out = torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(N, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
    g_en = torch.empty(N, dtype=torch.float32, device=dev)
    lg = torch.full((N + 1, V), float("nan"), dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, 1, Hkv, H, d, V, 0), dev)
    tv.verify_step_sampled(b, bid, tv.KvCache(kd, vd, L), to_dev(qv, dev), to_dev(hidden, dev), to_dev(W, dev),
                           to_dev(draft, dev), to_dev(qd.astype(np.float32), dev), to_dev(unif.astype(np.float32), dev),
                           T, out, g_am, g_t1, g_en, lg, res, ws)
    torch.cuda.synchronize()
    check_attention(out[0].float().cpu().numpy(), oracle.tree_attention(qv[0], k[0], v[0], L, parent))
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    assert np.abs(lg[:N].cpu().numpy() - logits).max() <= 1e-3
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
        want[0], want[1], want[2], L + want[0], 0)
    assert np.array_equal(bits(kd), oracle.kv_compact(k, L, want[1]))
    assert np.array_equal(bits(vd), oracle.kv_compact(v, L, want[1]))
    b.close()


def test_sampled_argument_errors(dev):
    b = tv.Bank(4, 0)
    bid, _ = b.add([-1, 0])
    i = torch.zeros(2, dtype=torch.int32, device=dev)
    f = torch.zeros((2, 4), dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    for temp in (0.0, -1.0, float("nan")):
        with pytest.raises(tv.TreeVerifyError) as e:
            tv.spec_sample_accept(b, bid, i, f, f[0], f, f[0], 0, temp, f[0], res)
        assert e.value.status == tv.TB_EINVAL
    # a bad draft token is never accepted and sets the status
    z = np.zeros((2, 4))
    r = _walk_on_gpu(dev, b, [-1, 0], [0, 9], z, np.full((2, 4), 0.25), np.zeros(4), T)
    assert r["status"] == tv.TB_EINVAL and r["accept_len"] == 1
    b.close()
