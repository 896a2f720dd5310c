"""GPU parity of the rotary embedding at the tree's position offsets (node i
at L + depth(i)) against the fp64 oracle, through the C ABI.

Attention: max-abs <= 1e-2 and mean-abs <= 1e-3 as everywhere.  The rotated
tree keys are stored back into the bf16 cache: they may differ from the
oracle's (fp64 rotation, rounded once) by one bf16 ulp where the float
rotation lands next to a rounding boundary, or by a tiny absolute amount
where the rotation cancels (see ROT_ABS_TOL); everything else in the cache
(prefix keys, all values) must be byte-identical, and acceptance, path and
bonus token exact.
"""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, abs_bits, bits, check_attention, check_attention_fuzz, gap_filtered_hidden, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

THETA = 10000.0


@pytest.fixture(scope="module")
def dev():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda:0")


@pytest.fixture(scope="module")
def bank(dev):
    b = tv.Bank(64, 0)
    yield b
    b.close()


def _ordered(b):
    """bf16 bit patterns -> integers ordered like the values (adjacent values differ by 1)."""
    x = b.astype(np.int32)
    return np.where(x & 0x8000, 0x8000 - x, x)


def _bf16_value(b):
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# Where the rotation cancels (x1 c - x2 s far below the inputs' magnitude) the
# absolute error of the fp32 rotation, a few roundings of 2^-24 of inputs that
# are N(0, 1) bf16 (|x1| + |x2| below 10), spans several bf16 ulps of the small
# result: such elements may differ by up to 2^-18 in value.
ROT_ABS_TOL = 2.0 ** -18


def check_rotated_keys(got, ref, what="rotated keys"):
    diff = np.abs(_ordered(got) - _ordered(ref))
    far = diff > 1
    if far.any():
        gap = np.abs(_bf16_value(got[far]) - _bf16_value(ref[far]))
        assert gap.max() <= ROT_ABS_TOL, f"{what}: {diff.max()} bf16 ulps and {gap.max():.2e} apart"
    frac = float((diff > 0).mean())
    assert frac < 0.01, f"{what}: {frac:.4f} of the elements differ"
    return frac


CASES = [
    # parent, L, layers, Hq, Hkv
    (synth.full_tree((2, 2)), 128, 1, 4, 4),
    (synth.bank_trees()[-1], 0, 1, 8, 2),        # L = 0: the tree alone, positions 0..5
    (synth.shape_c2().parent, 1024, 2, 8, 8),
    (synth.chain(17), 333, 1, 2, 2),
    ([-1], 77, 1, 4, 1),
    (synth.bank_trees()[-1], 16384, 1, 4, 4),    # positions near 16k (angles ~ 10^4 rad)
]


@pytest.mark.parametrize("d", [128, 64])
@pytest.mark.parametrize("parent,L,layers,Hq,Hkv", CASES)
def test_tree_attention_rope_parity(dev, bank, parent, L, layers, Hq, Hkv, d):
    parent = np.asarray(parent, np.int32)
    N = len(parent)
    bid, _ = bank.add(parent)
    seed = 40 + N + L + d
    k, v = synth.gen_kv(seed, layers, Hkv, L + N + 4, d, L + N)
    q = synth.gen_q(seed, layers, N, Hq, d)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    kv = tv.KvCache(kd, vd, L, rope_theta=THETA)
    out = torch.empty((layers, N, Hq, d), dtype=torch.bfloat16, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, layers, Hkv, Hq, d, 1, 0), dev)
    tv.tree_attention(bank, bid, kv, to_dev(q, dev), out, ws)
    torch.cuda.synchronize()
    got_k = bits(kd)
    for layer in range(layers):
        ref, k_rot = oracle.tree_attention_rope(q[layer], k[layer], v[layer], L, parent, THETA)
        check_attention(out[layer].float().cpu().numpy(), ref, f"layer {layer}")
        check_rotated_keys(got_k[layer][:, L:L + N], k_rot, f"layer {layer}")
        assert np.array_equal(got_k[layer][:, :L], k[layer][:, :L])          # prefix untouched
        assert np.array_equal(got_k[layer][:, L + N:], k[layer][:, L + N:])  # beyond the tree untouched
    assert np.array_equal(bits(vd), v)


def test_tree_attention_rope_layer_subset(dev, bank):
    parent = np.asarray(synth.bank_trees()[5], np.int32)
    N, L, layers, H, d = len(parent), 200, 3, 4, 128
    bid, _ = bank.add(parent)
    k, v = synth.gen_kv(5, layers, H, L + N, d, L + N)
    q = synth.gen_q(5, layers, N, H, d)
    kd = to_dev(k, dev)
    out = torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, layers, H, H, d, 1, 0), dev)
    tv.tree_attention(bank, bid, tv.KvCache(kd, to_dev(v, dev), L, rope_theta=THETA), to_dev(q[1:2], dev), out, ws, 1, 1)
    torch.cuda.synchronize()
    ref, k_rot = oracle.tree_attention_rope(q[1], k[1], v[1], L, parent, THETA)
    check_attention(out[0].float().cpu().numpy(), ref)
    got_k = bits(kd)
    check_rotated_keys(got_k[1][:, L:L + N], k_rot)
    assert np.array_equal(got_k[0], k[0]) and np.array_equal(got_k[2], k[2])  # only the layer run is rotated


def test_verify_step_rope_parity(dev, bank):
    sh = synth.shape_c2()
    parent = np.asarray(sh.parent, np.int32)
    N, L, H, d, D, V = sh.N, sh.L, sh.n_q_heads, sh.head_dim, sh.d_model, sh.vocab
    bid, _ = bank.add(parent)
    k, v = synth.gen_kv(7, 1, H, L + N + 3, d, L + N)
    q = synth.gen_q(7, 1, N, H, d)
    W = synth.gen_lm_head(7, V, D)
    hidden, am, t1, en = gap_filtered_hidden(7, N, W)
    drafts = synth.gen_drafts(7, parent, am, V, sh.p_match)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    out = torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(N, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
    g_en = torch.empty(N, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, 1, H, H, d, V, 0), dev)
    tv.verify_step(bank, bid, tv.KvCache(kd, vd, L, rope_theta=THETA), to_dev(q, dev), to_dev(hidden, dev),
                   to_dev(W, dev), to_dev(drafts, dev), out, g_am, g_t1, g_en, res, ws)
    torch.cuda.synchronize()
    ref, k_rot = oracle.tree_attention_rope(q[0], k[0], v[0], L, parent, THETA)
    check_attention(out[0].float().cpu().numpy(), ref)
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    ka, path, bonus = oracle.accept(parent, drafts, am)
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
    # the cache after the step: rotated tree keys, then the accepted rows compacted
    k_ref = k.copy()
    k_ref[0][:, L:L + N] = k_rot
    k_ref = oracle.kv_compact(k_ref, L, path)
    got_k = bits(kd)
    check_rotated_keys(got_k[0][:, L:L + N], k_ref[0][:, L:L + N])
    assert np.array_equal(got_k[0][:, :L], k[0][:, :L])
    assert np.array_equal(bits(vd), oracle.kv_compact(v, L, path))


@pytest.mark.parametrize("d", [128, 64])
def test_batched_rope_parity(dev, d):
    b = tv.Bank(16, 0)
    Hq, Hkv, D, V = 8, 2, 256, 1000
    trees = synth.bank_trees()
    parents = [trees[-1], trees[0], trees[5], trees[3]]
    Ls = [0, 5000, 129, 777]
    W = synth.gen_lm_head(50, V, D)
    rows = sum(len(p) for p in parents)
    hidden, am, t1, en = gap_filtered_hidden(51, rows, W)
    seqs, host = [], []
    for i, (parent, L) in enumerate(zip(parents, Ls)):
        parent = np.asarray(parent, np.int32)
        N = len(parent)
        k, v = synth.gen_kv(60 + i, 1, Hkv, L + N + 2, d, L + N)
        q = synth.gen_q(60 + i, 1, N, Hq, d)
        bid, _ = b.add(parent)
        s = tv.Seq(bid, tv.KvCache(to_dev(k, dev), to_dev(v, dev), L, rope_theta=THETA), to_dev(q, dev),
                   torch.zeros(N, dtype=torch.int32, device=dev),
                   torch.empty((1, N, Hq, d), dtype=torch.bfloat16, device=dev), tv.make_result(dev))
        seqs.append(s)
        host.append((parent, L, k, v, q))
    g_am = torch.empty(rows, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(rows, dtype=torch.float32, device=dev)
    g_en = torch.empty(rows, dtype=torch.float32, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(rows, 1, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_batched(b, seqs, to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws, tv.TB_NO_COMPACT)
    torch.cuda.synchronize()
    for s, (parent, L, k, v, q) in zip(seqs, host):
        N = len(parent)
        ref, k_rot = oracle.tree_attention_rope(q[0], k[0], v[0], L, parent, THETA)
        check_attention(s.attn_out[0].float().cpu().numpy(), ref, f"L={L}")
        check_rotated_keys(bits(s.kv.k)[0][:, L:L + N], k_rot)
    b.close()


def test_scheduled_rope_parity(dev):
    """Two steps of the device-driven loop with the rotary embedding: the
    positions come from the device-held prefix length."""
    b = tv.Bank(8, 0)
    trees = [synth.bank_trees()[i] for i in (3, 7)]
    ids = [b.add(t)[0] for t in trees]
    Hq, Hkv, d, D, V, L0, steps = 4, 2, 128, 256, 1000, 900, 2
    L_cap = L0 + 64 + 64 + 8
    k, v = synth.gen_kv(70, 1, Hkv, L_cap, d, L_cap)
    W = synth.gen_lm_head(70, V, D)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    trace = to_dev(np.array([0.0, 0.0], np.float32), dev)  # feature 0 < 1: step up to the 64-node tree
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, ids, a=1.0, b=2.0, trace=trace)
    state = tv.make_state(0, L0, dev)
    out = torch.empty((1, 64, Hq, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(64, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(64, dtype=torch.float32, device=dev)
    g_en = torch.empty(64, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, Hkv, Hq, d, V, 0), dev)
    k_ref, v_ref, rung, L = k.copy(), v.copy(), 0, L0
    for t in range(steps):
        q = synth.gen_q(80 + t, 1, 64, Hq, d)
        hidden, am, t1, en = gap_filtered_hidden(90 + t, 64, W)
        tab = np.zeros((2, 64), np.int32)
        for r, tr in enumerate(trees):
            tab[r, :len(tr)] = synth.gen_drafts(100 + t + r, tr, am[:len(tr)], V, 0.8)
        tv.verify_step_scheduled(b, pol, state, tv.KvCache(kd, vd, 0, rope_theta=THETA), to_dev(q, dev),
                                 to_dev(hidden, dev), to_dev(W, dev), to_dev(tab, dev), out, g_am, g_t1, g_en, res, ws)
        torch.cuda.synchronize()
        tree = np.asarray(trees[rung], np.int32)
        n = len(tree)
        ref, k_rot = oracle.tree_attention_rope(q[0][:n], k_ref[0], v_ref[0], L, tree, THETA)
        check_attention(out[0][:n].float().cpu().numpy(), ref, f"step {t}")
        ka, path, bonus = oracle.accept(tree, tab[rung][:n], am[:n])
        r = tv.parse_result(res)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["status"]) == (ka, path, bonus, 0)
        k_ref[0][:, L:L + n] = k_rot
        k_ref = oracle.kv_compact(k_ref, L, path)
        v_ref = oracle.kv_compact(v_ref, L, path)
        got_k = bits(kd)
        check_rotated_keys(got_k[0][:, L0:L + n], k_ref[0][:, L0:L + n], f"step {t}")
        # keep the oracle's cache on the GPU's bytes so that the next step compares like with like
        k_ref = got_k.copy()
        assert np.array_equal(bits(vd), v_ref)
        rung, L = min(rung + 1, 1), L + ka
    b.close()


def test_rope_argument_errors(dev, bank):
    bid, _ = bank.add([-1, 0])
    ws = tv.make_workspace(tv.tb_workspace_size(2, 1, 2, 2, 128, 1, 0), dev)
    q = torch.zeros((1, 2, 2, 128), dtype=torch.bfloat16, device=dev)
    k = torch.zeros((1, 2, 16, 128), dtype=torch.bfloat16, device=dev)
    for theta in (-1.0, float("nan"), float("inf")):
        with pytest.raises(tv.TreeVerifyError) as e:
            tv.tree_attention(bank, bid, tv.KvCache(k, k.clone(), 4, rope_theta=theta), q, torch.empty_like(q), ws)
        assert e.value.status == tv.TB_EINVAL


@pytest.mark.parametrize("seed", range(24))
def test_random_rope_attention(dev, seed):
    """Random shapes with the rotary embedding: random trees, prefix lengths
    0-16000, head_dim 64 and 128, GQA groups, one or two layers; attention
    within the derived bound of the fuzz tests (short prefixes give outputs
    of order 1), rotated keys as above, prefix keys and values untouched."""
    g = synth.rng(3300 + seed)
    n = int(g.integers(1, 65))
    parent = np.sort(synth.random_tree(g, n))
    parent[0] = -1
    d = int(g.choice([64, 128]))
    Hkv = int(g.choice([1, 2, 4]))
    group = int(g.choice([1, 2, 4]))
    while n * group > 256:
        group //= 2
    Hq = Hkv * group
    L = int(g.choice([0, 5, 130, 700, 3000, 16000]))
    layers = int(g.integers(1, 3))
    b = tv.Bank(4, 0)
    bid, _ = b.add(parent)
    k, v = synth.gen_kv(seed, layers, Hkv, L + n + 4, d, L + n)
    q = synth.gen_q(seed, layers, n, Hq, d)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    out = torch.empty((layers, n, Hq, d), dtype=torch.bfloat16, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(n, layers, Hkv, Hq, d, 1, 0), dev)
    tv.tree_attention(b, bid, tv.KvCache(kd, vd, L, rope_theta=THETA), to_dev(q, dev), out, ws)
    torch.cuda.synchronize()
    got_k = bits(kd)
    o = out.float().cpu().numpy()
    for layer in range(layers):
        ref, k_rot = oracle.tree_attention_rope(q[layer], k[layer], v[layer], L, parent, THETA)
        ref_a, _ = oracle.tree_attention_rope(q[layer], k[layer], abs_bits(v[layer]), L, parent, THETA)
        check_attention_fuzz(o[layer], ref, ref_a, f"seed {seed} layer {layer} (n={n} L={L} d={d} Hq={Hq} Hkv={Hkv})")
        check_rotated_keys(got_k[layer][:, L:L + n], k_rot, f"seed {seed} layer {layer}")
        assert np.array_equal(got_k[layer][:, :L], k[layer][:, :L])
    assert np.array_equal(bits(vd), v)
    b.close()
