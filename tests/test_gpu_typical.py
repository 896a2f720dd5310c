"""GPU parity of typical acceptance (the Medusa/Hydra rule the paper runs with
T = 0.7, eps = 0.09, alpha = 0.3) through the C ABI against the fp64 oracle.

Bit-exact: argmax, accept_len, path, bonus token, compacted KV bytes.
Tempered log-partition, tempered entropy, gathered draft logits: <= 1e-3 abs;
top-1 / entropy at temperature 1 as in the greedy tests.  Hidden rows keep an
oracle top-2 logit gap > 1e-2 and drafts keep every edge decision at least
1e-3 (relative) away from its threshold, so fp32 and fp64 decide alike.
"""
import numpy as np
import pytest

import oracle
from helpers import (LOGIT_TOL, STAT_TOL, TYPICAL, abs_bits, bits, check_attention, check_attention_fuzz,
                     gap_filtered_hidden, to_dev, typical_ambiguity, typical_drafts)
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda:0")


@pytest.fixture(scope="module")
def bank(dev):
    b = tv.Bank(512, 0)
    yield b
    b.close()


def _rows(seed, parent, D, V):
    """Gap-filtered hidden rows of a tree, the LM head, and the oracle's fp64 logits."""
    W = synth.gen_lm_head(seed, V, D)
    hidden, am, t1, en, logits = gap_filtered_hidden(seed, len(parent), W, want_logits=True)
    return W, hidden, am, t1, en, logits


def _f32(n, dev, fill=float("nan")):
    return torch.full((n,), fill, dtype=torch.float32, device=dev)


# ---------------------------------------------------------------- LM head (K2, typical mode)

LM_CASES = [
    # parent, D, V, temperature
    (synth.full_tree((2, 2)), 256, 1000, 0.7),
    (synth.shape_c2().parent, 4096, 32000, 0.7),
    (synth.bank_trees()[-1], 512, 4099, 1.3),   # 64 rows, ragged last vocab tile
    ([-1], 128, 129, 0.7),                      # single node: no edges to gather
    (synth.chain(17), 320, 2000, 0.25),
    (synth.bank_trees()[-1], 128, 100003, 0.7),  # several vocab tiles per persistent CTA
]


@pytest.mark.parametrize("parent,D,V,T", LM_CASES)
def test_lm_head_typical_matches_oracle(dev, bank, parent, D, V, T):
    parent = np.asarray(parent, np.int32)
    N = len(parent)
    bid, _ = bank.add(parent)
    W, hidden, am, t1, en, logits = _rows(100 + N, parent, D, V)
    drafts = typical_drafts(200 + N, parent, logits, T, *TYPICAL[1:])
    if N > 2:
        drafts[1] = -1      # out of range on both sides: never gathered
        drafts[2] = V
    g = [torch.full((N,), -1, dtype=torch.int32, device=dev)] + [_f32(N, dev) for _ in range(5)]
    ws = tv.make_workspace(tv.tb_workspace_size(N, 0, 0, 0, 0, V, 0), dev)
    tv.lm_head_stats_typical(bank, bid, to_dev(hidden, dev), to_dev(W, dev), T, to_dev(drafts, dev), *g, ws)
    torch.cuda.synchronize()
    g_am, g_t1, g_en, g_lz, g_et, g_dl = [x.cpu().numpy() for x in g]
    assert np.array_equal(g_am, am)
    assert np.abs(g_t1 - t1).max() <= STAT_TOL
    assert np.abs(g_en - en).max() <= STAT_TOL
    logz, ent = oracle.tempered_stats(logits, T)
    assert np.abs(g_lz - logz).max() <= LOGIT_TOL
    assert np.abs(g_et - ent).max() <= LOGIT_TOL
    assert np.isnan(g_dl[0])
    for j in range(1, N):
        if 0 <= drafts[j] < V:
            assert abs(g_dl[j] - logits[parent[j], drafts[j]]) <= LOGIT_TOL, j
        else:
            assert np.isnan(g_dl[j]), j


# ---------------------------------------------------------------- acceptance (K3, typical mode)

def _k3_inputs(logits, parent, drafts, T):
    logz, ent = oracle.tempered_stats(logits, T)
    dl = np.full(len(parent), np.nan, dtype=np.float32)
    for j in range(1, len(parent)):
        if 0 <= drafts[j] < logits.shape[1]:
            dl[j] = logits[parent[j], drafts[j]]
    return logz.astype(np.float32), ent.astype(np.float32), dl, logits.argmax(axis=1).astype(np.int32)


def _typical_on_gpu(dev, bank, parent, drafts, logits, T, eps, alpha, L=0):
    bid, _ = bank.add(parent)
    logz, ent, dl, am = _k3_inputs(logits, parent, drafts, T)
    res = tv.make_result(dev)
    tv.typical_accept(bank, bid, to_dev(np.asarray(drafts, np.int32), dev), to_dev(am, dev), to_dev(logz, dev),
                      to_dev(ent, dev), to_dev(dl, dev), logits.shape[1], L, res, T, eps, alpha)
    torch.cuda.synchronize()
    return tv.parse_result(res)


def test_typical_accept_random_vs_oracle(dev):
    b = tv.Bank(512, 0)
    g = synth.rng(21)
    T, eps, alpha = TYPICAL
    checked = 0
    for trial in range(240):
        n = int(g.integers(1, 65))
        if trial % 3 == 0:
            parent = synth.rank_product_tree(synth.BANK_BRANCHING, n)
        elif trial % 3 == 1:
            parent = synth.chain(n)
        else:
            parent = np.sort(synth.random_tree(g, n))
        parent = np.asarray(parent, np.int32)
        parent[0] = -1
        V = int(g.integers(3, 300))
        logits = g.standard_normal((n, V)) * float(g.uniform(0.2, 4.0))
        drafts = typical_drafts(3000 + trial, parent, logits, T, eps, alpha, p_likely=float(g.uniform(0.3, 1.0)))
        r = _typical_on_gpu(dev, b, parent, drafts, logits, T, eps, alpha, L=trial)
        k, path, bonus = oracle.typical_accept(parent, drafts, logits, T, eps, alpha)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
            k, path, bonus, trial + k, 0), trial
        checked += k > 1
    assert checked > 30  # many trials accept something beyond the root
    b.close()


def test_typical_accept_hand_and_limits(dev, bank):
    # two accepted depth-2 branches: the more likely one (larger index) wins
    parent = [-1, 0, 0, 1, 2]
    drafts = [0, 0, 1, 0, 0]
    z = np.zeros((5, 3))
    z[0] = [1.0, 1.2, -5.0]
    z[1] = [0.5, 0.0, 0.0]
    z[2] = [2.0, 0.0, 0.0]
    r = _typical_on_gpu(dev, bank, parent, drafts, z, 1.0, 0.09, 0.3)
    assert (r["accept_len"], r["path"], r["bonus_token"]) == (3, [0, 2, 4], 0)
    # an unreachable threshold accepts only the root
    g = synth.rng(22)
    parent = synth.bank_trees()[-1]
    z = g.standard_normal((64, 50))
    drafts = g.integers(0, 50, 64).astype(np.int32)
    r = _typical_on_gpu(dev, bank, parent, drafts, z, 0.7, 1.0, 1e9)
    assert (r["accept_len"], r["path"], r["bonus_token"]) == (1, [0], int(z[0].argmax()))
    # uniform logits accept every node: the deepest, smallest-id node (all likelihoods tie)
    r = _typical_on_gpu(dev, bank, parent, drafts, np.zeros((64, 50)), 0.7, 0.09, 0.3)
    k, path, bonus = oracle.typical_accept(parent, drafts, np.zeros((64, 50)), 0.7, 0.09, 0.3)
    assert (r["accept_len"], r["path"], r["bonus_token"]) == (k, path, bonus) and k == 6
    # duplicate sibling tokens tie exactly on both sides: the smaller id wins
    parent = [-1, 0, 0, 1, 2]
    z = np.zeros((5, 4))
    z[0] = [3.0, 0.0, 0.0, 0.0]
    r = _typical_on_gpu(dev, bank, parent, [0, 0, 0, 1, 1], z, 0.7, 0.09, 0.3)
    assert (r["accept_len"], r["path"]) == (3, [0, 1, 3])


def test_typical_accept_bad_token_status(dev, bank):
    z = np.zeros((3, 10))
    r = _typical_on_gpu(dev, bank, [-1, 0, 0], [0, 10, 3], z, 0.7, 0.09, 0.3)
    assert r["status"] == tv.TB_EINVAL and (r["accept_len"], r["path"]) == (2, [0, 2])


def test_typical_argument_errors(dev, bank):
    bid, _ = bank.add([-1, 0])
    i = torch.zeros(2, dtype=torch.int32, device=dev)
    f = torch.zeros(2, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    for T, eps, alpha in [(0.0, 0.09, 0.3), (-1.0, 0.09, 0.3), (float("nan"), 0.09, 0.3), (0.7, -0.1, 0.3),
                          (0.7, 0.09, float("inf"))]:
        with pytest.raises(tv.TreeVerifyError) as e:
            tv.typical_accept(bank, bid, i, i, f, f, f, 10, 0, res, T, eps, alpha)
        assert e.value.status == tv.TB_EINVAL
    h = torch.zeros((2, 64), dtype=torch.bfloat16, device=dev)
    W = torch.zeros((10, 64), dtype=torch.bfloat16, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(2, 0, 0, 0, 0, 10, 0), dev)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.lm_head_stats_typical(bank, bid, h, W, 0.0, i, i, f, f, f, f, f, ws)
    assert e.value.status == tv.TB_EINVAL


# ---------------------------------------------------------------- the full step

def _typical_case(seed, parent, L, n_layers, Hq, Hkv, d, D, V, T=TYPICAL[0]):
    parent = np.asarray(parent, np.int32)
    N = len(parent)
    L_cap = L + N + 3
    k, v = synth.gen_kv(seed, n_layers, Hkv, L_cap, d, L + N)
    q = synth.gen_q(seed, n_layers, N, Hq, d)
    W, hidden, am, t1, en, logits = _rows(seed, parent, D, V)
    drafts = typical_drafts(seed, parent, logits, T, *TYPICAL[1:])
    return dict(parent=parent, L=L, k=k, v=v, q=q, W=W, hidden=hidden, am=am, t1=t1, en=en, logits=logits,
                drafts=drafts)


@pytest.mark.parametrize("cfg", ["c1", "c2"])
def test_verify_step_typical_parity(dev, bank, cfg):
    sh = synth.SHAPES[cfg]()
    c = _typical_case(17, sh.parent, sh.L, sh.n_layers, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model,
                      sh.vocab)
    N, Hq, d = sh.N, sh.n_q_heads, sh.head_dim
    bid, _ = bank.add(c["parent"])
    kd, vd = to_dev(c["k"], dev), to_dev(c["v"], dev)
    kv = tv.KvCache(kd, vd, c["L"])
    out = torch.empty((sh.n_layers, N, Hq, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(N, dtype=torch.int32, device=dev)
    g_t1, g_en = _f32(N, dev), _f32(N, dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, sh.n_layers, sh.n_kv_heads, Hq, d, sh.vocab, 0), dev)
    tv.verify_step_typical(bank, bid, kv, to_dev(c["q"], dev), to_dev(c["hidden"], dev), to_dev(c["W"], dev),
                           to_dev(c["drafts"], dev), out, g_am, g_t1, g_en, res, ws, *TYPICAL)
    torch.cuda.synchronize()
    r = tv.parse_result(res)
    ref = oracle.tree_attention(c["q"][0], c["k"][0], c["v"][0], c["L"], c["parent"])
    check_attention(out[0].float().cpu().numpy(), ref)
    assert np.array_equal(g_am.cpu().numpy(), c["am"])
    assert np.abs(g_t1.cpu().numpy() - c["t1"]).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - c["en"]).max() <= STAT_TOL
    k, path, bonus = oracle.typical_accept(c["parent"], c["drafts"], c["logits"], *TYPICAL)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (k, path, bonus, c["L"] + k, 0)
    assert np.array_equal(bits(kd), oracle.kv_compact(c["k"], c["L"], path))
    assert np.array_equal(bits(vd), oracle.kv_compact(c["v"], c["L"], path))
    # the greedy entry point on the same inputs still follows the greedy rule
    kd2, vd2 = to_dev(c["k"], dev), to_dev(c["v"], dev)
    tv.verify_step(bank, bid, tv.KvCache(kd2, vd2, c["L"]), to_dev(c["q"], dev), to_dev(c["hidden"], dev),
                   to_dev(c["W"], dev), to_dev(c["drafts"], dev), out, g_am, g_t1, g_en, res, ws)
    torch.cuda.synchronize()
    kg, pg, bg = oracle.accept(c["parent"], c["drafts"], c["am"])
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"]) == (kg, pg, bg)


def test_verify_step_batched_typical(dev):
    """Ragged batch in typical mode: mixed trees, prefix lengths (incl. 0) and
    1-node trees; 300 LM-head rows so the head runs in two chunks and some
    sequences straddle the chunk boundary."""
    b = tv.Bank(32, 0)
    g = synth.rng(23)
    Hq, Hkv, d, D, V = 8, 2, 128, 256, 3000
    trees = synth.bank_trees()
    parents = [trees[-1], trees[0], trees[5], trees[-1], trees[6], trees[3], trees[-1], trees[-1]]
    Ls = [0, 40, 129, 7, 300, 1, 64, 200]
    W = synth.gen_lm_head(24, V, D)
    rows = sum(len(p) for p in parents)
    hidden, am, t1, en, logits = gap_filtered_hidden(25, rows, W, want_logits=True)
    seqs, host = [], []
    r0 = 0
    for i, (parent, L) in enumerate(zip(parents, Ls)):
        parent = np.asarray(parent, np.int32)
        N = len(parent)
        drafts = typical_drafts(600 + i, parent, logits[r0:r0 + N], *TYPICAL)
        k, v = synth.gen_kv(700 + i, 1, Hkv, L + N + 2, d, L + N)
        q = synth.gen_q(700 + i, 1, N, Hq, d)
        bid, _ = b.add(parent)
        s = tv.Seq(bid, tv.KvCache(to_dev(k, dev), to_dev(v, dev), L), to_dev(q, dev), to_dev(drafts, dev),
                   torch.empty((1, N, Hq, d), dtype=torch.bfloat16, device=dev), tv.make_result(dev))
        seqs.append(s)
        host.append((parent, L, k, v, q, drafts, r0))
        r0 += N
    g_am = torch.empty(rows, dtype=torch.int32, device=dev)
    g_t1, g_en = _f32(rows, dev), _f32(rows, dev)
    ws = tv.make_workspace(tv.tb_workspace_size(rows, 1, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_batched_typical(b, seqs, to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws, *TYPICAL)
    torch.cuda.synchronize()
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    for s, (parent, L, k, v, q, drafts, r0) in zip(seqs, host):
        N = len(parent)
        r = tv.parse_result(s.result)
        ka, path, bonus = oracle.typical_accept(parent, drafts, logits[r0:r0 + N], *TYPICAL)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        check_attention(s.attn_out[0].float().cpu().numpy(), oracle.tree_attention(q[0], k[0], v[0], L, parent))
        assert np.array_equal(bits(s.kv.k), oracle.kv_compact(k, L, path))
    b.close()


def test_batched_typical_many_edges_in_one_vocab_tile(dev):
    """16 sequences x 64 nodes whose drafts all fall in the first vocab tile:
    1008 gathers in one CTA, beyond its on-chip list, so the kernel rescans."""
    b = tv.Bank(4, 0)
    Hq, Hkv, d, D, V = 4, 4, 128, 128, 1000
    parent = np.asarray(synth.bank_trees()[-1], np.int32)
    bid, _ = b.add(parent)
    W = synth.gen_lm_head(26, V, D)
    hidden, am, t1, en, logits = gap_filtered_hidden(27, 16 * 64, W, want_logits=True)
    g = synth.rng(28)
    seqs, host = [], []
    for i in range(16):
        lg = logits[64 * i:64 * (i + 1)]
        for attempt in range(50):
            drafts = g.integers(0, 128, 64).astype(np.int32)
            close, tie = typical_ambiguity(parent, drafts, lg, *TYPICAL)
            if not close and not tie:
                break
        else:
            raise RuntimeError("no unambiguous draft set")
        k, v = synth.gen_kv(800 + i, 1, Hkv, 64 + 64, d, 64 + 64)
        q = synth.gen_q(800 + i, 1, 64, Hq, d)
        s = tv.Seq(bid, tv.KvCache(to_dev(k, dev), to_dev(v, dev), 64), to_dev(q, dev), to_dev(drafts, dev),
                   torch.empty((1, 64, Hq, d), dtype=torch.bfloat16, device=dev), tv.make_result(dev))
        seqs.append(s)
        host.append((drafts, lg))
    g_am = torch.empty(1024, dtype=torch.int32, device=dev)
    g_t1, g_en = _f32(1024, dev), _f32(1024, dev)
    ws = tv.make_workspace(tv.tb_workspace_size(1024, 1, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_batched_typical(b, seqs, to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws, *TYPICAL,
                                   flags=tv.TB_NO_COMPACT)
    torch.cuda.synchronize()
    for s, (drafts, lg) in zip(seqs, host):
        r = tv.parse_result(s.result)
        ka, path, bonus = oracle.typical_accept(parent, drafts, lg, *TYPICAL)
        assert (r["accept_len"], r["path"], r["bonus_token"]) == (ka, path, bonus)
    b.close()


@pytest.mark.parametrize("seed", range(16))
def test_random_typical_step(dev, seed):
    """Random shapes through verify_step_typical: random trees, prefix lengths
    0-2000, head_dim 64 and 128, GQA groups, one or two layers, vocabularies
    with ragged last tiles; attention within the derived bound of the fuzz
    tests, statistics, acceptance and compaction against the oracle."""
    g = synth.rng(7700 + seed)
    n = int(g.integers(1, 65))
    parent = np.sort(synth.random_tree(g, n))
    parent[0] = -1
    d = int(g.choice([64, 128]))
    Hkv = int(g.choice([1, 2, 4]))
    group = int(g.choice([1, 2, 4]))
    while n * group > 256:
        group //= 2
    Hq = Hkv * group
    L = int(g.choice([0, 5, 130, 700, 2000]))
    D = int(g.choice([64, 256]))
    V = int(g.choice([129, 1000, 3001]))
    layers = int(g.integers(1, 3))
    c = _typical_case(500 + seed, parent, L, layers, Hq, Hkv, d, D, V)
    b = tv.Bank(4, 0)
    bid, _ = b.add(c["parent"])
    kd, vd = to_dev(c["k"], dev), to_dev(c["v"], dev)
    out = torch.empty((layers, n, Hq, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(n, dtype=torch.int32, device=dev)
    g_t1, g_en = _f32(n, dev), _f32(n, dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(n, layers, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_typical(b, bid, tv.KvCache(kd, vd, L), to_dev(c["q"], dev), to_dev(c["hidden"], dev),
                           to_dev(c["W"], dev), to_dev(c["drafts"], dev), out, g_am, g_t1, g_en, res, ws, *TYPICAL)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy()
    for layer in range(layers):
        q, k, v = c["q"][layer], c["k"][layer], c["v"][layer]
        check_attention_fuzz(got[layer], oracle.tree_attention(q, k, v, L, parent),
                             oracle.tree_attention(q, k, abs_bits(v), L, parent), f"seed {seed} layer {layer}")
    assert np.array_equal(g_am.cpu().numpy(), c["am"])
    assert np.abs(g_t1.cpu().numpy() - c["t1"]).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - c["en"]).max() <= STAT_TOL
    k, path, bonus = oracle.typical_accept(c["parent"], c["drafts"], c["logits"], *TYPICAL)
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (k, path, bonus, L + k, 0)
    assert np.array_equal(bits(kd), oracle.kv_compact(c["k"], L, path))
    assert np.array_equal(bits(vd), oracle.kv_compact(c["v"], L, path))
    b.close()


@pytest.mark.parametrize("seed", range(8))
def test_random_batched_typical_step(dev, seed):
    """Random ragged batches in typical mode: 1-8 sequences with random trees
    and prefix lengths, head_dim 64 and 128, GQA groups, ragged vocabularies."""
    g = synth.rng(4400 + seed)
    d = int(g.choice([64, 128]))
    Hkv, group = int(g.choice([1, 2])), int(g.choice([1, 2, 4]))
    Hq = Hkv * group
    D, V = int(g.choice([64, 256])), int(g.choice([129, 1000, 3001]))
    batch = int(g.integers(1, 9))
    b = tv.Bank(16, 0)
    W = synth.gen_lm_head(seed, V, D)
    parents = []
    for i in range(batch):
        n = int(g.integers(1, 65))
        while n * group > 256:
            n //= 2
        p = np.sort(synth.random_tree(g, max(n, 1)))
        p[0] = -1
        parents.append(p)
    rows = sum(len(p) for p in parents)
    hidden, am, t1, en, logits = gap_filtered_hidden(seed + 50, rows, W, want_logits=True)
    seqs, host, r0 = [], [], 0
    for i, parent in enumerate(parents):
        N = len(parent)
        L = int(g.choice([0, 7, 130, 900]))
        drafts = typical_drafts(600 + 10 * seed + i, parent, logits[r0:r0 + N], *TYPICAL)
        k, v = synth.gen_kv(900 + 10 * seed + i, 1, Hkv, L + N + 2, d, L + N)
        q = synth.gen_q(900 + 10 * seed + i, 1, N, Hq, d)
        bid, _ = b.add(parent)
        s = tv.Seq(bid, tv.KvCache(to_dev(k, dev), to_dev(v, dev), L), to_dev(q, dev), to_dev(drafts, dev),
                   torch.empty((1, N, Hq, d), dtype=torch.bfloat16, device=dev), tv.make_result(dev))
        seqs.append(s)
        host.append((parent, L, k, v, q, drafts, r0))
        r0 += N
    g_am = torch.empty(rows, dtype=torch.int32, device=dev)
    g_t1, g_en = _f32(rows, dev), _f32(rows, dev)
    ws = tv.make_workspace(tv.tb_workspace_size(rows, 1, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_batched_typical(b, seqs, to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws, *TYPICAL)
    torch.cuda.synchronize()
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    for s, (parent, L, k, v, q, drafts, r0) in zip(seqs, host):
        N = len(parent)
        r = tv.parse_result(s.result)
        ka, path, bonus = oracle.typical_accept(parent, drafts, logits[r0:r0 + N], *TYPICAL)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        check_attention_fuzz(s.attn_out[0].float().cpu().numpy(), oracle.tree_attention(q[0], k[0], v[0], L, parent),
                             oracle.tree_attention(q[0], k[0], abs_bits(v[0]), L, parent), f"seed {seed}")
        assert np.array_equal(bits(s.kv.k), oracle.kv_compact(k, L, path))
    b.close()
