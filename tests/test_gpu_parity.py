"""GPU parity: every stage of the verification pass through the C ABI against
the fp64 oracle on the same seeded inputs.

Bit-exact: argmax, accept_len, path, bonus token, compacted KV bytes.
Attention: max-abs <= 1e-2 and mean-abs <= 1e-3.  top-1 / entropy: <= 1e-3 abs.
Hidden rows are drawn with an oracle top-2 logit gap > 1e-2.
"""
import zlib

import numpy as np
import pytest

import oracle
from helpers import ATT_MAX, STAT_TOL, bits, check_attention, gap_filtered_hidden, make_case, to_dev
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
    b = tv.Bank(256, 0)
    yield b
    b.close()


def _ws(dev, rows, d, V):
    return tv.make_workspace(tv.tb_workspace_size(rows, 1, 1, 1, d, V, 0), dev)


def _run_attention(bank, dev, parent, L, n_layers, Hq, Hkv, d, seed, layer_begin=0, n_run=None, L_cap=None):
    parent = np.asarray(parent, np.int32)
    N = len(parent)
    bid, order = bank.add(parent)
    assert np.array_equal(order, np.arange(N))
    L_cap = L + N + 5 if L_cap is None else L_cap
    k, v = synth.gen_kv(seed, n_layers, Hkv, L_cap, d, L + N)
    q = synth.gen_q(seed, n_layers, N, Hq, d)
    n_run = n_layers - layer_begin if n_run is None else n_run
    kv = tv.KvCache(to_dev(k, dev), to_dev(v, dev), L)
    qd = to_dev(q[layer_begin:layer_begin + n_run], dev)
    out = torch.full((n_run, N, Hq, d), float("nan"), dtype=torch.bfloat16, device=dev)
    ws = _ws(dev, 1, d, 1)
    tv.tree_attention(bank, bid, kv, qd, out, ws, layer_begin, n_run)
    torch.cuda.synchronize()
    assert tv.tb_workspace_status(ws) == 0
    got = out.float().cpu().numpy()
    for li in range(n_run):
        ref = oracle.tree_attention(q[layer_begin + li], k[layer_begin + li], v[layer_begin + li], L, parent)
        check_attention(got[li], ref, f"layer {layer_begin + li}")
    # the workspace counters are back at zero: a second call gives the same bytes
    out2 = torch.empty_like(out)
    tv.tree_attention(bank, bid, kv, qd, out2, ws, layer_begin, n_run)
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), out2.view(torch.int16))


ATTN_CASES = [
    # name, parent, L, layers, Hq, Hkv, d
    ("tiny-binary7", synth.full_tree((2, 2)), 128, 1, 4, 4, 64),
    ("decode-1node-L0", [-1], 0, 1, 2, 2, 128),
    ("decode-1node-L1000", [-1], 1000, 1, 4, 4, 128),
    ("chain64-ragged", synth.chain(64), 77, 1, 2, 2, 128),
    ("bank64-gqa4", synth.bank_trees()[-1], 300, 1, 8, 2, 128),
    ("tree26-L1024-h32", synth.shape_c2().parent, 1024, 1, 32, 32, 128),
    ("random63-L5-d64", np.sort(synth.random_tree(synth.rng(5), 63)), 5, 1, 4, 4, 64),
    ("two-nodes-L63", [-1, 0], 63, 1, 4, 1, 128),
    ("bank40-gqa4-d64", synth.bank_trees()[6], 190, 1, 8, 2, 64),
    ("bank64-gqa4-L2k", synth.bank_trees()[-1], 2048, 1, 32, 8, 128),
    ("chain2-L0", [-1, 0], 0, 1, 1, 1, 64),
    ("bank26-gqa8-d64", synth.bank_trees()[5], 700, 1, 16, 2, 64),      # 208 rows per kv head: two row blocks
    ("bank26-gqa8-d128", synth.bank_trees()[5], 700, 2, 16, 2, 128),
]


@pytest.mark.parametrize("name,parent,L,n_layers,Hq,Hkv,d", ATTN_CASES, ids=[c[0] for c in ATTN_CASES])
def test_tree_attention_parity(dev, bank, name, parent, L, n_layers, Hq, Hkv, d):
    _run_attention(bank, dev, parent, L, n_layers, Hq, Hkv, d, seed=zlib.crc32(name.encode()) % 1000)


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("L", [100, 250, 650, 800])
@pytest.mark.parametrize("parent,Hq,Hkv", [(synth.shape_c2().parent, 8, 2), (synth.bank_trees()[-1], 8, 2)],
                         ids=["tree26-gqa4", "tree64-gqa4-two-row-blocks"])
def test_tree_attention_whole_or_split_units(dev, bank, parent, Hq, Hkv, L, d):
    """Around the plan's whole-unit limit: units of 1-3, 6 and 7 key tiles
    ((L + N) / 128 rounded up), one or two 128-row blocks, both head widths.
    Up to six tiles a one-wave problem runs a whole unit per CTA; past that
    the tiles are split evenly and the split merge combines the pieces."""
    _run_attention(bank, dev, parent, L, 1, Hq, Hkv, d, seed=L + d + len(parent))


def test_tree_attention_non_bfs_input(dev, bank):
    """A topology given in non-breadth-first order is canonicalised; queries and
    tree K/V are then laid out in canonical order (order[c] = caller index)."""
    parent = synth.random_tree(synth.rng(9), 30)
    order, bfs_parent, _, _ = tv.tb_canonicalize(parent)
    assert not np.array_equal(order, np.arange(30))
    _run_attention(bank, dev, bfs_parent, 70, 1, 4, 4, 128, seed=9)


def test_tree_attention_layer_subset(dev, bank):
    _run_attention(bank, dev, synth.bank_trees()[4], 200, 4, 4, 4, 128, seed=3, layer_begin=1, n_run=2)


def test_tree_attention_large_L_multilayer(dev, bank):
    _run_attention(bank, dev, synth.bank_trees()[-1], 5000, 3, 8, 8, 128, seed=4)


LM_CASES = [(1, 256, 1000), (7, 256, 1000), (26, 4096, 4099), (64, 4096, 32000), (200, 512, 3000), (256, 256, 129),
            (232, 256, 4099),
            # several vocab tiles per persistent CTA (both TMEM accumulators reused), two CTAs
            # per SM for narrow rows and one for wide rows, ragged last tiles
            (26, 256, 128256), (232, 64, 60001), (100, 128, 50001)]


@pytest.mark.parametrize("R,D,V", LM_CASES)
def test_lm_head_parity(dev, R, D, V):
    W = synth.gen_lm_head(R + D + V, V, D)
    hidden, am, t1, en = gap_filtered_hidden(R * 7 + V, R, W)
    g_am = torch.full((R,), -1, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(R, dtype=torch.float32, device=dev)
    g_en = torch.empty(R, dtype=torch.float32, device=dev)
    ws = _ws(dev, R, 0, V)
    tv.lm_head_stats(to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws)
    torch.cuda.synchronize()
    assert tv.tb_workspace_status(ws) == 0
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_t1.cpu().numpy() - t1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    en_g = g_en.cpu().numpy()
    assert np.all(en_g >= -STAT_TOL) and np.all(en_g <= np.log(V) + STAT_TOL)
    # repeat with the same workspace: counters were reset
    g_am2 = torch.full((R,), -1, dtype=torch.int32, device=dev)
    tv.lm_head_stats(to_dev(hidden, dev), to_dev(W, dev), g_am2, g_t1, g_en, ws)
    torch.cuda.synchronize()
    assert torch.equal(g_am, g_am2)


def test_lm_head_uniform_logits(dev):
    R, D, V = 5, 64, 1300
    W = np.zeros((V, D), np.uint16)
    hidden = synth.normal_bf16(synth.rng(1), (R, D))
    g_am = torch.empty(R, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(R, dtype=torch.float32, device=dev)
    g_en = torch.empty(R, dtype=torch.float32, device=dev)
    ws = _ws(dev, R, 0, V)
    tv.lm_head_stats(to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws)
    torch.cuda.synchronize()
    assert g_am.cpu().tolist() == [0] * R  # every logit ties: lowest index
    assert np.allclose(g_en.cpu().numpy(), np.log(V), atol=STAT_TOL)
    assert np.allclose(g_t1.cpu().numpy(), 1.0 / V, atol=1e-6)


def _accept_on_gpu(dev, bank, parent, draft, argmax, vocab, L=0):
    bid, _ = bank.add(parent)
    res = tv.make_result(dev)
    tv.greedy_accept(bank, bid, to_dev(np.asarray(draft, np.int32), dev), to_dev(np.asarray(argmax, np.int32), dev),
                     vocab, L, res)
    torch.cuda.synchronize()
    return tv.parse_result(res)


def test_greedy_accept_hand_cases(dev, bank):
    import json
    import os

    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "hand_examples.json")))["acceptance_cases"]
    for c in g["cases"]:
        r = _accept_on_gpu(dev, bank, g["parent"], c["draft"], c["argmax"], 100, L=10)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
            c["accept_len"], c["path"], c["bonus"], 10 + c["accept_len"], 0), c["why"]


def test_greedy_accept_random_vs_oracle(dev):
    b = tv.Bank(512, 0)
    g = synth.rng(11)
    for trial in range(300):
        n = int(g.integers(1, 65))
        parent = synth.rank_product_tree(synth.BANK_BRANCHING, n) if trial % 2 else np.sort(
            synth.random_tree(g, n))  # sorted parents of a parent[i]<i tree: breadth-first order
        parent[0] = -1
        V = int(g.integers(2, 5))
        draft = g.integers(0, V, size=n).astype(np.int32)
        argmax = g.integers(0, V, size=n).astype(np.int32)
        r = _accept_on_gpu(dev, b, parent, draft, argmax, V, L=trial)
        k, path, bonus = oracle.accept(parent, draft, argmax)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"]) == (k, path, bonus, trial + k)
    b.close()


def test_greedy_accept_bad_token_status(dev, bank):
    r = _accept_on_gpu(dev, bank, [-1, 0, 0], [0, 5, 1000], [5, 1, 2], 1000)
    assert r["status"] == tv.TB_EINVAL and r["accept_len"] == 2 and r["path"] == [0, 1]


def test_kv_compact_vs_oracle(dev, bank):
    g = synth.rng(12)
    n_layers, H, d, L = 3, 4, 128, 50
    parent = synth.bank_trees()[-1]
    N = len(parent)
    k, v = synth.gen_kv(12, n_layers, H, L + N + 7, d, L + N)
    for trial in range(6):
        draft = g.integers(0, 3, size=N).astype(np.int32)
        argmax = g.integers(0, 3, size=N).astype(np.int32)
        kd, vd = to_dev(k, dev), to_dev(v, dev)
        kv = tv.KvCache(kd, vd, L)
        bid, _ = bank.add(parent)
        res = tv.make_result(dev)
        tv.greedy_accept(bank, bid, to_dev(draft, dev), to_dev(argmax, dev), 3, L, res)
        tv.kv_compact(kv, res)
        torch.cuda.synchronize()
        ka, path, _ = oracle.accept(parent, draft, argmax)
        assert tv.parse_result(res)["path"] == path
        assert np.array_equal(bits(kd), oracle.kv_compact(k, L, path))
        assert np.array_equal(bits(vd), oracle.kv_compact(v, L, path))


def test_kv_compact_from_path_arrays(dev, bank):
    """kv_compact from a caller's device path (exactly accept_len entries) and a
    device accept_len, as the boundary declares it: accepted paths of random
    drafts, the identity path and the root alone."""
    g = synth.rng(13)
    n_layers, H, d, L = 2, 4, 64, 33
    parent = synth.bank_trees()[-1]
    N = len(parent)
    k, v = synth.gen_kv(13, n_layers, H, L + N + 5, d, L + N)
    paths = []
    for trial in range(4):
        draft = g.integers(0, 3, size=N).astype(np.int32)
        argmax = g.integers(0, 3, size=N).astype(np.int32)
        paths.append(oracle.accept(parent, draft, argmax)[1])
    paths += [[0, 1, 2, 3], [0]]
    for path in paths:
        kd, vd = to_dev(k, dev), to_dev(v, dev)
        tv.kv_compact_path(tv.KvCache(kd, vd, L), to_dev(np.asarray(path, np.int32), dev),
                           to_dev(np.asarray([len(path)], np.int32), dev))
        torch.cuda.synchronize()
        assert np.array_equal(bits(kd), oracle.kv_compact(k, L, path)), path
        assert np.array_equal(bits(vd), oracle.kv_compact(v, L, path)), path


def test_attention_units_counted_without_overflow(dev, bank):
    """A cache whose layer x kv-head count is far beyond any real one (2^30
    units, past the 32-bit counts of the plan) is refused before anything is
    enqueued."""
    import ctypes

    bid, _ = bank.add([-1, 0])
    k = torch.zeros((1, 1, 64, 128), dtype=torch.bfloat16, device=dev)
    c = tv.TbKv(k.data_ptr(), k.data_ptr(), (1 << 10) * 64 * 128, 64 * 128, 1 << 20, 1 << 10, 128, 0, 64, 0.0)
    q = torch.zeros((1, 2, 1024, 128), dtype=torch.bfloat16, device=dev)
    ws = tv.make_workspace(1 << 20, dev)
    st = tv.load().tree_attention(bank.handle, bid, ctypes.byref(c), 0, 1 << 20, q.data_ptr(), 1024, q.data_ptr(),
                                  ws.data_ptr(), ws.numel(), None)
    assert st == tv.TB_EUNSUPPORTED
    assert b"attention units" in tv.load().tb_last_error()


def test_kv_compact_skips_invalid_path_entries(dev):
    """Entries the header declares untouched: path[j] <= j (the copy would go
    backwards) and a source slot at or past L_cap; the valid entry between
    them is still applied."""
    n_layers, H, d, L = 1, 2, 128, 20
    L_cap = L + 10
    k, v = synth.gen_kv(14, n_layers, H, L_cap, d, L_cap)
    path = [0, 0, 5, 1, L_cap - L + 3]
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    tv.kv_compact_path(tv.KvCache(kd, vd, L), to_dev(np.asarray(path, np.int32), dev),
                       to_dev(np.asarray([len(path)], np.int32), dev))
    torch.cuda.synchronize()
    want_k, want_v = k.copy(), v.copy()
    want_k[:, :, L + 2] = k[:, :, L + 5]  # the one valid move: slot L + 2 <- L + 5
    want_v[:, :, L + 2] = v[:, :, L + 5]
    assert np.array_equal(bits(kd), want_k)
    assert np.array_equal(bits(vd), want_v)


def _full_step(dev, bank, case, Hq, Hkv, d, flags=0):
    bid, _ = bank.add(case.parent)
    N, V, D = case.N, case.W.shape[0], case.W.shape[1]
    n_layers = case.k.shape[0]
    kd, vd = to_dev(case.k, dev), to_dev(case.v, dev)
    kv = tv.KvCache(kd, vd, case.L)
    out = torch.empty((n_layers, N, Hq, d), dtype=torch.bfloat16, device=dev)
    g_am = torch.empty(N, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
    g_en = torch.empty(N, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, n_layers, Hkv, Hq, d, V, 0), dev)
    tv.verify_step(bank, bid, kv, to_dev(case.q, dev), to_dev(case.hidden, dev), to_dev(case.W, dev),
                   to_dev(case.drafts.astype(np.int32), dev), out, g_am, g_t1, g_en, res, ws, flags)
    torch.cuda.synchronize()
    return out, g_am, g_t1, g_en, tv.parse_result(res), kd, vd


@pytest.mark.parametrize("cfg", ["c1", "c2"])
def test_verify_step_full_parity(dev, bank, cfg):
    sh = synth.SHAPES[cfg]()
    case = make_case(7, sh.parent, sh.L, sh.n_layers, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model,
                     sh.vocab, sh.p_match)
    out, g_am, g_t1, g_en, r, kd, vd = _full_step(dev, bank, case, sh.n_q_heads, sh.n_kv_heads, sh.head_dim)
    ref = oracle.tree_attention(case.q[0], case.k[0], case.v[0], case.L, case.parent)
    check_attention(out[0].float().cpu().numpy(), ref)
    assert np.array_equal(g_am.cpu().numpy(), case.argmax)
    assert np.abs(g_t1.cpu().numpy() - case.top1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - case.entropy).max() <= STAT_TOL
    k, path, bonus = oracle.accept(case.parent, case.drafts, case.argmax)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (k, path, bonus, case.L + k, 0)
    assert np.array_equal(bits(kd), oracle.kv_compact(case.k, case.L, path))
    assert np.array_equal(bits(vd), oracle.kv_compact(case.v, case.L, path))


# Steps whose LM head is longer than their attention: the attention grid is then
# capped at the SMs the LM head's CTAs leave free, so that both start at once.
# On a 152-SM GB300 these shapes get: 73 attention CTAs over 136 tiles (units
# of 17 tiles spread over several CTAs); 27 over 160 (units of 40 tiles); 27
# over 64 (units of 2 tiles); 54 over 128 across two layers with GQA group 4.
BESIDE_LM = [
    # parent, L, layers, Hq, Hkv, D, V
    (synth.shape_c2().parent, 2048, 1, 8, 8, 4096, 20000),
    (synth.bank_trees()[6], 5000, 1, 8, 4, 4096, 32000),
    (synth.bank_trees()[-1], 100, 1, 32, 32, 4096, 32000),
    (synth.chain(17), 1000, 2, 32, 8, 2048, 25000),
]


@pytest.mark.parametrize("parent,L,layers,Hq,Hkv,D,V", BESIDE_LM)
def test_verify_step_beside_lm_head(dev, bank, parent, L, layers, Hq, Hkv, D, V):
    case = make_case(11, parent, L, layers, Hq, Hkv, 128, D, V, 0.7)
    out, g_am, g_t1, g_en, r, kd, vd = _full_step(dev, bank, case, Hq, Hkv, 128)
    got = out.float().cpu().numpy()
    for layer in range(layers):
        check_attention(got[layer], oracle.tree_attention(case.q[layer], case.k[layer], case.v[layer], L, case.parent),
                        f"layer {layer}")
    assert np.array_equal(g_am.cpu().numpy(), case.argmax)
    assert np.abs(g_t1.cpu().numpy() - case.top1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - case.entropy).max() <= STAT_TOL
    k, path, bonus = oracle.accept(case.parent, case.drafts, case.argmax)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (k, path, bonus, L + k, 0)
    assert np.array_equal(bits(kd), oracle.kv_compact(case.k, L, path))
    assert np.array_equal(bits(vd), oracle.kv_compact(case.v, L, path))


def test_verify_step_no_compact_flag(dev, bank):
    sh = synth.shape_c1()
    case = make_case(9, sh.parent, sh.L, 1, 4, 4, 64, 256, 1000, 1.0)  # every draft matches
    *_, r, kd, vd = _full_step(dev, bank, case, 4, 4, 64, flags=tv.TB_NO_COMPACT)
    assert r["accept_len"] == 3
    assert np.array_equal(bits(kd), case.k)


def test_bank_switching_loop(dev):
    """Several steps over the bank with a growing L: each step matches the oracle."""
    b = tv.Bank(16, 0)
    trees = synth.bank_trees()
    ids = [b.add(t)[0] for t in trees]
    H, d, D, V, L0 = 4, 128, 256, 2000, 100
    L_cap = L0 + 6 * 64 + 64
    k, v = synth.gen_kv(21, 1, H, L_cap, d, L_cap)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    W = synth.gen_lm_head(21, V, D)
    Wd = to_dev(W, dev)
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, H, H, d, V, 0), dev)
    L = L0
    kh, vh = k.copy(), v.copy()
    for step, tix in enumerate([7, 3, 0, 5, 7, 1, 6]):
        parent = trees[tix]
        N = len(parent)
        q = synth.gen_q(100 + step, 1, N, H, d)
        hidden, am, t1, en = gap_filtered_hidden(100 + step, N, W)
        drafts = synth.gen_drafts(100 + step, parent, am, V, 0.8)
        out = torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev)
        g_am = torch.empty(N, dtype=torch.int32, device=dev)
        g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
        g_en = torch.empty(N, dtype=torch.float32, device=dev)
        res = tv.make_result(dev)
        kv = tv.KvCache(kd, vd, L)
        tv.verify_step(b, ids[tix], kv, to_dev(q, dev), to_dev(hidden, dev), Wd, to_dev(drafts, dev), out, g_am,
                       g_t1, g_en, res, ws)
        torch.cuda.synchronize()
        r = tv.parse_result(res)
        ref = oracle.tree_attention(q[0], kh[0], vh[0], L, parent)
        check_attention(out[0].float().cpu().numpy(), ref, f"step {step}")
        assert np.array_equal(g_am.cpu().numpy(), am)
        ka, path, bonus = oracle.accept(parent, drafts, am)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"]) == (ka, path, bonus, L + ka)
        kh, vh = oracle.kv_compact(kh, L, path), oracle.kv_compact(vh, L, path)
        assert np.array_equal(bits(kd), kh) and np.array_equal(bits(vd), vh)
        L = r["new_L"]
    b.close()


# ------------------------------------------------------------------ host validation through the ABI


def test_argument_errors(dev, bank):
    bid, _ = bank.add(synth.full_tree((2, 2)))
    k = torch.zeros((1, 2, 20, 64), dtype=torch.bfloat16, device=dev)
    q = torch.zeros((1, 7, 2, 64), dtype=torch.bfloat16, device=dev)
    out = torch.empty_like(q)
    ws = _ws(dev, 8, 64, 100)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tree_attention(bank, 999, tv.KvCache(k, k, 0), q, out, ws)
    assert e.value.status == tv.TB_ENOTFOUND
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tree_attention(bank, bid, tv.KvCache(k, k, 14), q, out, ws)  # 14 + 7 > 20
    assert e.value.status == tv.TB_ECAPACITY
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tree_attention(bank, bid, tv.KvCache(k, k, 0), q, out, ws[:1000])
    assert e.value.status == tv.TB_ECAPACITY
    q3 = torch.zeros((1, 7, 3, 64), dtype=torch.bfloat16, device=dev)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tree_attention(bank, bid, tv.KvCache(k, k, 0), q3, torch.empty_like(q3), ws)
    assert e.value.status == tv.TB_EINVAL
    k96 = torch.zeros((1, 2, 20, 96), dtype=torch.bfloat16, device=dev)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.tree_attention(bank, bid, tv.KvCache(k96, k96, 0), q, out, ws)
    assert e.value.status == tv.TB_EUNSUPPORTED
    h = torch.zeros((300, 64), dtype=torch.bfloat16, device=dev)
    W = torch.zeros((100, 64), dtype=torch.bfloat16, device=dev)
    o = torch.empty(300, dtype=torch.int32, device=dev)
    f = torch.empty(300, dtype=torch.float32, device=dev)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.lm_head_stats(h, W, o, f, f, ws)
    assert e.value.status == tv.TB_EUNSUPPORTED


def test_c4_full_size_sampled(dev):
    """The long-context workload at full size, in the launch configuration the
    benchmark times: 32 layers x 32 heads x 128, L=16384, 64-node tree, V=32000.
    Attention is compared on sampled (layer, head) pairs; LM-head stats,
    acceptance and the compacted tree region of every layer/head exactly."""
    sh = synth.shape_c4()
    N, L, H, d, D, V, nl = sh.N, sh.L, sh.n_q_heads, sh.head_dim, sh.d_model, sh.vocab, sh.n_layers
    b = tv.Bank(4, 0)
    bid, _ = b.add(sh.parent)
    bf = torch.bfloat16
    k = synth.device_normal_bf16_(torch.empty((nl, H, sh.L_cap, d), dtype=bf, device=dev), 41)
    v = synth.device_normal_bf16_(torch.empty((nl, H, sh.L_cap, d), dtype=bf, device=dev), 42)
    q = synth.device_normal_bf16_(torch.empty((nl, N, H, d), dtype=bf, device=dev), 43)
    W = synth.gen_lm_head(44, V, D)
    hidden, am, t1, en = gap_filtered_hidden(45, N, W)
    drafts = synth.gen_drafts(46, sh.parent, am, V, sh.p_match)
    samples = [(0, 0), (13, 7), (nl - 1, H - 1)]
    pre = {s: (bits(k[s[0], s[1], :L + N]), bits(v[s[0], s[1], :L + N])) for s in samples}
    tree_k, tree_v = bits(k[:, :, L:L + N]), bits(v[:, :, L:L + N])
    q_h = bits(q)
    kv = tv.KvCache(k, v, L)
    out = torch.empty((nl, N, H, d), dtype=bf, device=dev)
    g_am = torch.empty(N, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
    g_en = torch.empty(N, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, nl, H, H, d, V, 0), dev)
    tv.verify_step(b, bid, kv, q, to_dev(hidden, dev), to_dev(W, dev), to_dev(drafts, dev), out, g_am, g_t1, g_en,
                   res, ws)
    torch.cuda.synchronize()
    r = tv.parse_result(res)
    assert r["status"] == 0
    got = out.float().cpu().numpy()
    for layer, head in samples:
        kk, vv = pre[(layer, head)]
        ref = oracle.tree_attention(q_h[layer][:, head:head + 1], kk[None], vv[None], L, sh.parent)
        check_attention(got[layer][:, head:head + 1], ref, f"layer {layer} head {head}")
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_t1.cpu().numpy() - t1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    ka, path, bonus = oracle.accept(sh.parent, drafts, am)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"]) == (ka, path, bonus, L + ka)
    assert np.array_equal(bits(k[:, :, L:L + N]), oracle.kv_compact(tree_k, 0, path))
    assert np.array_equal(bits(v[:, :, L:L + N]), oracle.kv_compact(tree_v, 0, path))
    for layer, head in samples:  # the prefix is untouched
        assert np.array_equal(bits(k[layer, head, :L]), pre[(layer, head)][0][:L])
    b.close()
