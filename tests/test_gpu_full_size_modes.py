"""The long-context step at full size (32 layers x 32 heads x 128, L = 16384,
64-node tree, V = 32000; the benchmark's launch configuration) with typical
acceptance, with the rotary embedding applied by the library, and with
speculative sampling and the rotary embedding together.

Attention is compared with the fp64 oracle on sampled (layer, head) pairs;
the LM-head statistics, the acceptance and the compacted tree region of every
layer and head exactly (the rotated tree keys within one bf16 ulp).
"""
import numpy as np
import pytest

import oracle
from helpers import (STAT_TOL, TYPICAL, bits, check_attention, draw_decidable_walk, gap_filtered_hidden,
                     softmax_rows, to_dev, typical_drafts)
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
def full(dev):
    sh = synth.shape_c4()
    N, L, H, d, nl, D, V = sh.N, sh.L, sh.n_q_heads, sh.head_dim, sh.n_layers, sh.d_model, sh.vocab
    W = synth.gen_lm_head(54, V, D)
    hidden, am, t1, en, logits = gap_filtered_hidden(55, N, W, want_logits=True)
    return dict(sh=sh, N=N, L=L, H=H, d=d, nl=nl, D=D, V=V, W=W, hidden=hidden, am=am, t1=t1, en=en, logits=logits)


def _cache(dev, f, seed):
    bf = torch.bfloat16
    k = synth.device_normal_bf16_(torch.empty((f["nl"], f["H"], f["sh"].L_cap, f["d"]), dtype=bf, device=dev), seed)
    v = synth.device_normal_bf16_(torch.empty((f["nl"], f["H"], f["sh"].L_cap, f["d"]), dtype=bf, device=dev), seed + 1)
    q = synth.device_normal_bf16_(torch.empty((f["nl"], f["N"], f["H"], f["d"]), dtype=bf, device=dev), seed + 2)
    return k, v, q


def _outs(dev, f):
    N = f["N"]
    return (torch.empty((f["nl"], N, f["H"], f["d"]), dtype=torch.bfloat16, device=dev),
            torch.empty(N, dtype=torch.int32, device=dev), torch.empty(N, dtype=torch.float32, device=dev),
            torch.empty(N, dtype=torch.float32, device=dev), tv.make_result(dev),
            tv.make_workspace(tv.tb_workspace_size(N, f["nl"], f["H"], f["H"], f["d"], f["V"], 0), dev))


SAMPLES = [(0, 0), (17, 9), (31, 31)]


def test_full_size_typical(dev, full):
    f = full
    parent = np.asarray(f["sh"].parent, np.int32)
    N, L = f["N"], f["L"]
    b = tv.Bank(4, 0)
    bid, _ = b.add(parent)
    k, v, q = _cache(dev, f, 61)
    drafts = typical_drafts(62, parent, f["logits"], *TYPICAL)
    pre = {s: (bits(k[s[0], s[1], :L + N]), bits(v[s[0], s[1], :L + N])) for s in SAMPLES}
    tree_k, tree_v = bits(k[:, :, L:L + N]), bits(v[:, :, L:L + N])
    q_h = bits(q)
    out, g_am, g_t1, g_en, res, ws = _outs(dev, f)
    tv.verify_step_typical(b, bid, tv.KvCache(k, v, L), q, to_dev(f["hidden"], dev), to_dev(f["W"], dev),
                           to_dev(drafts, dev), out, g_am, g_t1, g_en, res, ws, *TYPICAL)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy()
    for layer, head in SAMPLES:
        kk, vv = pre[(layer, head)]
        ref = oracle.tree_attention(q_h[layer][:, head:head + 1], kk[None], vv[None], L, parent)
        check_attention(got[layer][:, head:head + 1], ref, f"layer {layer} head {head}")
    assert np.array_equal(g_am.cpu().numpy(), f["am"])
    assert np.abs(g_t1.cpu().numpy() - f["t1"]).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - f["en"]).max() <= STAT_TOL
    ka, path, bonus = oracle.typical_accept(parent, drafts, f["logits"], *TYPICAL)
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
    assert np.array_equal(bits(k[:, :, L:L + N]), oracle.kv_compact(tree_k, 0, path))
    assert np.array_equal(bits(v[:, :, L:L + N]), oracle.kv_compact(tree_v, 0, path))
    b.close()


def _ordered(x):
    x = x.astype(np.int32)
    return np.where(x & 0x8000, 0x8000 - x, x)


def test_full_size_rope(dev, full):
    f = full
    parent = np.asarray(f["sh"].parent, np.int32)
    N, L = f["N"], f["L"]
    b = tv.Bank(4, 0)
    bid, _ = b.add(parent)
    k, v, q = _cache(dev, f, 71)
    drafts = synth.gen_drafts(72, parent, f["am"], f["V"], f["sh"].p_match)
    pre = {s: (bits(k[s[0], s[1], :L + N]), bits(v[s[0], s[1], :L + N])) for s in SAMPLES}
    tree_v = bits(v[:, :, L:L + N])
    q_h = bits(q)
    out, g_am, g_t1, g_en, res, ws = _outs(dev, f)
    tv.verify_step(b, bid, tv.KvCache(k, v, L, rope_theta=10000.0), q, to_dev(f["hidden"], dev), to_dev(f["W"], dev),
                   to_dev(drafts, dev), out, g_am, g_t1, g_en, res, ws)
    torch.cuda.synchronize()
    ka, path, bonus = oracle.accept(parent, drafts, f["am"])
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
    got = out.float().cpu().numpy()
    for layer, head in SAMPLES:
        kk, vv = pre[(layer, head)]
        ref, k_rot = oracle.tree_attention_rope(q_h[layer][:, head:head + 1], kk[None], vv[None], L, parent)
        check_attention(got[layer][:, head:head + 1], ref, f"layer {layer} head {head}")
        # the cache holds the rotated tree keys, compacted along the accepted path
        want = oracle.kv_compact(k_rot[0][None], 0, path)[0]
        gk = bits(k[layer, head, :L + N])
        diff = np.abs(_ordered(gk[L:L + N]) - _ordered(want))
        assert diff.max() <= 1 and (diff > 0).mean() < 0.01
        assert np.array_equal(gk[:L], kk[:L])
    assert np.array_equal(bits(v[:, :, L:L + N]), oracle.kv_compact(tree_v, 0, path))
    b.close()


def test_full_size_sampled_rope(dev, full):
    """The walk of speculative sampling (8-CTA cluster kernel) after attention with
    the rotary embedding and the LM head writing every logit row: the launch of
    `bench.py --accept sampled --rope`.  Drafts from a draft distribution that
    mostly agrees with the target, uniforms that keep every decision decidable."""
    f = full
    parent = np.asarray(f["sh"].parent, np.int32)
    N, L, V = f["N"], f["L"], f["V"]
    T = 0.7
    g = synth.rng(82)
    qd = softmax_rows(f["logits"] / T * 1.3 + g.standard_normal((N, V)) * 0.5, 1.0)
    qd = (qd / qd.sum(axis=1, keepdims=True)).astype(np.float32).astype(np.float64)
    draft, unif, want = draw_decidable_walk(g, parent, f["logits"], qd, T)
    b = tv.Bank(4, 0)
    bid, _ = b.add(parent)
    k, v, q = _cache(dev, f, 81)
    pre = {s: (bits(k[s[0], s[1], :L + N]), bits(v[s[0], s[1], :L + N])) for s in SAMPLES}
    tree_v = bits(v[:, :, L:L + N])
    q_h = bits(q)
    out, g_am, g_t1, g_en, res, ws = _outs(dev, f)
    lg = torch.full((N + 1, V), float("nan"), dtype=torch.float32, device=dev)
    tv.verify_step_sampled(b, bid, tv.KvCache(k, v, L, rope_theta=10000.0), q, to_dev(f["hidden"], dev),
                           to_dev(f["W"], dev), to_dev(draft, dev), to_dev(qd.astype(np.float32), dev),
                           to_dev(unif.astype(np.float32), dev), T, out, g_am, g_t1, g_en, lg, res, ws)
    torch.cuda.synchronize()
    r = tv.parse_result(res)
    assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (
        want[0], want[1], want[2], L + want[0], 0)
    assert np.array_equal(g_am.cpu().numpy(), f["am"])
    assert np.abs(g_en.cpu().numpy() - f["en"]).max() <= STAT_TOL
    assert np.abs(lg[:N].cpu().numpy() - f["logits"]).max() <= 1e-3
    got = out.float().cpu().numpy()
    path = want[1]
    for layer, head in SAMPLES:
        kk, vv = pre[(layer, head)]
        ref, k_rot = oracle.tree_attention_rope(q_h[layer][:, head:head + 1], kk[None], vv[None], L, parent)
        check_attention(got[layer][:, head:head + 1], ref, f"layer {layer} head {head}")
        want_k = oracle.kv_compact(k_rot[0][None], 0, path)[0]
        gk = bits(k[layer, head, :L + N])
        diff = np.abs(_ordered(gk[L:L + N]) - _ordered(want_k))
        assert diff.max() <= 1 and (diff > 0).mean() < 0.01
        assert np.array_equal(gk[:L], kk[:L])
    assert np.array_equal(bits(v[:, :, L:L + N]), oracle.kv_compact(tree_v, 0, path))
    b.close()
