"""Pins for the oracle's rotary embedding and RoPE tree attention.

The rotation is tied to its defining properties (identity at position 0,
pair norms preserved, q.k depending only on the position difference) and to
closed forms for d = 2 and d = 4; the tree path is tied to torch's float64
scaled_dot_product_attention with a networkx ancestor mask, with every token
placed at L + depth (the TopologyBank's position offsets).
"""
import math

import networkx as nx
import numpy as np
import pytest
import torch

import oracle
from paper_2606_27550_gb300 import synth


def _bf(x):
    return synth.to_bf16_bits(np.asarray(x, dtype=np.float32))


def _f(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def test_rope_identity_at_position_zero():
    x = synth.normal_bf16(synth.rng(1), (5, 128))
    np.testing.assert_array_equal(oracle.rope(x, np.zeros(5, np.int32)), _f(x))


def test_rope_preserves_pair_norms():
    x = synth.normal_bf16(synth.rng(2), (7, 64))
    pos = np.array([1, 5, 77, 1000, 4095, 16384, 65000], np.int32)
    y = oracle.rope(x, pos)
    xf = _f(x)
    np.testing.assert_allclose(np.hypot(y[:, :32], y[:, 32:]), np.hypot(xf[:, :32], xf[:, 32:]), rtol=1e-12)


@pytest.mark.parametrize("m,n,s", [(0, 5, 3), (100, 7, 1000), (16000, 16384, 17)])
def test_rope_scores_depend_on_position_difference(m, n, s):
    g = synth.rng(3)
    a = synth.normal_bf16(g, (1, 128))
    b = synth.normal_bf16(g, (1, 128))
    d1 = oracle.rope(a, [m]) @ oracle.rope(b, [n]).T
    d2 = oracle.rope(a, [m + s]) @ oracle.rope(b, [n + s]).T
    assert d1[0, 0] == pytest.approx(d2[0, 0], rel=1e-9, abs=1e-9)


def test_rope_closed_forms():
    # d = 2: theta_0 = 1, a plain rotation by the position
    x = _bf([[1.0, 0.5]])
    for p in (1, 2, 100):
        y = oracle.rope(x, [p])
        assert y[0, 0] == pytest.approx(math.cos(p) - 0.5 * math.sin(p), abs=1e-14)
        assert y[0, 1] == pytest.approx(0.5 * math.cos(p) + math.sin(p), abs=1e-14)
    # d = 4, base 100: theta = (1, 100^(-1/2) = 0.1); pairs (0, 2) and (1, 3)
    x = _bf([[1.0, 2.0, 0.0, 0.0]])
    y = oracle.rope(x, [3], base=100.0)
    np.testing.assert_allclose(y[0], [math.cos(3), 2 * math.cos(0.3), math.sin(3), 2 * math.sin(0.3)], atol=1e-14)


def _sdpa_rope_reference(q, k, v, L, parent, base=10000.0):
    """torch float64 SDPA: tokens at L + depth, tree keys rotated then rounded to bf16,
    mask from networkx ancestors."""
    N, Hq, d = q.shape
    Hkv = k.shape[0]
    g = nx.DiGraph()
    g.add_nodes_from(range(N))
    g.add_edges_from((int(p), i) for i, p in enumerate(parent) if p >= 0)
    depth = [nx.shortest_path_length(g, 0, i) for i in range(N)]
    pos = np.array([L + dd for dd in depth], np.int32)
    mask = torch.zeros(N, L + N, dtype=torch.bool)
    mask[:, :L] = True
    for i in range(N):
        for j in nx.ancestors(g, i) | {i}:
            mask[i, L + j] = True
    qr = np.stack([oracle.rope(q[:, h], pos, base) for h in range(Hq)], 1)      # [N][Hq][d]
    kr = np.stack([_f(_bf(oracle.rope(k[h, L:L + N], pos, base))) for h in range(Hkv)])  # rounded to bf16
    kk = np.concatenate([_f(k[:, :L]), kr], 1)
    vv = _f(v[:, :L + N])
    qt = torch.from_numpy(qr).permute(1, 0, 2).unsqueeze(0)
    kt = torch.from_numpy(kk).unsqueeze(0).repeat_interleave(Hq // Hkv, 1)
    vt = torch.from_numpy(vv).unsqueeze(0).repeat_interleave(Hq // Hkv, 1)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
    return o[0].permute(1, 0, 2).numpy(), np.stack([_bf(oracle.rope(k[h, L:L + N], pos, base)) for h in range(Hkv)])


@pytest.mark.parametrize("seed,N,L,Hq,Hkv", [(0, 7, 20, 2, 2), (1, 26, 0, 4, 2), (2, 64, 300, 4, 1), (3, 1, 50, 2, 2)])
def test_rope_tree_attention_matches_sdpa(seed, N, L, Hq, Hkv):
    g = synth.rng(10 + seed)
    parent = synth.bank_trees()[-1][:N] if N in (1, 26, 64) else synth.full_tree((2, 2))
    parent = np.asarray(parent, np.int32)
    d = 128
    q = synth.normal_bf16(g, (N, Hq, d))
    k = synth.normal_bf16(g, (Hkv, L + N + 3, d))
    v = synth.normal_bf16(g, (Hkv, L + N + 3, d))
    got, k_rot = oracle.tree_attention_rope(q, k, v, L, parent)
    ref, k_ref = _sdpa_rope_reference(q, k, v, L, parent)
    np.testing.assert_allclose(got, ref, rtol=1e-9, atol=1e-10)
    np.testing.assert_array_equal(k_rot, k_ref)


def test_rope_chain_is_causal_attention_at_consecutive_positions():
    # a chain puts node i at L + i: causal attention over the step's tokens
    g = synth.rng(20)
    N, L, d = 9, 33, 128
    q = synth.normal_bf16(g, (N, 1, d))
    k = synth.normal_bf16(g, (1, L + N, d))
    v = synth.normal_bf16(g, (1, L + N, d))
    got, _ = oracle.tree_attention_rope(q, k, v, L, synth.chain(N))
    pos = np.arange(L, L + N, dtype=np.int32)
    qr = torch.from_numpy(oracle.rope(q[:, 0], pos))[None, None]
    kr = np.concatenate([_f(k[0, :L]), _f(_bf(oracle.rope(k[0, L:], pos)))])
    kt = torch.from_numpy(kr)[None, None]
    vt = torch.from_numpy(_f(v[0]))[None, None]
    mask = torch.ones(N, L + N, dtype=torch.bool)
    mask[:, L:] = torch.tril(torch.ones(N, N, dtype=torch.bool))
    o = torch.nn.functional.scaled_dot_product_attention(qr, kt, vt, attn_mask=mask)[0, 0].numpy()
    np.testing.assert_allclose(got[:, 0], o, rtol=1e-9, atol=1e-10)
