"""Pins for the fp64 oracle: each test ties it to something other than itself.

Attention is checked against torch's float64 scaled_dot_product_attention with
masks built from networkx ancestor sets (library routines), and against
closed forms; the LM-head statistics against torch float64 softmax/entropy and
closed forms; greedy acceptance against brute-force enumeration of root paths
on every small tree; compaction against its defining invariants.
"""
import itertools
import json
import math
import os

import networkx as nx
import numpy as np
import pytest
import torch

import oracle
from paper_2606_27550_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf(x):
    return synth.to_bf16_bits(np.asarray(x, dtype=np.float32))


def _f64(bits):
    return torch.from_numpy(synth.bf16_bits_to_f32(bits).astype(np.float64))


def _nx_ancestors_or_self(parent):
    g = nx.DiGraph()
    g.add_nodes_from(range(len(parent)))
    g.add_edges_from((int(p), i) for i, p in enumerate(parent) if p >= 0)
    return [sorted(nx.ancestors(g, i) | {i}) for i in range(len(parent))]


def _sdpa_tree_reference(q, k, v, L, parent):
    """torch float64 SDPA with an explicit boolean mask from networkx ancestors."""
    N, Hq, d = q.shape
    Hkv = k.shape[0]
    anc = _nx_ancestors_or_self(parent)
    mask = torch.zeros(N, L + N, dtype=torch.bool)
    mask[:, :L] = True
    for i, a in enumerate(anc):
        for j in a:
            mask[i, L + j] = True
    qt = _f64(q).permute(1, 0, 2).unsqueeze(0)            # [1, Hq, N, d]
    kt = _f64(k[:, : L + N]).unsqueeze(0)                   # [1, Hkv, L+N, d]
    vt = _f64(v[:, : L + N]).unsqueeze(0)
    if Hkv != Hq:
        kt = kt.repeat_interleave(Hq // Hkv, dim=1)
        vt = vt.repeat_interleave(Hq // Hkv, dim=1)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
    return o[0].permute(1, 0, 2).numpy()


# ---------------------------------------------------------------- tree sets


def test_tree_hand_example():
    g = json.load(open(os.path.join(GOLDEN, "hand_examples.json")))["binary_tree_7"]
    depth, in_anc = oracle.tree(g["parent"])
    assert depth.tolist() == g["depth"]
    assert [sorted(np.nonzero(r)[0].tolist()) for r in in_anc] == g["ancestors_or_self"]
    assert synth.full_tree((2, 2)).tolist() == g["parent"]


@pytest.mark.parametrize("seed", range(5))
def test_tree_sets_match_networkx(seed):
    parent = synth.random_tree(synth.rng(seed), 40)
    depth, in_anc = oracle.tree(parent)
    anc = _nx_ancestors_or_self(parent)
    assert [sorted(np.nonzero(r)[0].tolist()) for r in in_anc] == anc
    g = nx.DiGraph([(int(p), i) for i, p in enumerate(parent) if p >= 0])
    sp = nx.single_source_shortest_path_length(g, 0)
    assert depth.tolist() == [sp[i] for i in range(len(parent))]


@pytest.mark.parametrize("parent", [[0], [-1, 1], [-1, 2, 1], [-1, 5], [1, -1]])
def test_tree_rejects_invalid(parent):
    with pytest.raises(ValueError):
        oracle.tree(parent)


# ---------------------------------------------------------------- attention


def test_attention_hand_example():
    """d=4, one head, L=1, chain root->1.  Scores are 0 or 1 after the 1/sqrt(4) scale."""
    k = _bf([[[2, 0, 0, 0], [0, 2, 0, 0], [0, 0, 2, 0]]])
    v = _bf([[[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 1, 0]]])
    q = _bf([[[1, 0, 0, 0]], [[0, 0, 1, 1]]])
    o = oracle.tree_attention(q, k, v, 1, [-1, 0])
    e = math.e
    # root sees the prefix slot and itself: weights e/(e+1), 1/(e+1)
    np.testing.assert_allclose(o[0, 0], [e / (e + 1), 1 / (e + 1), 0, 0], rtol=0, atol=1e-15)
    # node 1 sees prefix, root and itself: weights 1, 1, e over (2+e)
    np.testing.assert_allclose(o[1, 0], [1 / (2 + e), 1 / (2 + e), e / (2 + e), 0], rtol=0, atol=1e-15)


@pytest.mark.parametrize("L,N,seed", [(0, 1, 0), (5, 1, 1), (37, 9, 2), (64, 64, 3)])
def test_chain_equals_causal_attention(L, N, seed):
    """A chain tree is ordinary causal attention over the L+N tokens."""
    g = synth.rng(seed)
    H, d = 3, 32
    k = synth.normal_bf16(g, (H, L + N, d))
    v = synth.normal_bf16(g, (H, L + N, d))
    q_all = synth.normal_bf16(g, (L + N, H, d))
    o = oracle.tree_attention(q_all[L:], k, v, L, synth.chain(N))
    qt = _f64(q_all).permute(1, 0, 2).unsqueeze(0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, _f64(k).unsqueeze(0), _f64(v).unsqueeze(0),
                                                           is_causal=True)
    ref = ref[0].permute(1, 0, 2).numpy()[L:]
    np.testing.assert_allclose(o, ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("L", [0, 1, 100])
def test_single_node_equals_decode_attention(L):
    g = synth.rng(10 + L)
    H, d = 4, 64
    k = synth.normal_bf16(g, (H, L + 1, d))
    v = synth.normal_bf16(g, (H, L + 1, d))
    q = synth.normal_bf16(g, (1, H, d))
    o = oracle.tree_attention(q, k, v, L, [-1])
    qt = _f64(q).permute(1, 0, 2).unsqueeze(0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, _f64(k).unsqueeze(0), _f64(v).unsqueeze(0))
    np.testing.assert_allclose(o, ref[0].permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("seed,N,L,Hq,Hkv", [(0, 7, 128, 4, 4), (1, 26, 50, 8, 2), (2, 64, 3, 4, 1), (3, 13, 0, 2, 2)])
def test_tree_attention_matches_masked_sdpa(seed, N, L, Hq, Hkv):
    g = synth.rng(seed)
    d = 32
    parent = synth.random_tree(g, N)
    k = synth.normal_bf16(g, (Hkv, L + N + 5, d))
    v = synth.normal_bf16(g, (Hkv, L + N + 5, d))
    q = synth.normal_bf16(g, (N, Hq, d))
    o = oracle.tree_attention(q, k, v, L, parent)
    ref = _sdpa_tree_reference(q, k, v, L, parent)
    np.testing.assert_allclose(o, ref, rtol=1e-12, atol=1e-12)


def test_attention_constant_values_and_zero_query():
    g = synth.rng(7)
    N, L, H, d = 26, 40, 2, 16
    parent = synth.rank_product_tree((4, 3, 2, 1), N)
    k = synth.normal_bf16(g, (H, L + N, d))
    q = synth.normal_bf16(g, (N, H, d))
    const = np.broadcast_to(_bf(np.linspace(-1, 1, d)), (H, L + N, d)).copy()
    o = oracle.tree_attention(q, k, const, L, parent)
    np.testing.assert_allclose(o, np.broadcast_to(synth.bf16_bits_to_f32(const[0, 0]), o.shape), atol=1e-14)
    v = synth.normal_bf16(g, (H, L + N, d))
    o0 = oracle.tree_attention(np.zeros_like(q), k, v, L, parent)
    vf = synth.bf16_bits_to_f32(v).astype(np.float64)
    for i, a in enumerate(_nx_ancestors_or_self(parent)):
        slots = list(range(L)) + [L + j for j in a]
        np.testing.assert_allclose(o0[i], vf[:, slots].mean(axis=1), atol=1e-13)


def test_attention_prefix_permutation_invariance():
    g = synth.rng(8)
    N, L, H, d = 9, 30, 2, 16
    parent = synth.random_tree(g, N)
    k = synth.normal_bf16(g, (H, L + N, d))
    v = synth.normal_bf16(g, (H, L + N, d))
    q = synth.normal_bf16(g, (N, H, d))
    perm = np.concatenate([g.permutation(L), np.arange(L, L + N)])
    o1 = oracle.tree_attention(q, k, v, L, parent)
    o2 = oracle.tree_attention(q, k[:, perm], v[:, perm], L, parent)
    np.testing.assert_allclose(o1, o2, atol=1e-13)


# ---------------------------------------------------------------- LM head


def test_lm_head_hand_example():
    W = _bf([[1, 0], [0, 1], [1, 1]])
    h = _bf([[1, 0.5]])
    am, top1, ent, gap = oracle.lm_head(h, W)
    z = [1.0, 0.5, 1.5]
    s = sum(math.exp(x - 1.5) for x in z)
    assert am[0] == 2
    assert top1[0] == pytest.approx(1 / s, abs=1e-15)
    assert ent[0] == pytest.approx(-sum((math.exp(x - 1.5) / s) * math.log(math.exp(x - 1.5) / s) for x in z), abs=1e-15)
    assert gap[0] == pytest.approx(0.5, abs=1e-15)


@pytest.mark.parametrize("seed,R,D,V", [(0, 7, 256, 1000), (1, 3, 64, 4099)])
def test_lm_head_matches_torch(seed, R, D, V):
    g = synth.rng(seed)
    W = synth.normal_bf16(g, (V, D), 0.02)
    h = synth.normal_bf16(g, (R, D))
    am, top1, ent, gap, logits = oracle.lm_head(h, W, want_logits=True)
    z = _f64(h) @ _f64(W).T
    np.testing.assert_allclose(logits, z.numpy(), rtol=1e-13, atol=1e-13)
    assert am.tolist() == torch.argmax(z, dim=1).tolist()
    p = torch.softmax(z, dim=1)
    np.testing.assert_allclose(top1, p.max(dim=1).values.numpy(), rtol=1e-12)
    np.testing.assert_allclose(ent, torch.distributions.Categorical(logits=z).entropy().numpy(), rtol=1e-10)
    top2 = torch.topk(z, 2, dim=1).values
    np.testing.assert_allclose(gap, (top2[:, 0] - top2[:, 1]).numpy(), rtol=1e-12, atol=1e-13)
    assert np.all(ent >= 0) and np.all(ent <= math.log(V) + 1e-12)


def test_lm_head_uniform_and_peaked():
    V, D = 777, 32
    am, top1, ent, _ = oracle.lm_head(_bf(np.ones((2, D))), np.zeros((V, D), dtype=np.uint16))
    assert am.tolist() == [0, 0]  # all logits tie: lowest index
    np.testing.assert_allclose(ent, math.log(V), rtol=1e-12)
    np.testing.assert_allclose(top1, 1 / V, rtol=1e-12)
    W = np.zeros((V, D), dtype=np.uint16)
    W[123] = _bf(np.full(D, 4.0))
    am, top1, ent, gap = oracle.lm_head(_bf(np.ones((1, D))), W)  # logit 128 on id 123, 0 elsewhere
    assert am[0] == 123 and gap[0] == 128.0
    assert top1[0] == pytest.approx(1.0, abs=1e-50) and ent[0] < 1e-50


# ---------------------------------------------------------------- acceptance


def test_acceptance_hand_cases():
    g = json.load(open(os.path.join(GOLDEN, "hand_examples.json")))["acceptance_cases"]
    for c in g["cases"]:
        assert oracle.accept(g["parent"], c["draft"], c["argmax"]) == (c["accept_len"], c["path"], c["bonus"]), c["why"]


def _brute_force_accept(parent, draft, argmax, tie="lex"):
    """Enumerate every root path with networkx; keep those whose every edge
    (u -> w) carries draft[w] == argmax[u]; take the longest.  Among equally
    long paths: lexicographically smallest (tie="lex"), or smallest end node
    (tie="end").  In breadth-first order the two rules agree."""
    g = nx.DiGraph()
    g.add_nodes_from(range(len(parent)))
    g.add_edges_from((int(p), i) for i, p in enumerate(parent) if p >= 0)
    paths = [[0]] + [p for t in range(1, len(parent)) for p in nx.all_simple_paths(g, 0, t)]
    good = [p for p in paths if all(draft[w] == argmax[u] for u, w in zip(p, p[1:]))]
    best = min(good, key=(lambda p: (-len(p), p)) if tie == "lex" else (lambda p: (-len(p), p[-1])))
    return len(best), best, int(argmax[best[-1]])


def _all_trees(n):
    for parents in itertools.product(*[range(i) for i in range(1, n)]):
        yield [-1] + list(parents)


def _is_bfs(parent):
    return all(parent[i] <= parent[i + 1] for i in range(1, len(parent) - 1))


@pytest.mark.parametrize("n,V", [(1, 2), (2, 2), (3, 2), (4, 2), (5, 2), (4, 3)])
def test_acceptance_brute_force_exhaustive(n, V):
    """Every tree with parent[i] < i on n nodes, every draft/argmax assignment
    over V tokens.  Breadth-first-ordered trees (the order the library
    canonicalises to) must give the lexicographically smallest longest path."""
    for parent in _all_trees(n):
        tie = "lex" if _is_bfs(parent) else "end"
        for draft_tail in itertools.product(range(V), repeat=n - 1):
            draft = [0] + list(draft_tail)
            for argmax in itertools.product(range(V), repeat=n):
                assert oracle.accept(parent, draft, argmax) == _brute_force_accept(parent, draft, argmax, tie)


@pytest.mark.parametrize("seed", range(30))
def test_acceptance_brute_force_random(seed):
    g = synth.rng(seed)
    n = int(g.integers(1, 65))
    parent = synth.random_tree(g, n)
    V = int(g.integers(2, 4))
    draft = g.integers(0, V, size=n).astype(np.int32)
    argmax = g.integers(0, V, size=n).astype(np.int32)
    assert oracle.accept(parent, draft, argmax) == _brute_force_accept(parent, draft, argmax, "end")
    bfs = synth.rank_product_tree(synth.BANK_BRANCHING, n)
    assert oracle.accept(bfs, draft, argmax) == _brute_force_accept(bfs, draft, argmax, "lex")


def test_acceptance_special_cases():
    assert oracle.accept([-1], [0], [42]) == (1, [0], 42)
    n = 64
    argmax = np.arange(100, 100 + n, dtype=np.int32)
    draft = np.concatenate([[0], argmax[:-1]]).astype(np.int32)  # every chain draft matches
    k, path, bonus = oracle.accept(synth.chain(n), draft, argmax)
    assert (k, path, bonus) == (n, list(range(n)), int(argmax[-1]))
    draft2 = draft.copy()
    draft2[1:] = 5  # nothing matches
    assert oracle.accept(synth.chain(n), draft2, argmax) == (1, [0], 100)


# ---------------------------------------------------------------- compaction


def test_compaction_invariants():
    g = synth.rng(3)
    cache = synth.normal_bf16(g, (2, 3, 50, 8))
    L = 20
    same = oracle.kv_compact(cache, L, [0, 1, 2])
    assert np.array_equal(same, cache)  # path [0..k) is the identity
    path = [0, 2, 6, 13]
    new = oracle.kv_compact(cache, L, path)
    for j, src in enumerate(path):
        assert np.array_equal(new[..., L + j, :], cache[..., L + src, :])
    untouched = [s for s in range(50) if not (L <= s < L + len(path))]
    assert np.array_equal(new[..., untouched, :], cache[..., untouched, :])
