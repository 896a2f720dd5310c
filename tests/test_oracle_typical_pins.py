"""Pins for the oracle's typical acceptance (Medusa/Hydra rule, T = 0.7,
eps = 0.09, alpha = 0.3 in the paper's runs).

Each test ties it to something other than itself: closed forms on hand
distributions (dyadic probabilities whose entropy is a multiple of ln 2),
limits (uniform logits, eps -> 0, an unreachable threshold, T -> 0 where the
rule becomes the separately pinned greedy rule), invariances (a constant added
to a row, logits and temperature scaled together), and brute force: torch's
Categorical for p and H, networkx for root paths.
"""
import math
from fractions import Fraction

import networkx as nx
import numpy as np
import pytest
import scipy.special
import torch

import oracle
from paper_2606_27550_gb300 import synth

EPS, ALPHA, T = 0.09, 0.3, 0.7


def _rows(parent, row0, V, fill=0.0):
    z = np.full((len(parent), V), fill)
    z[0] = row0
    return z


# ---------------------------------------------------------------- closed forms

def _closed_form_margins(p, eps, alpha):
    """p: exact probabilities (Fractions) of one row.  Returns (H, threshold)."""
    H = -sum(float(x) * math.log(float(x)) for x in p if x > 0)
    return H, min(eps, alpha * math.exp(-H))


def test_dyadic_row_temperature_one():
    # p = (1/2, 1/4, 1/8, 1/8): H = 1.75 ln 2, alpha e^-H = 0.3 * 2^-1.75 = 0.08919
    p = [Fraction(1, 2), Fraction(1, 4), Fraction(1, 8), Fraction(1, 8)]
    z0 = np.log([float(x) for x in p])
    parent = [-1, 0, 0, 0, 2]
    draft = [0, 1, 2, 3, 0]
    H, thr = _closed_form_margins(p, EPS, ALPHA)
    assert H == pytest.approx(1.75 * math.log(2), rel=1e-15)
    assert thr == pytest.approx(0.3 * 2 ** -1.75, rel=1e-15)
    # row of node 2 is uniform over 4 tokens: 1/4 > min(0.09, 0.3/4)
    z = _rows(parent, z0, 4)
    k, path, bonus, det = oracle.typical_accept(parent, draft, z, 1.0, EPS, ALPHA, detail=True)
    for j in (1, 2, 3):
        assert det["margin"][j] == pytest.approx((float(p[draft[j]]) - thr) / thr, rel=1e-12)
    assert det["margin"][4] == pytest.approx((0.25 - 0.075) / 0.075, rel=1e-12)
    assert det["accepted"].tolist() == [True] * 5
    # deepest accepted node is 4 (depth 2); its path log-likelihood ln(1/8) + ln(1/4)
    assert det["loglik"][4] == pytest.approx(math.log(0.125) + math.log(0.25), rel=1e-12)
    assert (k, path, bonus) == (3, [0, 2, 4], 0)

    # alpha = 0.5, eps = 1: threshold 0.5 * 2^-1.75 = 0.1487 rejects the 1/8 tokens
    k, path, bonus, det = oracle.typical_accept(parent, draft, z, 1.0, 1.0, 0.5, detail=True)
    assert det["accepted"].tolist() == [True, True, False, False, False]
    assert (k, path, bonus) == (2, [0, 1], 0)


def test_dyadic_row_temperature_half():
    # T = 1/2 squares and renormalises: (16, 4, 1, 1) / 22
    base = [Fraction(1, 2), Fraction(1, 4), Fraction(1, 8), Fraction(1, 8)]
    q = [x * x for x in base]
    q = [x / sum(q) for x in q]
    assert q == [Fraction(16, 22), Fraction(4, 22), Fraction(1, 22), Fraction(1, 22)]
    z0 = np.log([float(x) for x in base])
    parent, draft = [-1, 0, 0, 0], [0, 0, 1, 2]
    H, thr = _closed_form_margins(q, EPS, ALPHA)
    k, path, bonus, det = oracle.typical_accept(parent, draft, _rows(parent, z0, 4), 0.5, EPS, ALPHA, detail=True)
    for j in (1, 2, 3):
        assert det["margin"][j] == pytest.approx((float(q[draft[j]]) - thr) / thr, rel=1e-12)
    # 16/22 and 4/22 pass; 1/22 = 0.045 is below min(0.09, 0.3 e^-H)
    assert det["accepted"].tolist() == [True, True, True, False]
    # equally deep: node 1 (p = 16/22) has the larger log-likelihood
    assert (k, path, bonus) == (2, [0, 1], 0)


def test_two_token_logistic():
    # V = 2: p(token 1) = sigmoid((b - a) / T), H the binary entropy
    for a, b in [(0.0, 1.0), (2.0, -1.0), (0.3, 0.31)]:
        s = 1.0 / (1.0 + math.exp(-(b - a) / T))
        H = -(s * math.log(s) + (1 - s) * math.log(1 - s))
        thr = min(EPS, ALPHA * math.exp(-H))
        _, _, _, det = oracle.typical_accept([-1, 0], [0, 1], np.array([[a, b], [0.0, 0.0]]), T, EPS, ALPHA,
                                             detail=True)
        assert det["margin"][1] == pytest.approx((s - thr) / thr, rel=1e-12)
        assert det["accepted"][1] == (s > thr)


def test_log_likelihood_decides_between_equal_depths():
    # two depth-2 branches, both accepted; the larger-index one is more likely
    parent = [-1, 0, 0, 1, 2]
    draft = [0, 0, 1, 0, 0]
    z = np.zeros((5, 3))
    z[0] = [1.0, 1.2, -5.0]     # p(token 0) < p(token 1)
    z[1] = [0.5, 0.0, 0.0]
    z[2] = [2.0, 0.0, 0.0]      # node 4's token is likelier than node 3's
    k, path, bonus, det = oracle.typical_accept(parent, draft, z, 1.0, EPS, ALPHA, detail=True)
    assert det["accepted"].all()
    assert det["loglik"][4] > det["loglik"][3]
    assert (k, path) == (3, [0, 2, 4])
    assert bonus == 0  # z[4] = 0 everywhere: lowest index on ties


# ---------------------------------------------------------------- limits

@pytest.mark.parametrize("seed", range(4))
def test_uniform_logits_accept_every_node(seed):
    # p = 1/V > alpha / V for alpha < 1: every edge passes, whatever eps is
    g = synth.rng(seed)
    n = 2 + int(g.integers(0, 40))
    parent = synth.random_tree(g, n)
    V = 17
    draft = g.integers(0, V, n)
    for eps in (1e-9, 0.09, 1.0):
        k, path, bonus, det = oracle.typical_accept(parent, draft, np.zeros((n, V)), T, eps, ALPHA, detail=True)
        assert det["accepted"].all()
        depth, _ = oracle.tree(parent)
        assert k == depth.max() + 1
        # all log-likelihoods of equal depth tie: the smallest deepest index wins
        assert path[-1] == int(np.flatnonzero(depth == depth.max())[0])
        assert bonus == 0


def test_threshold_limits():
    g = synth.rng(11)
    parent = synth.random_tree(g, 30)
    z = g.standard_normal((30, 50)) * 3
    draft = g.integers(0, 50, 30)
    # eps -> 0: the threshold vanishes and every finite-logit edge passes
    _, _, _, det = oracle.typical_accept(parent, draft, z, T, 1e-300, ALPHA, detail=True)
    assert det["accepted"].all()
    # threshold 1 is out of reach of any probability: only the root
    k, path, bonus = oracle.typical_accept(parent, draft, z, T, 1.0, 1e9)
    assert (k, path, bonus) == (1, [0], int(np.argmax(z[0])))


def test_out_of_range_draft_is_rejected():
    parent = [-1, 0, 0, 0]
    z = np.zeros((4, 5))
    k, path, _, det = oracle.typical_accept(parent, [0, -1, 5, 3], z, T, EPS, ALPHA, detail=True)
    assert det["accepted"].tolist() == [True, False, False, True]
    assert (k, path) == (2, [0, 3])


@pytest.mark.parametrize("seed", range(6))
def test_low_temperature_reduces_to_greedy(seed):
    # T -> 0: p concentrates on the argmax (p = 1 exactly once e^(-gap/T)
    # underflows), H -> 0, threshold -> min(eps, alpha) < 1: an edge passes
    # iff its token is the greedy one, and log-likelihoods all tie at 0.
    g = synth.rng(100 + seed)
    n = int(g.integers(2, 65))
    parent = synth.random_tree(g, n)
    V = 40
    z = np.stack([g.permutation(V) for _ in range(n)]) * 0.1  # distinct logits, gaps >= 0.1
    am = z.argmax(axis=1).astype(np.int32)
    draft = g.integers(0, V, n).astype(np.int32)
    hit = g.random(n) < 0.6
    for j in range(1, n):
        if hit[j]:
            draft[j] = am[parent[j]]
    gaps = np.sort(z, axis=1)
    assert (gaps[:, -1] - gaps[:, -2]).min() > 1e-3
    got = oracle.typical_accept(parent, draft, z, 1e-6, EPS, ALPHA)
    assert got == oracle.accept(parent, draft, am)


@pytest.mark.parametrize("seed", range(4))
def test_shift_and_scale_invariance(seed):
    g = synth.rng(200 + seed)
    n = 24
    parent = synth.random_tree(g, n)
    z = g.standard_normal((n, 30)) * 2
    draft = g.integers(0, 30, n)
    ref = oracle.typical_accept(parent, draft, z, T, EPS, ALPHA, detail=True)
    shifted = z + g.standard_normal((n, 1)) * 10
    for got in (oracle.typical_accept(parent, draft, shifted, T, EPS, ALPHA, detail=True),
                oracle.typical_accept(parent, draft, z * 2.5, T * 2.5, EPS, ALPHA, detail=True)):
        assert got[:3] == ref[:3]
        np.testing.assert_allclose(got[3]["margin"], ref[3]["margin"], rtol=1e-9, atol=1e-12)
        np.testing.assert_allclose(got[3]["loglik"], ref[3]["loglik"], rtol=1e-9, atol=1e-12)


# ---------------------------------------------------------------- brute force

def _brute_force(parent, draft, z, temp, eps, alpha):
    """p and H from torch's Categorical, root paths from networkx; the rule
    applied edge by edge along every path."""
    n, V = z.shape
    dist = torch.distributions.Categorical(logits=torch.from_numpy(z) / temp)
    probs, ent = dist.probs.numpy(), dist.entropy().numpy()
    g = nx.DiGraph()
    g.add_nodes_from(range(n))
    g.add_edges_from((int(p), i) for i, p in enumerate(parent) if p >= 0)
    best = None
    for i in range(n):
        route = nx.shortest_path(g, 0, i)
        ok, ll = True, 0.0
        for a, b in zip(route[:-1], route[1:]):
            tok = int(draft[b])
            pe = probs[a, tok] if 0 <= tok < V else 0.0
            ok &= pe > min(eps, alpha * math.exp(-ent[a]))
            ll += math.log(pe) if pe > 0 else -math.inf
        if ok:
            key = (len(route), ll, -i)
            if best is None or key > best[0]:
                best = (key, route)
    route = best[1]
    return len(route), route, int(np.argmax(z[route[-1]]))


@pytest.mark.parametrize("seed", range(12))
def test_matches_brute_force(seed):
    g = synth.rng(300 + seed)
    n = int(g.integers(2, 65))
    parent = synth.random_tree(g, n)
    V = int(g.integers(3, 200))
    z = g.standard_normal((n, V)) * float(g.random()) * 6
    # half the drafts are drawn from the parent's tempered distribution, half uniform
    w = np.exp((z - z.max(axis=1, keepdims=True)) / T)
    w /= w.sum(axis=1, keepdims=True)
    draft = g.integers(0, V, n).astype(np.int32)
    for j in range(1, n):
        if g.random() < 0.5:
            draft[j] = int(g.choice(V, p=w[parent[j]]))
    k, path, bonus, det = oracle.typical_accept(parent, draft, z, T, EPS, ALPHA, detail=True)
    if np.abs(det["margin"][1:]).min() < 1e-9:
        pytest.skip("an edge sits on the threshold")
    assert (k, path, bonus) == _brute_force(parent, draft, z, T, EPS, ALPHA)


# ---------------------------------------------------------------- tempered statistics

def test_tempered_stats_closed_form():
    base = np.log([0.5, 0.25, 0.125, 0.125])
    logz, ent = oracle.tempered_stats(base[None], 0.5)
    # sum_v e^(2 ln p_v) = sum p_v^2 = 22/64; entropy of (16, 4, 1, 1)/22
    q = np.array([16, 4, 1, 1]) / 22
    assert logz[0] == pytest.approx(math.log(22 / 64), rel=1e-14)
    assert ent[0] == pytest.approx(-(q * np.log(q)).sum(), rel=1e-14)
    logz, ent = oracle.tempered_stats(base[None], 1.0)
    assert logz[0] == pytest.approx(0.0, abs=1e-15)
    assert ent[0] == pytest.approx(1.75 * math.log(2), rel=1e-14)
    logz, ent = oracle.tempered_stats(np.full((1, 1000), 3.0), 0.7)
    assert logz[0] == pytest.approx(3.0 / 0.7 + math.log(1000), rel=1e-14)
    assert ent[0] == pytest.approx(math.log(1000), rel=1e-14)


@pytest.mark.parametrize("T_", [0.3, 0.7, 1.0, 2.0])
def test_tempered_stats_match_libraries(T_):
    # against scipy's logsumexp and torch's Categorical entropy; at T = 1 the
    # entropy also equals the (separately pinned) LM-head entropy
    g = synth.rng(400)
    z = g.standard_normal((9, 777)) * 2.5
    logz, ent = oracle.tempered_stats(z, T_)
    np.testing.assert_allclose(logz, scipy.special.logsumexp(z / T_, axis=1), rtol=1e-12)
    cat = torch.distributions.Categorical(logits=torch.from_numpy(z) / T_)
    np.testing.assert_allclose(ent, cat.entropy().numpy(), rtol=1e-11, atol=1e-12)
    # logits and temperature scaled together: unchanged
    logz2, ent2 = oracle.tempered_stats(z * 3.0, T_ * 3.0)
    np.testing.assert_allclose(logz2, logz, rtol=1e-12)
    np.testing.assert_allclose(ent2, ent, rtol=1e-12)


def test_tempered_entropy_at_one_equals_lm_head_entropy():
    g = synth.rng(401)
    W = synth.normal_bf16(g, (300, 64), 0.3)
    h = synth.normal_bf16(g, (5, 64))
    _, _, ent1, _, logits = oracle.lm_head(h, W, want_logits=True)
    _, ent = oracle.tempered_stats(logits, 1.0)
    np.testing.assert_allclose(ent, ent1, rtol=1e-12)
