"""Pins for the oracle's speculative sampling on a draft tree (Sec. 2.1 rule,
siblings tried in order with the residual updated after each rejection).

The defining property is losslessness: when the children of a node are drawn
independently from q, the first emitted token (the accepted child's token or
the replacement drawn from the residual) is distributed exactly as the
target p.  That is checked by Monte Carlo against p for one, two and three
children; hand-worked residuals and limits (q = p accepts every first child,
a token with q = 0 is always accepted, a token with p = 0 never) complete it.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2606_27550_gb300 import synth

T = 0.7


def _softmax(z, temp):
    w = np.exp((z - z.max()) / temp)
    return w / w.sum()


def test_hand_residuals():
    # p = (0.5, 0.3, 0.2) at T = 1 from log-probabilities; q = (0.2, 0.6, 0.2)
    p = np.array([0.5, 0.3, 0.2])
    z = np.log(p)
    q = np.array([0.2, 0.6, 0.2])
    parent = [-1, 0, 0]
    logits = np.stack([z, z, z])
    qs = np.stack([q, q, q])
    # child 1 (token 1): ratio 0.3 / 0.6 = 0.5
    k, path, tok, det = oracle.spec_sample(parent, [0, 1, 2], logits, qs, 1.0, [0, 0.4, 0.9, 0.5, 0, 0], detail=True)
    assert (k, path) == (2, [0, 1]) and det["ratio_margin"][1] == pytest.approx(0.1)
    # rejected: residual max(0, p - q) = (0.3, 0, 0) -> (1, 0, 0); child 2 (token 2) has r = 0: rejected;
    # the second residual max(0, (1, 0, 0) - q) = (0.8, 0, 0) -> (1, 0, 0): the token is 0 whatever the uniform
    for x in (0.0, 0.5, 0.999):
        k, path, tok = oracle.spec_sample(parent, [0, 1, 2], logits, qs, 1.0, [0, 0.6, 0.0, x, 0, 0])
        assert (k, path, tok) == (1, [0], 0)
    # a leaf: the token after it is drawn from its own target p by inverse CDF
    k, path, tok = oracle.spec_sample(parent, [0, 1, 2], logits, qs, 1.0, [0, 0.1, 0, 0, 0.55, 0])
    assert (k, path, tok) == (2, [0, 1], 1)  # cumulative (0.5, 0.8, 1.0): 0.55 falls in token 1


def test_limits():
    g = synth.rng(3)
    parent = synth.bank_trees()[-1]
    n, V = len(parent), 40
    z = g.standard_normal((n, V)) * 2
    p = np.stack([_softmax(z[i], T) for i in range(n)])
    unif = g.random(2 * n)
    draft = g.integers(0, V, n).astype(np.int32)
    # q = p: every ratio is 1 > u, so each node's first child is accepted
    k, path, _ = oracle.spec_sample(parent, draft, z, p, T, unif)
    want, u = [0], 0
    while True:
        kids = [c for c in range(u + 1, n) if parent[c] == u]
        if not kids:
            break
        u = kids[0]
        want.append(u)
    assert path == want and k == len(want)
    # q(t) = 0 for every drafted token: always accepted, same walk
    q = np.full((n, V), 1.0 / (V - 1))
    for c in range(1, n):
        q[parent[c]] = 1.0 / (V - 1)
    draft2 = np.zeros(n, np.int32)
    q[:, 0] = 0.0
    q /= q.sum(axis=1, keepdims=True)
    assert oracle.spec_sample(parent, draft2, z, q, T, unif)[1] == want
    # a token outside the vocabulary has p = 0: never accepted
    assert oracle.spec_sample(parent, np.full(n, V, np.int32), z, p, T, np.zeros(2 * n))[:2] == (1, [0])


@pytest.mark.parametrize("n_children", [1, 2, 3])
def test_first_token_is_distributed_as_the_target(n_children):
    g = synth.rng(10 + n_children)
    V = 6
    z0 = g.standard_normal(V) * 1.5
    p = _softmax(z0, T)
    q = _softmax(g.standard_normal(V) * 1.5, 1.0)
    parent = [-1] + [0] * n_children
    n = len(parent)
    logits = np.tile(z0, (n, 1))
    qs = np.tile(q, (n, 1))
    trials = 30000
    counts = np.zeros(V)
    for _ in range(trials):
        draft = np.concatenate([[0], g.choice(V, size=n_children, p=q)]).astype(np.int32)
        k, path, tok = oracle.spec_sample(parent, draft, logits, qs, T, g.random(2 * n))
        first = draft[path[1]] if k > 1 else tok
        counts[first] += 1
    freq = counts / trials
    # binomial standard error <= 0.0029: 5 sigma
    assert np.abs(freq - p).max() < 0.015, (freq, p)


def test_second_token_given_acceptance_follows_the_child_target():
    # chain root -> 1 -> 2: given node 1 accepted, the next emitted token is distributed as p_1
    g = synth.rng(20)
    V = 5
    z = g.standard_normal((3, V)) * 1.5
    p1 = _softmax(z[1], T)
    q = np.stack([_softmax(g.standard_normal(V), 1.0) for _ in range(3)])
    counts = np.zeros(V)
    hits = 0
    for _ in range(30000):
        draft = np.array([0, g.choice(V, p=q[0]), g.choice(V, p=q[1])], np.int32)
        k, path, tok = oracle.spec_sample([-1, 0, 1], draft, z, q, T, g.random(6))
        if k >= 2:
            hits += 1
            counts[draft[2] if k == 3 else tok] += 1
    assert hits > 5000
    assert np.abs(counts / hits - p1).max() < 0.02


def test_closed_form_residual_matches_the_sequential_update():
    """After k rejected siblings the residual is max(0, p - c_k q) / S_k, with
    c_0 = 0, S_0 = 1 and, after each rejection, c <- c + S, S <- sum_v max(0,
    p - c q) -- the form the GPU walk evaluates.  The oracle applies the rule's
    sequential update norm(max(0, r - q)); its ratio margins give r(t_c) / q(t_c)
    - unif[c] for every child it tries, so r at each tried token is compared
    with the closed form."""
    g = synth.rng(41)
    n = 7
    parent = [-1] + [0] * (n - 1)  # a root with six children: up to six rejections in a row
    compared = deepest = 0
    for trial in range(60):
        V = int(g.choice([5, 50, 500]))
        z = g.standard_normal((n, V)) * float(g.uniform(0.5, 3.0))
        qs = np.stack([_softmax(g.standard_normal(V) * float(g.uniform(0.5, 3.0)), 1.0) for _ in range(n)])
        draft = np.concatenate([[0], g.integers(0, V, n - 1)]).astype(np.int32)
        unif = g.random(2 * n) * float(g.choice([1.0, 0.2]))  # small uniforms: more acceptances, fewer residuals
        unif = np.where(g.random(2 * n) < 0.5, 1.0 - 1e-12, unif)  # and near-1 ones: long runs of rejections
        _, _, _, det = oracle.spec_sample(parent, draft, z, qs, T, unif, detail=True)
        p = _softmax(z[0], T)
        q = qs[0]
        c, S = 0.0, 1.0
        k = 0
        for child in range(1, n):
            margin = det["ratio_margin"][child]
            if np.isnan(margin):
                break  # not tried: a sibling before it was accepted
            t = draft[child]
            r_oracle = (margin + unif[child]) * q[t]
            r_closed = p[t] if k == 0 else (max(0.0, p[t] - c * q[t]) / S if S > 0 else 0.0)
            assert r_oracle == pytest.approx(r_closed, rel=1e-9, abs=1e-15), (trial, child)
            compared += 1
            if margin > 0:
                break  # accepted
            c, S = c + S, float(np.maximum(p - (c + S) * q, 0.0).sum())
            k += 1
        deepest = max(deepest, k)
    assert compared > 150 and deepest >= 5
