"""Case builders shared by the GPU parity tests (inputs from synth, expected
values from the oracle only)."""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

import oracle
from paper_2606_27550_gb300 import synth

ATT_MAX, ATT_MEAN = 1e-2, 1e-3  # attention: max-abs / mean-abs vs the fp64 oracle
STAT_TOL = 1e-3                 # top-1 probability and entropy: abs
GAP_MIN = 1e-2                  # top-2 logit gap of every generated hidden row


def to_dev(a, device="cuda"):
    import torch

    t = torch.from_numpy(np.ascontiguousarray(a))
    if a.dtype == np.uint16:
        t = t.view(torch.int16).view(torch.bfloat16)
    return t.to(device)


def bits(t) -> np.ndarray:
    """bf16 torch tensor -> numpy uint16 bit patterns."""
    import torch

    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def gap_filtered_hidden(seed: int, n: int, W, want_logits: bool = False):
    """n hidden rows whose oracle top-2 logit gap exceeds GAP_MIN, with their oracle
    stats (and their fp64 logits when want_logits)."""
    D = W.shape[1]
    for attempt in range(8):
        pool = synth.gen_hidden_pool(seed + 1000 * attempt, n + max(8, n // 2), D)
        out = oracle.lm_head(pool, W, want_logits=want_logits)
        am, t1, en, gap = out[:4]
        keep = np.nonzero(gap > GAP_MIN)[0][:n]
        if len(keep) == n:
            rows = (pool[keep], am[keep], t1[keep], en[keep])
            return rows + (out[4][keep],) if want_logits else rows
    raise RuntimeError("could not draw hidden rows with a clear top-2 gap")


@dataclass
class Case:
    parent: np.ndarray
    L: int
    L_cap: int
    k: np.ndarray      # [layers][Hkv][L_cap][d] bf16 bits
    v: np.ndarray
    q: np.ndarray      # [layers][N][Hq][d]
    W: np.ndarray      # [V][D]
    hidden: np.ndarray  # [N][D]
    argmax: np.ndarray
    top1: np.ndarray
    entropy: np.ndarray
    drafts: np.ndarray

    @property
    def N(self):
        return len(self.parent)


def make_case(seed: int, parent, L: int, n_layers: int, Hq: int, Hkv: int, d: int, D: int, V: int, p_match: float,
              L_cap: int | None = None) -> Case:
    parent = np.asarray(parent, dtype=np.int32)
    N = len(parent)
    L_cap = L + N + 3 if L_cap is None else L_cap
    k, v = synth.gen_kv(seed, n_layers, Hkv, L_cap, d, L + N)
    q = synth.gen_q(seed, n_layers, N, Hq, d)
    W = synth.gen_lm_head(seed, V, D)
    hidden, am, t1, en = gap_filtered_hidden(seed, N, W)
    drafts = synth.gen_drafts(seed, parent, am, V, p_match)
    return Case(parent, L, L_cap, k, v, q, W, hidden, am, t1, en, drafts)


def check_attention(got: np.ndarray, ref: np.ndarray, what: str = "attention"):
    err = np.abs(got.astype(np.float64) - ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert err.max() <= ATT_MAX, f"{what}: max |err| {err.max():.3e} > {ATT_MAX}"
    assert err.mean() <= ATT_MEAN, f"{what}: mean |err| {err.mean():.3e} > {ATT_MEAN}"
    return float(err.max()), float(err.mean())


def attention_bound(ref, ref_abs_v):
    """Per-element error bound of the kernels' attention: bf16 output and bf16
    probabilities in P V (2^-8 each), and 2^-12 A for the fp32 steps."""
    return 2.0 ** -8 * np.abs(ref) + (2.0 ** -8 + 2.0 ** -12) * ref_abs_v


def check_attention_fuzz(got, ref, ref_abs_v, what):
    """got vs the oracle's ref, with ref_abs_v the oracle's attention over |V|."""
    got = got.astype(np.float64)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - ref)
    elem = attention_bound(ref, ref_abs_v)
    bound = np.maximum(1e-2, elem)
    worst = np.argmax(err - bound)
    n_over = int((err > 1e-2).sum())
    if n_over:
        print(f"{what}: {n_over} of {err.size} elements beyond 1e-2, within the derived bound")
    assert (err <= bound).all(), (f"{what}: |err| {err.flat[worst]:.3e} at |ref| {abs(ref.flat[worst]):.3f}, "
                                  f"bound {bound.flat[worst]:.3e}")
    mean_bound = max(1e-3, 0.5 * float(elem.mean()))
    if err.mean() > 1e-3:
        print(f"{what}: mean |err| {err.mean():.3e} beyond 1e-3, within the derived {mean_bound:.3e}")
    assert err.mean() <= mean_bound, f"{what}: mean |err| {err.mean():.3e} > {mean_bound:.3e}"


def abs_bits(a):
    """|x| of bf16 bit patterns (sign bit cleared)."""
    return (a & np.uint16(0x7FFF)).astype(np.uint16)


# typical acceptance: the paper's settings (temperature, posterior threshold, mixing coefficient)
TYPICAL = (0.7, 0.09, 0.3)
MARGIN_MIN = 1e-3  # |p - threshold| / threshold of every edge, so fp32 and fp64 decide alike
LL_GAP_MIN = 1e-3  # path log-likelihood gap between the best deepest accepted node and any other
LOGIT_TOL = 1e-3   # gathered draft logits and tempered log-partitions: abs


def typical_ambiguity(parent, drafts, logits, T, eps, alpha):
    """Edges whose decision sits within MARGIN_MIN of the threshold, and whether the
    choice among the deepest accepted nodes is within LL_GAP_MIN (different tokens)."""
    k, path, bonus, det = oracle.typical_accept(parent, drafts, logits, T, eps, alpha, detail=True)
    close = [j for j in range(1, len(parent)) if abs(det["margin"][j]) < MARGIN_MIN]
    depth = synth.depth_of(parent)
    cand = [i for i in range(len(parent)) if det["accepted"][i] and depth[i] == k - 1]
    lls = sorted((det["loglik"][i] for i in cand), reverse=True)
    tie = len(lls) > 1 and 0 < lls[0] - lls[1] < LL_GAP_MIN
    return close, tie


def typical_drafts(seed: int, parent, logits, T, eps, alpha, p_likely: float = 0.7):
    """Draft tokens whose typical-acceptance decisions are all clear of the threshold.

    Each non-root node proposes, with probability p_likely, a token drawn from its
    parent's tempered target distribution (what a trained head tends to propose),
    else a uniform token.  Tokens whose edge margin is within MARGIN_MIN are redrawn;
    a near-tie between equally deep accepted paths redraws everything."""
    parent = np.asarray(parent)
    n, V = logits.shape
    w = np.exp((logits - logits.max(axis=1, keepdims=True)) / T)
    w /= w.sum(axis=1, keepdims=True)
    for attempt in range(20):
        g = synth.rng(seed + 7919 * attempt, 9)
        drafts = np.zeros(n, dtype=np.int32)

        def draw(j):
            if g.random() < p_likely:
                return int(g.choice(V, p=w[parent[j]]))
            return int(g.integers(0, V))

        for j in range(1, n):
            drafts[j] = draw(j)
        for _ in range(20):
            close, tie = typical_ambiguity(parent, drafts, logits, T, eps, alpha)
            if not close:
                break
            for j in close:
                drafts[j] = draw(j)
        close, tie = typical_ambiguity(parent, drafts, logits, T, eps, alpha)
        if not close and not tie:
            return drafts
    raise RuntimeError("could not draw unambiguous drafts")


# ---------------------------------------------------------------- speculative sampling

WALK_MARGIN = 1e-4  # every decision of the oracle's walk at least this far from its boundary


def softmax_rows(z, temp):
    w = np.exp((z - z.max(axis=1, keepdims=True)) / temp)
    return w / w.sum(axis=1, keepdims=True)


def draw_decidable_walk(g, parent, z, q, temp, p_from_q=0.8):
    """Drafts (children of u drawn from q_u, else uniform) and uniforms that keep
    every decision of the oracle's walk -- a uniform against a probability ratio,
    or against a CDF -- at least WALK_MARGIN from its boundary, so float32 and
    float64 decide alike.  Returns (draft, unif, (accept_len, path, token))."""
    n, V = z.shape
    draft = np.zeros(n, np.int32)
    for c in range(1, n):
        u = parent[c]
        draft[c] = g.choice(V, p=q[u] / q[u].sum()) if g.random() < p_from_q else g.integers(0, V)
    for _ in range(200):
        unif = g.random(2 * n).astype(np.float32).astype(np.float64)
        k, path, tok, det = oracle.spec_sample(parent, draft, z, q, temp, unif, detail=True)
        rm = det["ratio_margin"]
        tried = rm[~np.isnan(rm)]
        if (np.abs(tried[np.isfinite(tried)]) > WALK_MARGIN).all() and det["cdf_margin"] > WALK_MARGIN:
            return draft, unif, (k, path, tok)
    raise RuntimeError("no unambiguous uniforms")
