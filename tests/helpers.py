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


def gap_filtered_hidden(seed: int, n: int, W):
    """n hidden rows whose oracle top-2 logit gap exceeds GAP_MIN, with their oracle stats."""
    D = W.shape[1]
    for attempt in range(8):
        pool = synth.gen_hidden_pool(seed + 1000 * attempt, n + max(8, n // 2), D)
        am, t1, en, gap = oracle.lm_head(pool, W)
        keep = np.nonzero(gap > GAP_MIN)[0][:n]
        if len(keep) == n:
            return pool[keep], am[keep], t1[keep], en[keep]
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
