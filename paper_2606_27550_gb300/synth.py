"""Seeded synthetic inputs for the tree-verification pass.

This module is shared by the CUDA path's tests and benchmark and by the
CPU oracle's tests.  It holds no arithmetic of the method itself: it draws
random numbers, rounds them to bf16 bit patterns, and builds draft-tree
parent arrays.  Everything that attention, the LM head, acceptance or
compaction compute lives either in the CUDA library or in ``oracle/``.

Random numbers come from numpy's Philox generator, a counter-based
generator, so every input is a pure function of its seed.

Draft-tree shapes (Sec. 2.3: Medusa/Hydra trees are Cartesian products of
the heads' top-k candidates, shipped with precomputed masks, position
offsets and gather indices).  A node is the tuple of child ranks on its
path from the root, ``nu = (r1, .., rd)`` with ``rk < branching[k-1]``.
The n-node tree keeps the first n tuples ordered by (sum of ranks, depth,
lexicographic), the tie-break order of the greedy frontier construction
(Sec. 3.1, Algorithm 1: argmax over (a(nu), -sum nu, -|nu|)), here used
without the acceptance score.  The order is prefix-closed, so any prefix
is a valid tree.  Parent arrays are returned in breadth-first order
(depth, then tuple), so parent[i] < i and parent[0] == -1.
"""
from __future__ import annotations

import itertools
from dataclasses import dataclass, field

import numpy as np

# --------------------------------------------------------------------------
# random numbers and bf16 bit patterns
# --------------------------------------------------------------------------


def rng(seed: int, stream: int = 0) -> np.random.Generator:
    """Counter-based generator (Philox 4x64) keyed by (seed, stream)."""
    return np.random.Generator(np.random.Philox(key=[int(seed) & (2**64 - 1), int(stream) & (2**64 - 1)]))


def to_bf16_bits(x) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even.

    Inputs are finite; NaN/Inf are not produced by these generators."""
    f = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def bf16_bits_to_f32(b) -> np.ndarray:
    """bf16 bit patterns -> float32 (exact)."""
    b = np.ascontiguousarray(np.asarray(b, dtype=np.uint16))
    return (b.astype(np.uint32) << 16).view(np.float32)


def normal_bf16(g: np.random.Generator, shape, std: float = 1.0) -> np.ndarray:
    return to_bf16_bits(g.standard_normal(size=shape, dtype=np.float32) * np.float32(std))


# --------------------------------------------------------------------------
# draft trees
# --------------------------------------------------------------------------


def rank_product_tree(branching, n: int) -> np.ndarray:
    """First n nodes of the rank-product tree for ``branching``.

    Returns parent[] (int32, BFS order, parent[0] = -1)."""
    tuples = [()]
    for depth in range(1, len(branching) + 1):
        tuples.extend(itertools.product(*[range(b) for b in branching[:depth]]))
    if n < 1 or n > len(tuples):
        raise ValueError(f"n={n} outside 1..{len(tuples)} for branching {branching}")
    tuples.sort(key=lambda t: (sum(t), len(t), t))
    kept = tuples[:n]
    kept.sort(key=lambda t: (len(t), t))  # breadth-first order
    index = {t: i for i, t in enumerate(kept)}
    parent = np.full(n, -1, dtype=np.int32)
    for t, i in index.items():
        if t:
            parent[i] = index[t[:-1]]
    return parent


def full_tree(branching) -> np.ndarray:
    """Complete tree with the given per-depth branching (e.g. (2, 2): 7 nodes)."""
    size = 1
    width = 1
    for b in branching:
        width *= b
        size += width
    return rank_product_tree(branching, size)


def chain(n: int) -> np.ndarray:
    parent = np.arange(-1, n - 1, dtype=np.int32)
    return parent


def random_tree(g: np.random.Generator, n: int) -> np.ndarray:
    """Random tree on n nodes with parent[i] < i (not necessarily BFS order)."""
    parent = np.full(n, -1, dtype=np.int32)
    for i in range(1, n):
        parent[i] = int(g.integers(0, i))
    return parent


def depth_of(parent) -> np.ndarray:
    """Depth per node for a parent array with parent[i] < i (input bookkeeping
    used to size buffers and pick trees; not the library's or oracle's code)."""
    d = np.zeros(len(parent), dtype=np.int32)
    for i in range(1, len(parent)):
        d[i] = d[parent[i]] + 1
    return d


# The universal branching of the bank and of the 64-node long-context tree.
BANK_BRANCHING = (4, 3, 2, 2, 2)
BANK_SIZES = (1, 2, 4, 8, 16, 26, 40, 64)


def bank_trees():
    return [rank_product_tree(BANK_BRANCHING, n) for n in BANK_SIZES]


# --------------------------------------------------------------------------
# workload shapes
# --------------------------------------------------------------------------


@dataclass
class Shape:
    name: str
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_model: int
    vocab: int
    L: int
    parent: np.ndarray
    p_match: float
    w_std: float = 0.02
    L_cap: int = 0
    extra: dict = field(default_factory=dict)

    def __post_init__(self):
        if self.L_cap == 0:
            self.L_cap = self.L + 64

    @property
    def N(self) -> int:
        return len(self.parent)


def shape_c1() -> Shape:
    """Tiny single layer: 4 heads x 64, d_model 256, L=128, binary tree of 7."""
    return Shape("tiny-1layer-H4d64-V1000-L128-N7", 1, 4, 4, 64, 256, 1000, 128, full_tree((2, 2)), 0.7)


def shape_c2() -> Shape:
    """7B-shaped single layer: 32x128 MHA, d_model 4096, V=32000, L=1024, 26-node tree."""
    return Shape("7b-1layer-H32d128-V32000-L1024-N26", 1, 32, 32, 128, 4096, 32000, 1024,
                 rank_product_tree((4, 3, 2, 1), 26), 0.6)


def shape_c3() -> Shape:
    """Bank switching: 7B shapes, L starts at 2048 and grows by accept_len."""
    s = Shape("7b-bank8-H32d128-V32000-L2048", 1, 32, 32, 128, 4096, 32000, 2048,
              bank_trees()[-1], 0.6, L_cap=2048 + 1000 * 6 + 64)
    s.extra["steps"] = 1000
    return s


def shape_c4() -> Shape:
    """Long-context full decode step: 32 layers, L=16384, 64-node depth-5 tree."""
    return Shape("7b-32layer-H32d128-V32000-L16384-N64", 32, 32, 32, 128, 4096, 32000, 16384,
                 rank_product_tree(BANK_BRANCHING, 64), 0.5)


@dataclass
class BatchShape:
    """Ragged batch: one (tree, L, p_match) per sequence, shared model shapes."""
    name: str
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_model: int
    vocab: int
    parents: list
    Ls: list
    p_match: list
    w_std: float = 0.02

    @property
    def Ns(self):
        return [len(p) for p in self.parents]


def batch_c5(seed: int = 5, batch: int = 8, vocab: int = 128256, L_range=(512, 8192)) -> BatchShape:
    """Ragged batched verify: GQA 32 q / 8 kv heads x 128, d_model 4096; each
    sequence draws its tree from the bank sizes >= 4, L ~ U[512, 8192] and its
    draft-match probability ~ U[0.3, 0.9]."""
    g = rng(seed, 7)
    trees = [t for t in bank_trees() if len(t) >= 4]
    parents = [trees[int(g.integers(0, len(trees)))] for _ in range(batch)]
    Ls = [int(g.integers(L_range[0], L_range[1] + 1)) for _ in range(batch)]
    ps = [float(g.uniform(0.3, 0.9)) for _ in range(batch)]
    return BatchShape(f"7b-gqa32x8-batch{batch}-V{vocab}-ragged", 1, 32, 8, 128, 4096, vocab, parents, Ls, ps)


SHAPES = {"c1": shape_c1, "c2": shape_c2, "c3": shape_c3, "c4": shape_c4}


# --------------------------------------------------------------------------
# tensors for one verify step
# --------------------------------------------------------------------------


def gen_kv(seed: int, n_layers: int, n_kv_heads: int, L_cap: int, head_dim: int, n_valid: int):
    """K and V caches, layout [layers][kv_heads][L_cap][head_dim] as bf16 bits.

    Slots >= n_valid are filled with a large finite sentinel so that a
    kernel that reads past the valid keys produces visibly wrong output."""
    g = rng(seed, 1)
    shp = (n_layers, n_kv_heads, L_cap, head_dim)
    k = np.empty(shp, dtype=np.uint16)
    v = np.empty(shp, dtype=np.uint16)
    for layer in range(n_layers):
        k[layer] = normal_bf16(g, shp[1:])
        v[layer] = normal_bf16(g, shp[1:])
    if n_valid < L_cap:
        k[:, :, n_valid:, :] = to_bf16_bits(np.float32(1000.0))
        v[:, :, n_valid:, :] = to_bf16_bits(np.float32(1000.0))
    return k, v


def gen_q(seed: int, n_layers: int, N: int, n_q_heads: int, head_dim: int) -> np.ndarray:
    """Post-rotary queries, layout [layers][N][q_heads][head_dim], bf16 bits."""
    return normal_bf16(rng(seed, 2), (n_layers, N, n_q_heads, head_dim))


def gen_lm_head(seed: int, vocab: int, d_model: int, std: float = 0.02) -> np.ndarray:
    """LM-head weight, nn.Linear layout [vocab][d_model], bf16 bits."""
    return normal_bf16(rng(seed, 3), (vocab, d_model), std)


def gen_hidden_pool(seed: int, rows: int, d_model: int) -> np.ndarray:
    """Pool of final hidden rows ~N(0,1), bf16 bits, [rows][d_model]."""
    return normal_bf16(rng(seed, 4), (rows, d_model))


def gen_drafts(seed: int, parent, argmax_of_node, vocab: int, p_match: float) -> np.ndarray:
    """Draft tokens for each node.

    Non-root node i copies the target argmax of its parent with probability
    p_match, else takes a token drawn uniformly from the other vocab-1 ids.
    ``argmax_of_node`` is the greedy target token per node, supplied by the
    caller.  The root's entry is 0 and is ignored by acceptance."""
    g = rng(seed, 5)
    n = len(parent)
    drafts = np.zeros(n, dtype=np.int32)
    coin = g.random(n)
    other = g.integers(0, vocab - 1, size=n)
    for i in range(1, n):
        a = int(argmax_of_node[parent[i]])
        if coin[i] < p_match:
            drafts[i] = a
        else:
            o = int(other[i])
            drafts[i] = o if o < a else o + 1
    return drafts


def ar1_entropy_trace(seed: int, steps: int, mu=2.0, phi=0.9, sigma=0.35, hmax=None) -> np.ndarray:
    """AR(1) entropy trace H_t = mu + phi (H_{t-1} - mu) + sigma eps_t, clipped to [0, hmax]."""
    g = rng(seed, 6)
    eps = g.standard_normal(steps)
    h = np.empty(steps)
    prev = mu
    for t in range(steps):
        prev = mu + phi * (prev - mu) + sigma * eps[t]
        h[t] = prev
    hi = np.inf if hmax is None else hmax
    return np.clip(h, 0.0, hi)


# --------------------------------------------------------------------------
# device-side generation for the large workloads (torch's Philox CUDA generator)
# --------------------------------------------------------------------------


def device_normal_bf16_(out, seed: int, std: float = 1.0, chunk_rows: int = 1 << 16):
    """Fill a bf16 torch tensor (any device) in place with N(0, std^2), seeded.

    The tensor is processed as rows of its last dimension in chunks so that
    the float32 temporaries stay small."""
    import torch

    flat = out.view(-1, out.shape[-1])
    g = torch.Generator(device=out.device)
    g.manual_seed(int(seed))
    for r0 in range(0, flat.shape[0], chunk_rows):
        r1 = min(flat.shape[0], r0 + chunk_rows)
        tmp = torch.randn((r1 - r0, flat.shape[1]), generator=g, device=out.device, dtype=torch.float32)
        if std != 1.0:
            tmp.mul_(std)
        flat[r0:r1].copy_(tmp)
    return out
