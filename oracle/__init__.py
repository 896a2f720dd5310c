"""fp64 CPU oracle of the tree-verification pass (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU baseline
leg import this package.  The product library never does.

``oracle.c`` holds the arithmetic (tree sets, attention, LM head, greedy and
typical acceptance); this module compiles it with gcc, loads it with ctypes and adds
the KV compaction, which is a plain gather written out below.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, OpenMP, -O2, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".{os.getpid()}.tmp"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i32, i64 = ctypes.c_int, ctypes.c_int64
            lib.oracle_tree.argtypes = [P, i32, P, P]
            lib.oracle_tree_attention.argtypes = [P, P, P, i64, i32, i32, i32, i32, i32, P, P]
            lib.oracle_lm_head.argtypes = [P, P, i32, i32, i32, P, P, P, P, P]
            lib.oracle_accept.argtypes = [P, i32, P, P, P, P, P]
            lib.oracle_num_threads.argtypes = []
            lib.oracle_set_num_threads.argtypes = [i32]
            lib.oracle_set_num_threads.restype = ctypes.c_int
            d = ctypes.c_double
            lib.oracle_typical_accept.argtypes = [P, i32, P, P, i32, d, d, d, P, P, P, P, P, P]
            lib.oracle_typical_accept.restype = ctypes.c_int
            lib.oracle_tempered_stats.argtypes = [P, i32, i32, d, P, P]
            lib.oracle_spec_sample.argtypes = [P, i32, P, P, P, i32, d, P, P, P, P, P, P]
            lib.oracle_spec_sample.restype = ctypes.c_int
            lib.oracle_rope.argtypes = [P, i32, i32, P, d, P]
            lib.oracle_rope.restype = ctypes.c_int
            lib.oracle_tree_attention_rope.argtypes = [P, P, P, i64, i32, i32, i32, i32, i32, P, d, P, P]
            lib.oracle_tree_attention_rope.restype = ctypes.c_int
            lib.oracle_tempered_stats.restype = ctypes.c_int
            for f in (lib.oracle_tree, lib.oracle_tree_attention, lib.oracle_lm_head,
                      lib.oracle_accept, lib.oracle_num_threads):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def set_num_threads(n: int) -> int:
    """Threads of the oracle's OpenMP loops from now on; returns the previous count."""
    return int(_load().oracle_set_num_threads(int(n)))


def tree(parent):
    """(depth[n], in_anc[n][n] bool) for a parent array rooted at node 0."""
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    n = len(parent)
    depth = np.zeros(n, dtype=np.int32)
    in_anc = np.zeros((n, n), dtype=np.uint8)
    if _load().oracle_tree(_ptr(parent), n, _ptr(depth), _ptr(in_anc)) != 0:
        raise ValueError("not a tree rooted at node 0")
    return depth, in_anc.astype(bool)


def tree_attention(q, k, v, L: int, parent, n_kv_heads: int | None = None):
    """One layer of tree-masked attention.

    q: [N][Hq][d] bf16 bits.  k, v: [Hkv][S][d] bf16 bits with S >= L + N.
    Returns float64 [N][Hq][d]."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    N, Hq, d = q.shape
    Hkv = k.shape[0] if n_kv_heads is None else n_kv_heads
    if k.shape[1] < L + N or k.shape != v.shape or k.shape[2] != d:
        raise ValueError("bad kv shape")
    out = np.zeros((N, Hq, d), dtype=np.float64)
    rc = _load().oracle_tree_attention(_ptr(q), _ptr(k), _ptr(v), k.shape[1] * d, L, N, Hq, Hkv, d,
                                        _ptr(parent), _ptr(out))
    if rc != 0:
        raise ValueError(f"oracle_tree_attention rc={rc}")
    return out


def lm_head(hidden, W, want_logits: bool = False):
    """(argmax int32[R], top1 f64[R], entropy f64[R], gap f64[R][, logits f64[R][V]])."""
    hidden = np.ascontiguousarray(hidden, dtype=np.uint16)
    W = np.ascontiguousarray(W, dtype=np.uint16)
    R, D = hidden.shape
    V = W.shape[0]
    if W.shape[1] != D:
        raise ValueError("d_model mismatch")
    argmax = np.zeros(R, dtype=np.int32)
    top1 = np.zeros(R)
    ent = np.zeros(R)
    gap = np.zeros(R)
    logits = np.zeros((R, V)) if want_logits else None
    rc = _load().oracle_lm_head(_ptr(hidden), _ptr(W), R, D, V, _ptr(argmax), _ptr(top1), _ptr(ent),
                                _ptr(gap), _ptr(logits) if want_logits else None)
    if rc != 0:
        raise ValueError(f"oracle_lm_head rc={rc}")
    return (argmax, top1, ent, gap, logits) if want_logits else (argmax, top1, ent, gap)


def accept(parent, draft, argmax):
    """(accept_len, path list, bonus token)."""
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    draft = np.ascontiguousarray(draft, dtype=np.int32)
    argmax = np.ascontiguousarray(argmax, dtype=np.int32)
    n = len(parent)
    path = np.zeros(max(n, 1), dtype=np.int32)
    alen = np.zeros(1, dtype=np.int32)
    bonus = np.zeros(1, dtype=np.int32)
    if _load().oracle_accept(_ptr(parent), n, _ptr(draft), _ptr(argmax), _ptr(alen), _ptr(path),
                             _ptr(bonus)) != 0:
        raise ValueError("not a tree rooted at node 0")
    k = int(alen[0])
    return k, [int(x) for x in path[:k]], int(bonus[0])


def kv_compact(cache, L: int, path):
    """KV-cache update after acceptance: slot L + j takes the contents of slot
    L + path[j] for j < len(path); every other slot is unchanged.

    cache: [..., S, d] (any dtype).  Returns a new array; reads only the old one."""
    old = np.asarray(cache)
    new = old.copy()
    for j, src in enumerate(path):
        new[..., L + j, :] = old[..., L + src, :]
    return new


def typical_accept(parent, draft, logits, temperature: float, eps: float, alpha: float, detail: bool = False):
    """Typical acceptance: (accept_len, path list, bonus token[, detail dict]).

    logits: float64 [N][V], the target logits after every node.  detail adds
    per-edge margins (p - threshold) / threshold, per-node path
    log-likelihoods and per-node accepted flags."""
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    draft = np.ascontiguousarray(draft, dtype=np.int32)
    logits = np.ascontiguousarray(logits, dtype=np.float64)
    n, V = logits.shape
    if n != len(parent) or len(draft) < n:
        raise ValueError("one logit row and one draft token per node")
    path = np.zeros(max(n, 1), dtype=np.int32)
    alen = np.zeros(1, dtype=np.int32)
    bonus = np.zeros(1, dtype=np.int32)
    margin = np.zeros(n)
    loglik = np.zeros(n)
    acc = np.zeros(n, dtype=np.int32)
    if _load().oracle_typical_accept(_ptr(parent), n, _ptr(draft), _ptr(logits), V, temperature, eps, alpha,
                                     _ptr(alen), _ptr(path), _ptr(bonus), _ptr(margin), _ptr(loglik),
                                     _ptr(acc)) != 0:
        raise ValueError("bad tree, vocab or temperature")
    k = int(alen[0])
    out = (k, [int(x) for x in path[:k]], int(bonus[0]))
    if detail:
        return out + ({"margin": margin, "loglik": loglik, "accepted": acc.astype(bool)},)
    return out


def tempered_stats(logits, temperature: float):
    """(logz float64[R], entropy float64[R]) of softmax(logits / T) per row."""
    logits = np.ascontiguousarray(logits, dtype=np.float64)
    R, V = logits.shape
    logz = np.zeros(R)
    ent = np.zeros(R)
    if _load().oracle_tempered_stats(_ptr(logits), R, V, temperature, _ptr(logz), _ptr(ent)) != 0:
        raise ValueError("bad shape or temperature")
    return logz, ent


# ---------------------------------------------------------------- per-step tree selection (Sec. 4)

def path_value(p0: float, head_probs) -> float:
    """Path-value score (Sec. 4): g_d = p0 * p_1 * ... * p_d and
    s = max(p0, g_1, ..., g_D).  Evaluated in float64."""
    s = g = float(p0)
    for p in head_probs:
        g *= float(p)
        s = max(s, g)
    return s


def policy_next(kind: str, rung: int, n_rungs: int, feature: float, a: float = 0.0, b: float = 0.0, edges=()):
    """Next rung of the per-step policies (Sec. 4 "Policy"):
      'ladder'    hysteretic step ladder: one rung up when feature < a, one down
                  when feature > b, else stay (clamped to the rungs);
      'binary'    rung 1 (aggressive tree) when feature > a = tau_on, rung 0 when
                  feature <= b = tau_off, else unchanged;
      'threshold' threshold_ladder: the number of edges that are <= feature."""
    if kind == "ladder":
        if feature < a:
            return min(rung + 1, n_rungs - 1)
        if feature > b:
            return max(rung - 1, 0)
        return rung
    if kind == "binary":
        if feature > a:
            return 1
        if feature <= b:
            return 0
        return rung
    if kind == "threshold":
        k = 0
        while k < n_rungs - 1 and feature >= edges[k]:
            k += 1
        return k
    raise ValueError(kind)


# ---------------------------------------------------------------- rotary position embedding

def rope(x, pos, base: float = 10000.0):
    """Rotary embedding of bf16 rows x [rows][d] at positions pos[rows] (float64 out)."""
    x = np.ascontiguousarray(x, dtype=np.uint16)
    rows, d = x.shape
    pos = np.ascontiguousarray(pos, dtype=np.int32)
    y = np.zeros((rows, d))
    if _load().oracle_rope(_ptr(x), rows, d, _ptr(pos), base, _ptr(y)) != 0:
        raise ValueError("bad shape or base")
    return y


def tree_attention_rope(q, k, v, L: int, parent, base: float = 10000.0):
    """One layer of tree-masked attention with the rotary embedding at the tree's
    position offsets (node i at L + depth(i)); q and the tree slots of k are
    pre-rotary, the prefix keys already rotated.

    Returns (out float64 [N][Hq][d], rotated tree keys as bf16 bits [Hkv][N][d])."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    N, Hq, d = q.shape
    Hkv = k.shape[0]
    if k.shape[1] < L + N or k.shape != v.shape or k.shape[2] != d:
        raise ValueError("bad kv shape")
    out = np.zeros((N, Hq, d))
    k_rot = np.zeros((Hkv, N, d), dtype=np.uint16)
    rc = _load().oracle_tree_attention_rope(_ptr(q), _ptr(k), _ptr(v), k.shape[1] * d, L, N, Hq, Hkv, d,
                                            _ptr(parent), base, _ptr(out), _ptr(k_rot))
    if rc != 0:
        raise ValueError(f"oracle_tree_attention_rope rc={rc}")
    return out, k_rot


# ---------------------------------------------------------------- speculative sampling (Sec. 2.1)

def spec_sample(parent, draft, logits, q, temperature: float, unif, detail: bool = False):
    """Speculative sampling on the tree: (accept_len, path, token[, detail]).

    logits, q: float64 [N][V] (target logits per node; draft distribution of each
    node's children); unif: [2N] uniforms in [0, 1) (unif[c] decides child c,
    unif[N + u] draws the token after the final node u)."""
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    draft = np.ascontiguousarray(draft, dtype=np.int32)
    logits = np.ascontiguousarray(logits, dtype=np.float64)
    q = np.ascontiguousarray(q, dtype=np.float64)
    unif = np.ascontiguousarray(unif, dtype=np.float64)
    n, V = logits.shape
    if q.shape != logits.shape or len(unif) < 2 * n or len(parent) != n:
        raise ValueError("shapes")
    path = np.zeros(max(n, 1), dtype=np.int32)
    alen = np.zeros(1, dtype=np.int32)
    tok = np.zeros(1, dtype=np.int32)
    rm = np.zeros(n)
    cm = np.zeros(1)
    if _load().oracle_spec_sample(_ptr(parent), n, _ptr(draft), _ptr(logits), _ptr(q), V, temperature, _ptr(unif),
                                  _ptr(alen), _ptr(path), _ptr(tok), _ptr(rm), _ptr(cm)) != 0:
        raise ValueError("bad tree, vocab or temperature")
    k = int(alen[0])
    out = (k, [int(x) for x in path[:k]], int(tok[0]))
    if detail:
        return out + ({"ratio_margin": rm, "cdf_margin": float(cm[0])},)
    return out
