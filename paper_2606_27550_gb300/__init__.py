"""GB300 tree-verification library: Python binding of libtreeverify.so.

Thin ctypes marshalling over the C ABI declared in include/treeverify.h; the
functions keep the C names.  Every step of the verification pass runs in the
library's CUDA kernels; this module only turns torch tensors into pointers
and sizes.  PyTorch provides device memory and streams.

Importing this module does not require a GPU; calling the compute entry
points does, and a missing library raises immediately (there is no CPU
fallback).
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# TB_DEBUG_BOUNDS=1 in the environment selects the debug build of the library,
# whose kernels check their global indices (build.build(debug_bounds=True))
LIB_PATH = os.path.join(_HERE, "libtreeverify_debug.so" if os.environ.get("TB_DEBUG_BOUNDS") == "1"
                        else "libtreeverify.so")

TB_OK, TB_EINVAL, TB_ENOMEM, TB_ECUDA, TB_ENOTFOUND, TB_ECAPACITY, TB_ETIMEOUT, TB_EUNSUPPORTED = (
    0, -1, -2, -3, -4, -5, -6, -7)
TB_MAX_NODES = 64
TB_NO_COMPACT = 1
TB_DEBUG_EXPIRE_WAIT = 1 << 30
RESULT_INTS = 4 + TB_MAX_NODES  # sizeof(tb_result) / 4

API = ("tb_canonicalize", "tb_create", "tb_add_topology", "tb_get_topology", "tb_destroy", "tb_workspace_size",
       "tb_workspace_init", "tb_workspace_status", "tree_attention", "lm_head_stats", "greedy_accept",
       "kv_compact", "verify_step", "verify_step_batched", "lm_head_stats_noalloc", "lm_head_stats_noalloc_status",
       "tb_last_error",
       "tb_schedule_hysteretic_ladder", "tb_schedule_binary", "tb_schedule_threshold_ladder",
       "lm_head_stats_typical", "typical_accept", "verify_step_typical", "verify_step_batched_typical",
       "verify_step_scheduled", "spec_sample_accept", "verify_step_sampled", "tb_debug_bounds_violations",
       "tb_debug_bounds_build", "tb_launch_count")


class TreeVerifyError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        super().__init__(f"{where} failed ({status}): {message}")
        self.status = status


class TbKv(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("layer_stride", ctypes.c_int64),
                ("head_stride", ctypes.c_int64), ("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("L", ctypes.c_int32), ("L_cap", ctypes.c_int32),
                ("rope_theta", ctypes.c_float)]


class TbSeq(ctypes.Structure):
    _fields_ = [("bank_id", ctypes.c_int32), ("reserved", ctypes.c_int32), ("kv", TbKv), ("q", ctypes.c_void_p),
                ("draft_tokens", ctypes.c_void_p), ("attn_out", ctypes.c_void_p), ("result", ctypes.c_void_p)]


class TbTypical(ctypes.Structure):
    _fields_ = [("temperature", ctypes.c_float), ("eps", ctypes.c_float), ("alpha", ctypes.c_float),
                ("reserved", ctypes.c_int32)]


TB_POLICY_HYSTERETIC_LADDER, TB_POLICY_BINARY, TB_POLICY_THRESHOLD_LADDER = 0, 1, 2
TB_FEATURE_TRACE, TB_FEATURE_PATH_VALUE, TB_FEATURE_ENTROPY = 0, 1, 2
STATE_INTS = 8  # sizeof(tb_state) / 4


class TbPolicy(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("feature", ctypes.c_int32), ("n_rungs", ctypes.c_int32),
                ("bank_ids", ctypes.c_int32 * 8), ("a", ctypes.c_float), ("b", ctypes.c_float),
                ("edges", ctypes.c_float * 7), ("trace", ctypes.c_void_p), ("n_trace", ctypes.c_int32),
                ("n_heads", ctypes.c_int32), ("node_stride", ctypes.c_int32)]


# the paper's verification settings (temperature, posterior threshold, mixing coefficient)
PAPER_TYPICAL = (0.7, 0.09, 0.3)

TB_MAX_BATCH = 16

_lib = None


def load(path: str = LIB_PATH):
    """Loads libtreeverify.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with paper_2606_27550_gb300.build.build()")
    lib = ctypes.CDLL(path)
    P, i32, i64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t
    sig = {
        "tb_canonicalize": [P, i32, P, P, P, P],
        "tb_create": [P, i32, i32],
        "tb_add_topology": [P, P, i32, P, P],
        "tb_get_topology": [P, i32, P, P, P, P],
        "tb_destroy": [P],
        "tb_workspace_size": [i32, i32, i32, i32, i32, i32, i32],
        "tb_workspace_init": [P, sz, P],
        "tb_workspace_status": [P, P],
        "tree_attention": [P, i32, P, i32, i32, P, i32, P, P, sz, P],
        "lm_head_stats": [P, i32, P, i32, i32, P, P, P, P, sz, P],
        "greedy_accept": [P, i32, P, P, i32, i32, P, P],
        "kv_compact": [P, P, P, P],
        "verify_step": [P, i32, P, P, i32, P, P, i32, i32, P, P, P, P, P, P, P, sz, i32, P],
        "lm_head_stats_noalloc": [P, i32, P, i32, i32, P, P, P, i32, P],
        "lm_head_stats_noalloc_status": [P, P],
        "tb_debug_bounds_violations": [P],
        "tb_debug_bounds_build": [],
        "tb_launch_count": [P],
        "verify_step_batched": [P, i32, P, i32, P, P, i32, i32, P, P, P, P, sz, i32, P],
        "tb_last_error": [],
        "lm_head_stats_typical": [P, i32, P, P, i32, i32, ctypes.c_float, P, P, P, P, P, P, P, P, sz, P],
        "typical_accept": [P, i32, P, P, P, P, P, i32, i32, P, P, P],
        "verify_step_typical": [P, i32, P, P, i32, P, P, i32, i32, P, P, P, P, P, P, P, P, sz, i32, P],
        "verify_step_batched_typical": [P, i32, P, i32, P, P, i32, i32, P, P, P, P, P, sz, i32, P],
        "verify_step_scheduled": [P, P, P, P, P, i32, P, P, i32, i32, P, P, P, P, P, P, P, sz, i32, P],
        "spec_sample_accept": [P, i32, P, P, P, P, P, i32, i32, ctypes.c_float, P, P, P],
        "verify_step_sampled": [P, i32, P, P, i32, P, P, i32, i32, P, P, P, ctypes.c_float, P, P, P, P, P, P, P, sz,
                                i32, P],
    }
    for name, args in sig.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ctypes.c_int
    d = ctypes.c_double
    lib.tb_schedule_hysteretic_ladder.argtypes = [i32, i32, d, d, d]
    lib.tb_schedule_binary.argtypes = [i32, d, d, d]
    lib.tb_schedule_threshold_ladder.argtypes = [d, P, i32]
    for f in (lib.tb_schedule_hysteretic_ladder, lib.tb_schedule_binary, lib.tb_schedule_threshold_ladder):
        f.restype = ctypes.c_int
    lib.tb_workspace_size.restype = ctypes.c_size_t
    lib.tb_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(rc: int, where: str):
    if rc != TB_OK:
        raise TreeVerifyError(rc, where, load().tb_last_error().decode())


def _ptr(t) -> int | None:
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch

        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# --------------------------------------------------------------------- topologies


def tb_canonicalize(parent):
    """(order, bfs_parent, depth, anc) of a parent array (pure host)."""
    parent = np.ascontiguousarray(parent, dtype=np.int32)
    n = len(parent)
    order = np.zeros(n, np.int32)
    bp = np.zeros(n, np.int32)
    depth = np.zeros(n, np.int32)
    anc = np.zeros(n, np.uint64)
    _check(load().tb_canonicalize(_ptr(parent), n, _ptr(order), _ptr(bp), _ptr(depth), _ptr(anc)), "tb_canonicalize")
    return order, bp, depth, anc


class Bank:
    """A TopologyBank on one device (tb_create / tb_add_topology / tb_destroy)."""

    def __init__(self, max_topologies: int = 64, device: int = 0):
        h = ctypes.c_void_p()
        _check(load().tb_create(ctypes.byref(h), max_topologies, device), "tb_create")
        self.handle = h
        self.device = device
        self.sizes: list[int] = []

    def add(self, parent):
        """Adds a topology; returns (bank_id, order) with order[canonical] = caller index."""
        parent = np.ascontiguousarray(parent, dtype=np.int32)
        out = ctypes.c_int()
        order = np.zeros(len(parent), np.int32)
        _check(load().tb_add_topology(self.handle, _ptr(parent), len(parent), ctypes.byref(out), _ptr(order)),
               "tb_add_topology")
        self.sizes.append(len(parent))
        return out.value, order

    def get(self, bank_id: int):
        n = ctypes.c_int()
        parent = np.zeros(TB_MAX_NODES, np.int32)
        depth = np.zeros(TB_MAX_NODES, np.int32)
        anc = np.zeros(TB_MAX_NODES, np.uint64)
        _check(load().tb_get_topology(self.handle, bank_id, ctypes.byref(n), _ptr(parent), _ptr(depth), _ptr(anc)),
               "tb_get_topology")
        k = n.value
        return parent[:k].copy(), depth[:k].copy(), anc[:k].copy()

    def n_nodes(self, bank_id: int) -> int:
        return self.sizes[bank_id]

    def close(self):
        if self.handle:
            _check(load().tb_destroy(self.handle), "tb_destroy")
            self.handle = None

    def __del__(self):  # pragma: no cover
        try:
            self.close()
        except Exception:
            pass


# --------------------------------------------------------------------- KV cache, workspace, result


@dataclass
class KvCache:
    """bf16 K and V caches shaped [n_layers][n_kv_heads][L_cap][head_dim]."""

    k: object
    v: object
    L: int
    rope_theta: float = 0.0  # > 0: the call rotary-embeds q and the tree keys at L + depth

    def as_c(self) -> TbKv:
        n_layers, n_kv_heads, L_cap, head_dim = self.k.shape
        s = self.k.stride()
        return TbKv(self.k.data_ptr(), self.v.data_ptr(), s[0], s[1], n_layers, n_kv_heads, head_dim, self.L, L_cap,
                    float(self.rope_theta))


def tb_workspace_size(max_rows: int, n_layers: int, n_kv_heads: int, n_q_heads: int, head_dim: int, vocab: int,
                      device: int = -1) -> int:
    return int(load().tb_workspace_size(max_rows, n_layers, n_kv_heads, n_q_heads, head_dim, vocab, device))


def make_workspace(nbytes: int, device="cuda"):
    """Zero-filled device workspace (torch uint8)."""
    import torch

    return torch.zeros(nbytes, dtype=torch.uint8, device=device)


def tb_workspace_init(ws, stream=None):
    _check(load().tb_workspace_init(_ptr(ws), ws.numel(), _stream(stream)), "tb_workspace_init")


def tb_workspace_status(ws) -> int:
    st = ctypes.c_int32()
    _check(load().tb_workspace_status(_ptr(ws), ctypes.byref(st)), "tb_workspace_status")
    return st.value


def make_result(device="cuda"):
    """Device buffer for one tb_result (int32[68])."""
    import torch

    return torch.zeros(RESULT_INTS, dtype=torch.int32, device=device)


def parse_result(res) -> dict:
    """The tb_result block (a device or host tensor, or a sequence of ints) as a dict."""
    if hasattr(res, "cpu"):
        r = res.cpu().tolist()  # one copy and one conversion (iterating a tensor makes a tensor per element)
    else:
        r = [int(x) for x in res]
    k = r[0]
    return {"accept_len": k, "bonus_token": r[1], "new_L": r[2], "status": r[3], "path": r[4:4 + k]}


# --------------------------------------------------------------------- the pass


def tree_attention(bank: Bank, bank_id: int, kv: KvCache, q, out, ws, layer_begin: int = 0, n_layers: int | None = None,
                   stream=None):
    """q, out: bf16 [n_layers][N][n_q_heads][head_dim]."""
    c = kv.as_c()
    nl = c.n_layers - layer_begin if n_layers is None else n_layers
    _check(load().tree_attention(bank.handle, bank_id, ctypes.byref(c), layer_begin, nl, _ptr(q), q.shape[2],
                                 _ptr(out), _ptr(ws), ws.numel(), _stream(stream)), "tree_attention")


def lm_head_stats(hidden, lm_head, argmax, top1, entropy, ws, stream=None):
    """hidden bf16 [R][d_model]; lm_head bf16 [V][d_model]; outputs [R]."""
    R, D = hidden.shape
    _check(load().lm_head_stats(_ptr(hidden), R, _ptr(lm_head), D, lm_head.shape[0], _ptr(argmax), _ptr(top1),
                                _ptr(entropy), _ptr(ws), ws.numel(), _stream(stream)), "lm_head_stats")


def greedy_accept(bank: Bank, bank_id: int, draft, argmax, vocab: int, L: int, result, stream=None):
    _check(load().greedy_accept(bank.handle, bank_id, _ptr(draft), _ptr(argmax), vocab, L, _ptr(result),
                                _stream(stream)), "greedy_accept")


def kv_compact_path(kv: KvCache, path, accept_len, stream=None):
    """KV-cache update from a device path (int32 [accept_len]) and a device
    accept_len (int32 [1])."""
    c = kv.as_c()
    _check(load().kv_compact(ctypes.byref(c), _ptr(path), _ptr(accept_len), _stream(stream)), "kv_compact")


def kv_compact(kv: KvCache, result, stream=None):
    """KV-cache update from a device result block (greedy_accept's): its path
    and accept_len fields."""
    kv_compact_path(kv, result[4:], result[:1], stream)


def verify_step(bank: Bank, bank_id: int, kv: KvCache, q, hidden, lm_head, draft, attn_out, argmax, top1, entropy,
                result, ws, flags: int = 0, stream=None):
    c = kv.as_c()
    _check(load().verify_step(bank.handle, bank_id, ctypes.byref(c), _ptr(q), q.shape[2], _ptr(hidden),
                              _ptr(lm_head), hidden.shape[1], lm_head.shape[0], _ptr(draft), _ptr(attn_out),
                              _ptr(argmax), _ptr(top1), _ptr(entropy), _ptr(result), _ptr(ws), ws.numel(), flags,
                              _stream(stream)), "verify_step")


def lm_head_stats_noalloc(hidden, lm_head, argmax, top1, entropy, flags: int = 0, stream=None):
    """lm_head_stats with the library's built-in scratch array instead of a
    caller workspace, for callers that cannot allocate device memory."""
    R, D = hidden.shape
    _check(load().lm_head_stats_noalloc(_ptr(hidden), R, _ptr(lm_head), D, lm_head.shape[0], _ptr(argmax),
                                        _ptr(top1), _ptr(entropy), flags, _stream(stream)), "lm_head_stats_noalloc")


def tb_debug_bounds_violations() -> int:
    """Failed index checks of the debug build's kernels since the last call
    (0 in a normal build); synchronises the device."""
    n = ctypes.c_uint32(0)
    _check(load().tb_debug_bounds_violations(ctypes.byref(n)), "tb_debug_bounds_violations")
    return int(n.value)


def tb_debug_bounds_build() -> bool:
    return bool(load().tb_debug_bounds_build())


def tb_launch_count() -> int:
    """Kernels the library has enqueued in this process (host-side count; a
    CUDA graph's replays are not counted again)."""
    n = ctypes.c_uint64(0)
    _check(load().tb_launch_count(ctypes.byref(n)), "tb_launch_count")
    return int(n.value)


def lm_head_stats_noalloc_status(stream=None) -> int:
    """Device-detected status (TB_OK or TB_ETIMEOUT) of the last
    lm_head_stats_noalloc call on `stream`; waits for the stream."""
    st = ctypes.c_int32(0)
    _check(load().lm_head_stats_noalloc_status(ctypes.byref(st), _stream(stream)), "lm_head_stats_noalloc_status")
    return st.value


@dataclass
class Seq:
    """One sequence of verify_step_batched."""

    bank_id: int
    kv: KvCache
    q: object
    draft_tokens: object
    attn_out: object
    result: object

    def as_c(self) -> TbSeq:
        return TbSeq(self.bank_id, 0, self.kv.as_c(), _ptr(self.q), _ptr(self.draft_tokens), _ptr(self.attn_out),
                     _ptr(self.result))


def verify_step_batched(bank: Bank, seqs, hidden, lm_head, argmax, top1, entropy, ws, flags: int = 0, stream=None):
    """hidden bf16 [sum N_b][d_model] (sequence 0 first); argmax/top1/entropy [sum N_b]."""
    arr = (TbSeq * len(seqs))(*[s.as_c() for s in seqs])
    _check(load().verify_step_batched(bank.handle, len(seqs), arr, seqs[0].q.shape[2], _ptr(hidden), _ptr(lm_head),
                                      hidden.shape[1], lm_head.shape[0], _ptr(argmax), _ptr(top1), _ptr(entropy),
                                      _ptr(ws), ws.numel(), flags, _stream(stream)), "verify_step_batched")


# --------------------------------------------------------------------- typical acceptance


def _typical(temperature: float, eps: float, alpha: float) -> TbTypical:
    return TbTypical(float(temperature), float(eps), float(alpha), 0)


def lm_head_stats_typical(bank: Bank, bank_id: int, hidden, lm_head, temperature: float, draft, argmax, top1, entropy,
                          logz_t, entropy_t, draft_logit, ws, stream=None):
    """hidden bf16 [N][d_model] (the tree's rows); every output [N]."""
    _check(load().lm_head_stats_typical(bank.handle, bank_id, _ptr(hidden), _ptr(lm_head), hidden.shape[1],
                                        lm_head.shape[0], float(temperature), _ptr(draft), _ptr(argmax), _ptr(top1),
                                        _ptr(entropy), _ptr(logz_t), _ptr(entropy_t), _ptr(draft_logit), _ptr(ws),
                                        ws.numel(), _stream(stream)), "lm_head_stats_typical")


def typical_accept(bank: Bank, bank_id: int, draft, argmax, logz_t, entropy_t, draft_logit, vocab: int, L: int,
                   result, temperature: float, eps: float, alpha: float, stream=None):
    t = _typical(temperature, eps, alpha)
    _check(load().typical_accept(bank.handle, bank_id, _ptr(draft), _ptr(argmax), _ptr(logz_t), _ptr(entropy_t),
                                 _ptr(draft_logit), vocab, L, ctypes.byref(t), _ptr(result), _stream(stream)),
           "typical_accept")


def verify_step_typical(bank: Bank, bank_id: int, kv: KvCache, q, hidden, lm_head, draft, attn_out, argmax, top1,
                        entropy, result, ws, temperature: float, eps: float, alpha: float, flags: int = 0,
                        stream=None):
    c = kv.as_c()
    t = _typical(temperature, eps, alpha)
    _check(load().verify_step_typical(bank.handle, bank_id, ctypes.byref(c), _ptr(q), q.shape[2], _ptr(hidden),
                                      _ptr(lm_head), hidden.shape[1], lm_head.shape[0], _ptr(draft), _ptr(attn_out),
                                      _ptr(argmax), _ptr(top1), _ptr(entropy), ctypes.byref(t), _ptr(result),
                                      _ptr(ws), ws.numel(), flags, _stream(stream)), "verify_step_typical")


def verify_step_batched_typical(bank: Bank, seqs, hidden, lm_head, argmax, top1, entropy, ws, temperature: float,
                                eps: float, alpha: float, flags: int = 0, stream=None):
    arr = (TbSeq * len(seqs))(*[s.as_c() for s in seqs])
    t = _typical(temperature, eps, alpha)
    _check(load().verify_step_batched_typical(bank.handle, len(seqs), arr, seqs[0].q.shape[2], _ptr(hidden),
                                              _ptr(lm_head), hidden.shape[1], lm_head.shape[0], _ptr(argmax),
                                              _ptr(top1), _ptr(entropy), ctypes.byref(t), _ptr(ws), ws.numel(),
                                              flags, _stream(stream)), "verify_step_batched_typical")


# --------------------------------------------------------------------- speculative sampling


def spec_sample_accept(bank: Bank, bank_id: int, draft, logits, logz_t, draft_probs, uniforms, L: int,
                       temperature: float, scratch, result, stream=None):
    """logits, draft_probs float [N][V]; logz_t [N]; uniforms [2N]; scratch [V]."""
    _check(load().spec_sample_accept(bank.handle, bank_id, _ptr(draft), _ptr(logits), _ptr(logz_t),
                                     _ptr(draft_probs), _ptr(uniforms), logits.shape[1], L, float(temperature),
                                     _ptr(scratch), _ptr(result), _stream(stream)), "spec_sample_accept")


def verify_step_sampled(bank: Bank, bank_id: int, kv: KvCache, q, hidden, lm_head, draft, draft_probs, uniforms,
                        temperature: float, attn_out, argmax, top1, entropy, logits, result, ws, flags: int = 0,
                        stream=None):
    """logits: float [N + 1][V] scratch (rows 0..N-1 receive the target logits)."""
    c = kv.as_c()
    _check(load().verify_step_sampled(bank.handle, bank_id, ctypes.byref(c), _ptr(q), q.shape[2], _ptr(hidden),
                                      _ptr(lm_head), hidden.shape[1], lm_head.shape[0], _ptr(draft),
                                      _ptr(draft_probs), _ptr(uniforms), float(temperature), _ptr(attn_out),
                                      _ptr(argmax), _ptr(top1), _ptr(entropy), _ptr(logits), _ptr(result), _ptr(ws),
                                      ws.numel(), flags, _stream(stream)), "verify_step_sampled")


# --------------------------------------------------------------------- device-driven loop


def make_policy(kind: int, feature: int, bank_ids, a: float = 0.0, b: float = 0.0, edges=(), trace=None,
                n_heads: int = 0, node_stride: int = 0) -> TbPolicy:
    """tb_policy; `trace` is a device float tensor, which the returned policy
    keeps alive (the library holds only its address)."""
    pol = TbPolicy()
    pol.kind, pol.feature, pol.n_rungs = kind, feature, len(bank_ids)
    for i, x in enumerate(bank_ids):
        pol.bank_ids[i] = int(x)
    pol.a, pol.b = float(a), float(b)
    for i, x in enumerate(edges):
        pol.edges[i] = float(x)
    if trace is not None:
        pol.trace = _ptr(trace)
        pol._trace_ref = trace
        pol.n_trace = trace.numel() // max(1, n_heads) if feature == TB_FEATURE_PATH_VALUE else trace.numel()
    pol.n_heads = n_heads
    pol.node_stride = node_stride
    return pol


def make_state(rung: int, L: int, device="cuda"):
    """A device tb_state (int32 words) at the given rung and prefix length."""
    import torch

    t = torch.zeros(STATE_INTS, dtype=torch.int32)
    t[0], t[1] = rung, L
    return t.to(device)


def parse_state(st) -> dict:
    import numpy as np

    h = st.cpu().numpy()
    return {"rung": int(h[0]), "L": int(h[1]), "step": int(h[2]), "feature": float(h[3:4].view(np.float32)[0]),
            "accept_len": int(h[4])}


def verify_step_scheduled(bank: Bank, policy: TbPolicy, state, kv: KvCache, q, hidden, lm_head, drafts, attn_out,
                          argmax, top1, entropy, result, ws, flags: int = 0, stream=None):
    """q / attn_out [n_layers][N_max][Hq][head_dim]; hidden [N_max][d_model]; drafts [n_rungs][N_max]."""
    c = kv.as_c()
    _check(load().verify_step_scheduled(bank.handle, ctypes.byref(policy), _ptr(state), ctypes.byref(c), _ptr(q),
                                        q.shape[2], _ptr(hidden), _ptr(lm_head), hidden.shape[1], lm_head.shape[0],
                                        _ptr(drafts), _ptr(attn_out), _ptr(argmax), _ptr(top1), _ptr(entropy),
                                        _ptr(result), _ptr(ws), ws.numel(), flags, _stream(stream)),
           "verify_step_scheduled")


# --------------------------------------------------------------------- per-step tree selection


def tb_schedule_hysteretic_ladder(current: int, n_trees: int, feature: float, up_below: float,
                                  down_above: float) -> int:
    return int(load().tb_schedule_hysteretic_ladder(current, n_trees, feature, up_below, down_above))


def tb_schedule_binary(aggressive: int, s: float, tau_on: float, tau_off: float) -> int:
    return int(load().tb_schedule_binary(int(aggressive), s, tau_on, tau_off))


def tb_schedule_threshold_ladder(s: float, edges) -> int:
    e = np.ascontiguousarray(edges, dtype=np.float64)
    return int(load().tb_schedule_threshold_ladder(s, _ptr(e), len(e) + 1))
