"""The Python binding's marshalling, without a GPU: every wrapper is called
against a stand-in library that checks each C call's argument count against
the signature the binding declares (and returns TB_OK), so a wrapper that
passes the wrong arguments fails here rather than on the GPU."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2606_27550_gb300 as tv


class _Fn:
    def __init__(self, name, argtypes):
        self.name, self.argtypes, self.calls = name, argtypes, []

    def __call__(self, *args):
        assert len(args) == len(self.argtypes), f"{self.name}: {len(args)} arguments, declared {len(self.argtypes)}"
        self.calls.append(args)
        return 0


class _FakeLib:
    def __init__(self, real_sigs):
        for name, argtypes in real_sigs.items():
            setattr(self, name, _Fn(name, argtypes))

    def tb_last_error(self):
        return b""


@pytest.fixture
def fake(monkeypatch):
    # the declared signatures, read from the binding's loader without loading the library
    sigs = {}

    class _Rec:
        def __getattr__(self, name):
            f = type("F", (), {})()
            sigs[name] = f
            return f

    src = tv.load.__code__
    assert src is not None
    import inspect

    text = inspect.getsource(tv.load)
    start = text.index("sig = {")
    body = text[start:text.index("}", start) + 1]
    P, i32, i64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t
    table = eval(body[len("sig = "):], {"P": P, "i32": i32, "i64": i64, "sz": sz, "ctypes": ctypes})
    lib = _FakeLib(table)
    monkeypatch.setattr(tv, "_lib", lib)
    monkeypatch.setattr(tv, "load", lambda path=None: lib)
    return lib


class _Bank:
    handle = 1


def test_every_wrapper_marshals_its_declared_arguments(fake):
    t = lambda *shape, dt=torch.bfloat16: torch.zeros(shape, dtype=dt)  # noqa: E731
    bank = _Bank()
    kv = tv.KvCache(t(1, 2, 16, 128), t(1, 2, 16, 128), 4, rope_theta=10000.0)
    ws = torch.zeros(64, dtype=torch.uint8)
    res = torch.zeros(tv.RESULT_INTS, dtype=torch.int32)
    i32 = lambda *n: torch.zeros(n, dtype=torch.int32)  # noqa: E731
    f32 = lambda *n: torch.zeros(n, dtype=torch.float32)  # noqa: E731
    q, h, W = t(1, 3, 4, 128), t(3, 64), t(10, 64)
    s = 0  # a raw stream handle
    tv.tree_attention(bank, 0, kv, q, q, ws, stream=s)
    tv.lm_head_stats(h, W, i32(3), f32(3), f32(3), ws, stream=s)
    tv.greedy_accept(bank, 0, i32(3), i32(3), 10, 4, res, stream=s)
    tv.kv_compact(kv, res, stream=s)
    tv.verify_step(bank, 0, kv, q, h, W, i32(3), q, i32(3), f32(3), f32(3), res, ws, stream=s)
    tv.lm_head_stats_noalloc(h, W, i32(3), f32(3), f32(3), stream=s)
    tv.lm_head_stats_noalloc_status(stream=s)
    seq = tv.Seq(0, kv, q, i32(3), q, res)
    tv.verify_step_batched(bank, [seq, seq], t(6, 64), W, i32(6), f32(6), f32(6), ws, stream=s)
    tv.lm_head_stats_typical(bank, 0, h, W, 0.7, i32(3), i32(3), f32(3), f32(3), f32(3), f32(3), f32(3), ws, stream=s)
    tv.typical_accept(bank, 0, i32(3), i32(3), f32(3), f32(3), f32(3), 10, 4, res, 0.7, 0.09, 0.3, stream=s)
    tv.verify_step_typical(bank, 0, kv, q, h, W, i32(3), q, i32(3), f32(3), f32(3), res, ws, 0.7, 0.09, 0.3,
                           stream=s)
    tv.verify_step_batched_typical(bank, [seq], h, W, i32(3), f32(3), f32(3), ws, 0.7, 0.09, 0.3, stream=s)
    pol = tv.make_policy(tv.TB_POLICY_BINARY, tv.TB_FEATURE_ENTROPY, [0, 1], a=0.5, b=0.4)
    tv.verify_step_scheduled(bank, pol, i32(8), kv, q, h, W, i32(2, 3), q, i32(3), f32(3), f32(3), res, ws, stream=s)
    tv.spec_sample_accept(bank, 0, i32(3), f32(3, 10), f32(3), f32(3, 10), f32(6), 4, 0.7, f32(10), res, stream=s)
    tv.verify_step_sampled(bank, 0, kv, q, h, W, i32(3), f32(3, 10), f32(6), 0.7, q, i32(3), f32(3), f32(3),
                           f32(4, 10), res, ws, stream=s)
    called = {n for n in tv.API if getattr(fake, n, None) is not None and getattr(getattr(fake, n), "calls", [])}
    wrapped = {"tree_attention", "lm_head_stats", "greedy_accept", "kv_compact", "verify_step",
               "lm_head_stats_noalloc", "lm_head_stats_noalloc_status", "verify_step_batched", "lm_head_stats_typical", "typical_accept",
               "verify_step_typical", "verify_step_batched_typical", "verify_step_scheduled", "spec_sample_accept",
               "verify_step_sampled"}
    assert wrapped <= called
    # the kv struct carries the rotary base
    c = fake.tree_attention.calls[0][2]._obj
    assert c.rope_theta == pytest.approx(10000.0) and c.L == 4 and c.L_cap == 16


def test_policy_keeps_its_trace_alive():
    """The library holds only the trace's address: the policy object keeps the
    tensor alive, so a trace passed inline is not freed under it."""
    import gc

    t = torch.arange(4, dtype=torch.float32)
    ptr = t.data_ptr()
    pol = tv.make_policy(tv.TB_POLICY_BINARY, tv.TB_FEATURE_TRACE, [0, 1], a=1.0, b=0.5, trace=t)
    del t
    gc.collect()
    assert pol.trace == ptr and pol._trace_ref.data_ptr() == ptr and pol.n_trace == 4


def test_kv_compact_passes_the_result_fields(fake):
    """kv_compact(kv, result) hands the C call the result block's path and
    accept_len fields: path 16 bytes in (after accept_len, bonus_token, new_L,
    status), accept_len at the start."""
    t = lambda *shape: torch.zeros(shape, dtype=torch.bfloat16)  # noqa: E731
    kv = tv.KvCache(t(1, 2, 16, 64), t(1, 2, 16, 64), 4)
    res = torch.zeros(tv.RESULT_INTS, dtype=torch.int32)
    tv.kv_compact(kv, res, stream=0)
    _, path, accept_len, _ = fake.kv_compact.calls[-1]
    assert path == res.data_ptr() + 16 and accept_len == res.data_ptr()
    p, n = torch.zeros(3, dtype=torch.int32), torch.zeros(1, dtype=torch.int32)
    tv.kv_compact_path(kv, p, n, stream=0)
    _, path, accept_len, _ = fake.kv_compact.calls[-1]
    assert path == p.data_ptr() and accept_len == n.data_ptr()
