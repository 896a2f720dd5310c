"""lm_head_stats_noalloc: the LM head for callers that cannot allocate device
memory (a host framework that owns every allocation, a sandbox without
cudaMalloc).  Its scratch is the library's built-in array instead of a caller
workspace; its outputs must match lm_head_stats on the same inputs, call after
call, although the array keeps the previous call's contents, and they must
match the fp64 oracle at the tolerances of the other LM-head parity tests.

This file sorts last so that a run stopping at the first failure has already
run every other test; it also passes alone in a fresh process.
"""
import time

import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, gap_filtered_hidden
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).view(torch.int16).view(torch.bfloat16).cuda()


@pytest.fixture(scope="module")
def built():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)


def _outs(R):
    return (torch.full((R,), -1, dtype=torch.int32, device="cuda"),
            torch.full((R,), -1.0, dtype=torch.float32, device="cuda"),
            torch.full((R,), -1.0, dtype=torch.float32, device="cuda"))


def _host(o):
    return tuple(x.cpu().numpy() for x in o)


def test_noalloc_matches_workspace_entry_point_and_oracle(built):
    """Shapes in the order widest plan first, then a small one, then the 7B
    shape, so that partials and counters a larger plan left in the shared array
    could leak into the smaller calls that follow.  Each shape: the workspace
    entry point once, the no-alloc variant twice back to back; the no-alloc
    outputs must equal the workspace entry point's bit for bit (same kernel,
    same plan) and the oracle's (argmax exact on rows with a clear top-2 gap,
    top-1 and entropy within 1e-3)."""
    for R, D, V in [(256, 64, 200000), (7, 256, 1000), (64, 4096, 32000)]:
        W_h = synth.gen_lm_head(31 + V, V, D)
        h_h, am_ref, t1_ref, en_ref = gap_filtered_hidden(77 + R, R, W_h)
        W, h = _dev(W_h), _dev(h_h)
        ws_out = _outs(R)
        ws = tv.make_workspace(tv.tb_workspace_size(R, 0, 0, 0, 0, V, 0))
        tv.lm_head_stats(h, W, *ws_out, ws)
        torch.cuda.synchronize()
        ref = _host(ws_out)
        for call in range(2):
            o = _outs(R)
            tv.lm_head_stats_noalloc(h, W, *o)
            assert tv.lm_head_stats_noalloc_status() == tv.TB_OK
            got = _host(o)
            for x, y in zip(got, ref):
                assert np.array_equal(x, y), f"R={R} V={V} call {call}: differs from lm_head_stats"
            assert np.array_equal(got[0], am_ref), f"R={R} V={V}: argmax vs oracle"
            assert np.abs(got[1] - t1_ref).max() <= STAT_TOL, f"R={R} V={V}: top1 vs oracle"
            assert np.abs(got[2] - en_ref).max() <= STAT_TOL, f"R={R} V={V}: entropy vs oracle"


@pytest.mark.parametrize("R", [7, 232])
def test_noalloc_timeout_is_reported_and_next_call_recovers(built, R):
    """A bounded device wait that runs out (the TB_DEBUG_EXPIRE_WAIT test hook:
    the epilogue waits on a barrier nothing arrives on) leaves the outputs
    unwritten and shows only in lm_head_stats_noalloc_status; the next call
    clears the status word and computes the right result.  7 rows run the
    plan of independent CTAs, 232 rows the CTA-pair plan, whose CTAs give up
    together and drain each other's copies before they exit."""
    D, V = 256, 1000
    W_h = synth.gen_lm_head(5, V, D)
    h_h, am_ref, t1_ref, en_ref = gap_filtered_hidden(6, R, W_h)
    W, h = _dev(W_h), _dev(h_h)
    o = _outs(R)
    t0 = time.time()
    tv.lm_head_stats_noalloc(h, W, *o, flags=tv.TB_DEBUG_EXPIRE_WAIT)
    assert tv.lm_head_stats_noalloc_status() == tv.TB_ETIMEOUT
    assert time.time() - t0 < 20.0
    assert o[0].cpu().tolist() == [-1] * R
    o = _outs(R)
    tv.lm_head_stats_noalloc(h, W, *o)
    assert tv.lm_head_stats_noalloc_status() == tv.TB_OK
    got = _host(o)
    assert np.array_equal(got[0], am_ref)
    assert np.abs(got[1] - t1_ref).max() <= STAT_TOL and np.abs(got[2] - en_ref).max() <= STAT_TOL


def test_noalloc_argument_errors_match_workspace_entry_point(built):
    """Both entry points reject the same inputs with the same codes."""
    W = torch.zeros((100, 64), dtype=torch.bfloat16, device="cuda")
    h = torch.zeros((300, 64), dtype=torch.bfloat16, device="cuda")
    o = _outs(300)
    ws = tv.make_workspace(tv.tb_workspace_size(256, 0, 0, 0, 0, 100, 0))
    codes = []
    for fn in (lambda: tv.lm_head_stats(h, W, *o, ws), lambda: tv.lm_head_stats_noalloc(h, W, *o)):
        with pytest.raises(tv.TreeVerifyError) as ei:
            fn()
        codes.append(ei.value.status)
    assert codes == [tv.TB_EUNSUPPORTED, tv.TB_EUNSUPPORTED]
    with pytest.raises(tv.TreeVerifyError) as ei:
        tv.lm_head_stats_noalloc(h[:4], W, *[x[:4] for x in o], flags=1)
    assert ei.value.status == tv.TB_EINVAL
