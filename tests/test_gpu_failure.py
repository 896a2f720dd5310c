"""Failure detection on the GPU without a fault: a bounded device wait that
runs out.  With the TB_DEBUG_EXPIRE_WAIT test hook the LM-head kernel waits on
a barrier nothing arrives on; after about a second it records TB_ETIMEOUT,
lets its issued work retire, frees TMEM and returns.  The step's result and
the workspace status report the time-out, and after tb_workspace_init the
same context computes correct results again."""
import time

import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, make_case, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu


def test_bounded_wait_expires_and_context_recovers():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda:0")
    sh = synth.shape_c1()
    case = make_case(13, sh.parent, sh.L, 1, 4, 4, 64, 256, 1000, 0.7)
    bank = tv.Bank(4, 0)
    bid, _ = bank.add(case.parent)
    N = case.N
    ws = tv.make_workspace(tv.tb_workspace_size(N, 1, 4, 4, 64, 1000, 0), dev)

    def step(flags):
        kv = tv.KvCache(to_dev(case.k, dev), to_dev(case.v, dev), case.L)
        out = torch.empty((1, N, 4, 64), dtype=torch.bfloat16, device=dev)
        am = torch.full((N,), -7, dtype=torch.int32, device=dev)
        t1 = torch.empty(N, dtype=torch.float32, device=dev)
        en = torch.empty(N, dtype=torch.float32, device=dev)
        res = tv.make_result(dev)
        tv.verify_step(bank, bid, kv, to_dev(case.q, dev), to_dev(case.hidden, dev), to_dev(case.W, dev),
                       to_dev(case.drafts, dev), out, am, t1, en, res, ws, flags)
        torch.cuda.synchronize()
        return tv.parse_result(res), am, t1, en

    t0 = time.time()
    r, am, _, _ = step(tv.TB_DEBUG_EXPIRE_WAIT)
    took = time.time() - t0
    assert r["status"] == tv.TB_ETIMEOUT
    assert tv.tb_workspace_status(ws) == tv.TB_ETIMEOUT
    assert am.cpu().tolist() == [-7] * N  # outputs of the stopped kernel are not written
    assert took < 20.0
    # the context is still usable: re-initialise the workspace and verify normally
    tv.tb_workspace_init(ws)
    r, am, t1, en = step(0)
    assert r["status"] == tv.TB_OK and tv.tb_workspace_status(ws) == tv.TB_OK
    assert np.array_equal(am.cpu().numpy(), case.argmax)
    assert np.abs(t1.cpu().numpy() - case.top1).max() <= STAT_TOL
    ka, path, bonus = oracle.accept(case.parent, case.drafts, case.argmax)
    assert (r["accept_len"], r["path"], r["bonus_token"]) == (ka, path, bonus)
    bank.close()
