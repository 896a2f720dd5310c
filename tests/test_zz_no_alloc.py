"""lm_head_stats_noalloc: the LM head for callers that cannot allocate device
memory (a host framework that owns every allocation, a sandbox without
cudaMalloc).  Its scratch is the library's built-in array instead of a caller
workspace; its outputs must match lm_head_stats on the same inputs, call after
call, although the array keeps the previous call's contents.

This file sorts last so that a run stopping at the first failure has already
run every other test; it also passes alone in a fresh process.
"""
import numpy as np
import pytest

from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

STAT_TOL = 1e-3  # top-1 probability and entropy, as in the other parity tests


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).view(torch.int16).view(torch.bfloat16).cuda()


@pytest.fixture(scope="module")
def built():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("R,D,V", [(64, 4096, 32000), (7, 256, 1000)])
def test_noalloc_matches_workspace_entry_point(built, R, D, V):
    W = _dev(synth.gen_lm_head(31 + V, V, D))
    outs = []
    for call in range(3):  # call 0: reference entry point; calls 1, 2: no-alloc variant, back to back
        h = _dev(synth.gen_hidden_pool(77 + call, R, D)) if call == 0 else h
        am = torch.full((R,), -1, dtype=torch.int32, device="cuda")
        t1 = torch.full((R,), -1.0, dtype=torch.float32, device="cuda")
        en = torch.full((R,), -1.0, dtype=torch.float32, device="cuda")
        if call == 0:
            ws = tv.make_workspace(tv.tb_workspace_size(R, 0, 0, 0, 0, V, 0))
            tv.lm_head_stats(h, W, am, t1, en, ws)
        else:
            tv.lm_head_stats_noalloc(h, W, am, t1, en)
        torch.cuda.synchronize()
        outs.append((am.cpu().numpy(), t1.cpu().numpy(), en.cpu().numpy()))
    ref = outs[0]
    for got in outs[1:]:
        assert np.array_equal(got[0], ref[0])
        assert np.abs(got[1] - ref[1]).max() <= STAT_TOL
        assert np.abs(got[2] - ref[2]).max() <= STAT_TOL
        assert np.all(got[0] >= 0) and np.all(got[0] < V)


def test_noalloc_rejects_oversized_scratch(built):
    R, D, V = 256, 64, 200000  # needs more partial scratch than the built-in array holds
    h = torch.zeros((R, D), dtype=torch.bfloat16, device="cuda")
    W = torch.zeros((V, D), dtype=torch.bfloat16, device="cuda")
    o = torch.empty(R, dtype=torch.int32, device="cuda")
    f = torch.empty(R, dtype=torch.float32, device="cuda")
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.lm_head_stats_noalloc(h, W, o, f, f)
    assert e.value.status == tv.TB_ECAPACITY
    assert "built-in array" in str(e.value)
