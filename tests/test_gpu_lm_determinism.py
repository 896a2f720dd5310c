"""The LM head's statistics do not depend on where its vocab tiles ran.

The kernel hands tiles out dynamically (a CTA, or CTA pair, that starts late
takes fewer), so which CTA folds which tile changes from launch to launch;
each tile's statistics go to a slot of their own and the row merge combines
the slots in a fixed order.  Here the LM head runs alone, then several times
right behind a long attention launch on another stream that holds the SMs and
releases them one by one, and every output must be identical bit for bit: the
two-CTAs-per-SM plan (26 rows), the CTA-pair plan (232 rows) and the tempered
sums of typical acceptance (64 rows)."""
import numpy as np
import pytest

from helpers import to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu

V, D = 128256, 4096


@pytest.fixture(scope="module")
def env():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda:0")
    bf = torch.bfloat16
    W = synth.device_normal_bf16_(torch.empty((V, D), dtype=bf, device=dev), 71, std=0.02)
    # the SM holder: 8 layers x 32 kv heads x 128 at L = 8192, a 64-node tree
    nl, H, d, L = 8, 32, 128, 8192
    parent = synth.bank_trees()[-1]
    N = len(parent)
    bank = tv.Bank(4, 0)
    bid, _ = bank.add(parent)
    k = synth.device_normal_bf16_(torch.empty((nl, H, L + N, d), dtype=bf, device=dev), 72)
    v = synth.device_normal_bf16_(torch.empty((nl, H, L + N, d), dtype=bf, device=dev), 73)
    q = synth.device_normal_bf16_(torch.empty((nl, N, H, d), dtype=bf, device=dev), 74)
    out = torch.empty((nl, N, H, d), dtype=bf, device=dev)
    ws_a = tv.make_workspace(tv.tb_workspace_size(N, nl, H, H, d, 1000, 0), dev)
    side = torch.cuda.Stream()
    kv = tv.KvCache(k, v, L)

    def hold_sms():
        side.wait_stream(torch.cuda.current_stream())
        tv.tree_attention(bank, bid, kv, q, out, ws_a, 0, nl, stream=side)

    yield dev, W, hold_sms, side, bank, bid, parent
    torch.cuda.synchronize()
    bank.close()


def _u32(t):
    return t.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("R", [26, 232])
def test_greedy_stats_independent_of_placement(env, R):
    dev, W, hold_sms, side, _, _, _ = env
    h = synth.device_normal_bf16_(torch.empty((R, D), dtype=torch.bfloat16, device=dev), 80 + R)
    ws = tv.make_workspace(tv.tb_workspace_size(R, 1, 1, 1, 128, V, 0), dev)

    def run(concurrent):
        am = torch.empty(R, dtype=torch.int32, device=dev)
        t1, en = (torch.empty(R, dtype=torch.float32, device=dev) for _ in range(2))
        if concurrent:
            hold_sms()
        tv.lm_head_stats(h, W, am, t1, en, ws)
        torch.cuda.synchronize()
        return _u32(am), _u32(t1), _u32(en)

    ref = run(False)
    for i in range(4):
        got = run(i % 2 == 0)
        for a, b, name in zip(got, ref, ("argmax", "top1", "entropy")):
            assert np.array_equal(a, b), f"R={R} run {i}: {name} differs"


def test_typical_stats_independent_of_placement(env):
    dev, W, hold_sms, side, bank, bid, parent = env
    N = len(parent)
    h = synth.device_normal_bf16_(torch.empty((N, D), dtype=torch.bfloat16, device=dev), 90)
    g = synth.rng(91)
    drafts = to_dev(g.integers(0, V, N).astype(np.int32), dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, 1, 1, 1, 128, V, 0), dev)

    def run(concurrent):
        am = torch.empty(N, dtype=torch.int32, device=dev)
        outs = [torch.empty(N, dtype=torch.float32, device=dev) for _ in range(5)]
        if concurrent:
            hold_sms()
        tv.lm_head_stats_typical(bank, bid, h, W, 0.7, drafts, am, *outs, ws)
        torch.cuda.synchronize()
        # draft_logit is written for non-root nodes only
        return [_u32(am)] + [_u32(o) for o in outs[:4]] + [_u32(outs[4])[1:]]

    ref = run(False)
    for i in range(4):
        got = run(i % 2 == 0)
        for j, (a, b) in enumerate(zip(got, ref)):
            assert np.array_equal(a, b), f"run {i}: output {j} differs"
