"""The bank-switching loop at the 7B single-layer shapes: the hysteretic step
ladder picks each step's tree from the 8-tree bank off a seeded AR(1) entropy
trace, L grows by accept_len, the KV cache is compacted every step; every
step is checked against the fp64 oracle (attention on sampled heads, LM-head
stats, acceptance, and the whole compacted cache)."""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, gap_filtered_hidden, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu


def test_bank_loop_7b_shapes():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    dev = torch.device("cuda:0")
    sh = synth.shape_c3()
    H, d, D, V = sh.n_q_heads, sh.head_dim, sh.d_model, sh.vocab
    steps = 10
    L = sh.L
    L_cap = L + steps * 6 + 64
    trees = synth.bank_trees()
    bank = tv.Bank(16, 0)
    ids = [bank.add(t)[0] for t in trees]
    k, v = synth.gen_kv(31, 1, H, L_cap, d, L_cap)
    kd, vd = to_dev(k, dev), to_dev(v, dev)
    W = synth.gen_lm_head(31, V, D)
    Wd = to_dev(W, dev)
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, H, H, d, V, 0), dev)
    # a trace that walks up the ladder and back: low entropy first, then high
    trace = np.concatenate([np.full(6, 1.0), np.full(4, 3.0)])
    kix = 0
    seen = []
    for step in range(steps):
        kix = tv.tb_schedule_hysteretic_ladder(kix, len(trees), float(trace[step]), 1.5, 2.5)
        seen.append(kix)
        parent = trees[kix]
        N = len(parent)
        q = synth.gen_q(200 + step, 1, N, H, d)
        hidden, am, t1, en = gap_filtered_hidden(200 + step, N, W)
        drafts = synth.gen_drafts(200 + step, parent, am, V, sh.p_match)
        out = torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev)
        g_am = torch.empty(N, dtype=torch.int32, device=dev)
        g_t1 = torch.empty(N, dtype=torch.float32, device=dev)
        g_en = torch.empty(N, dtype=torch.float32, device=dev)
        res = tv.make_result(dev)
        tv.verify_step(bank, ids[kix], tv.KvCache(kd, vd, L), to_dev(q, dev), to_dev(hidden, dev), Wd,
                       to_dev(drafts, dev), out, g_am, g_t1, g_en, res, ws)
        torch.cuda.synchronize()
        r = tv.parse_result(res)
        got = out.float().cpu().numpy()
        for head in (0, 17, H - 1):
            ref = oracle.tree_attention(q[0][:, head:head + 1], k[0][head:head + 1], v[0][head:head + 1], L, parent)
            check_attention(got[0][:, head:head + 1], ref, f"step {step} head {head}")
        assert np.array_equal(g_am.cpu().numpy(), am)
        assert np.abs(g_t1.cpu().numpy() - t1).max() <= STAT_TOL
        assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
        ka, path, bonus = oracle.accept(parent, drafts, am)
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        k, v = oracle.kv_compact(k, L, path), oracle.kv_compact(v, L, path)
        assert np.array_equal(bits(kd), k) and np.array_equal(bits(vd), v)
        L = r["new_L"]
    assert seen == [1, 2, 3, 4, 5, 6, 5, 4, 3, 2]
    bank.close()
