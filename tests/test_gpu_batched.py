"""GPU parity of verify_step_batched (ragged batches: one tree, prefix length
and KV cache per sequence) against the fp64 oracle, through the C ABI."""
import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, gap_filtered_hidden, to_dev
from paper_2606_27550_gb300 import synth

torch = pytest.importorskip("torch")
tv = pytest.importorskip("paper_2606_27550_gb300")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    from paper_2606_27550_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    return torch.device("cuda:0")


def _run_batch(dev, parents, Ls, ps, Hq, Hkv, d, D, V, seed, W=None, full_attention=True, n_layers=1,
               host_kv=True):
    bank = tv.Bank(32, 0)
    B = len(parents)
    Ns = [len(p) for p in parents]
    ids = [bank.add(p)[0] for p in parents]
    if W is None:
        W = synth.gen_lm_head(seed, V, D)
    hidden, am, t1, en = gap_filtered_hidden(seed + 1, sum(Ns), W)
    seqs, host = [], []
    r0 = 0
    for b in range(B):
        L, N = Ls[b], Ns[b]
        L_cap = L + N + 7
        if host_kv:
            k, v = synth.gen_kv(seed + 10 * b, n_layers, Hkv, L_cap, d, L + N)
            kd, vd = to_dev(k, dev), to_dev(v, dev)
        else:
            kd = synth.device_normal_bf16_(torch.empty((n_layers, Hkv, L_cap, d), dtype=torch.bfloat16, device=dev),
                                           seed + 10 * b)
            vd = synth.device_normal_bf16_(torch.empty_like(kd), seed + 10 * b + 1)
            k = v = None
        q = synth.gen_q(seed + 10 * b, n_layers, N, Hq, d)
        drafts = synth.gen_drafts(seed + b, parents[b], am[r0:r0 + N], V, ps[b])
        s = tv.Seq(ids[b], tv.KvCache(kd, vd, L), to_dev(q, dev), to_dev(drafts, dev),
                   torch.empty((n_layers, N, Hq, d), dtype=torch.bfloat16, device=dev), tv.make_result(dev))
        seqs.append(s)
        host.append(dict(k=k, v=v, q=q, drafts=drafts, tree_k=bits(kd[:, :, L:L + N]), tree_v=bits(vd[:, :, L:L + N]),
                         r0=r0))
        r0 += N
    R = sum(Ns)
    g_am = torch.full((R,), -1, dtype=torch.int32, device=dev)
    g_t1 = torch.empty(R, dtype=torch.float32, device=dev)
    g_en = torch.empty(R, dtype=torch.float32, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(R, n_layers, Hkv, Hq, d, V, 0), dev)
    tv.verify_step_batched(bank, seqs, to_dev(hidden, dev), to_dev(W, dev), g_am, g_t1, g_en, ws)
    torch.cuda.synchronize()
    assert tv.tb_workspace_status(ws) == 0
    assert np.array_equal(g_am.cpu().numpy(), am)
    assert np.abs(g_t1.cpu().numpy() - t1).max() <= STAT_TOL
    assert np.abs(g_en.cpu().numpy() - en).max() <= STAT_TOL
    for b, s in enumerate(seqs):
        h, L, N = host[b], Ls[b], Ns[b]
        r = tv.parse_result(s.result)
        ka, path, bonus = oracle.accept(parents[b], h["drafts"], am[h["r0"]:h["r0"] + N])
        assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == (ka, path, bonus, L + ka, 0)
        out = s.attn_out.float().cpu().numpy()
        if h["k"] is not None:
            for layer in range(n_layers):
                heads = range(Hkv) if full_attention else [0, Hkv - 1]
                grp = Hq // Hkv
                for g in heads:
                    ref = oracle.tree_attention(h["q"][layer][:, g * grp:(g + 1) * grp], h["k"][layer][g:g + 1],
                                                h["v"][layer][g:g + 1], L, parents[b])
                    check_attention(out[layer][:, g * grp:(g + 1) * grp], ref, f"seq {b} layer {layer} kv head {g}")
        # compaction of every layer / head, tree region only changes
        assert np.array_equal(bits(s.kv.k[:, :, L:L + N]), oracle.kv_compact(h["tree_k"], 0, path))
        assert np.array_equal(bits(s.kv.v[:, :, L:L + N]), oracle.kv_compact(h["tree_v"], 0, path))
    bank.close()
    return seqs


def test_batched_small_mixed(dev):
    trees = synth.bank_trees()
    parents = [trees[7], trees[0], trees[3], synth.chain(20), trees[5]]
    Ls = [300, 0, 129, 1000, 64]
    _run_batch(dev, parents, Ls, [0.7, 0.5, 0.9, 1.0, 0.3], Hq=8, Hkv=2, d=128, D=256, V=1000, seed=3)


def test_batched_two_layers_mha(dev):
    trees = synth.bank_trees()
    _run_batch(dev, [trees[6], trees[2], trees[7]], [77, 513, 5], [0.6, 0.6, 0.6], Hq=4, Hkv=4, d=128, D=128,
               V=777, seed=4, n_layers=2)


def test_batched_more_than_256_rows(dev):
    """384 LM-head rows: the LM head runs in chunks of 256 rows."""
    trees = synth.bank_trees()
    parents = [trees[7]] * 6
    _run_batch(dev, parents, [40, 90, 130, 10, 0, 260], [0.8] * 6, Hq=2, Hkv=1, d=128, D=128, V=515, seed=5,
               full_attention=False)


def test_batched_head_dim_64(dev):
    trees = synth.bank_trees()
    _run_batch(dev, [trees[4], trees[7]], [100, 33], [0.7, 0.7], Hq=4, Hkv=4, d=64, D=256, V=1000, seed=6)


def test_batched_max_batch(dev):
    trees = synth.bank_trees()
    g = synth.rng(8)
    parents = [trees[int(g.integers(1, 8))] for _ in range(tv.TB_MAX_BATCH)]
    Ls = [int(g.integers(0, 700)) for _ in range(tv.TB_MAX_BATCH)]
    _run_batch(dev, parents, Ls, [0.7] * tv.TB_MAX_BATCH, Hq=4, Hkv=2, d=128, D=128, V=600, seed=7,
               full_attention=False)


def test_batched_c5_full_size(dev):
    """The ragged batch at full size: batch 8, GQA 32/8 x 128, d_model 4096,
    V = 128256, L ~ U[512, 8192], trees of 4-64 nodes; LM-head stats of every
    row, acceptance and compaction exactly, attention on two kv heads per
    sequence."""
    sh = synth.batch_c5()
    Wd = synth.device_normal_bf16_(torch.empty((sh.vocab, sh.d_model), dtype=torch.bfloat16, device=dev), 55, 0.02)
    W = bits(Wd)
    del Wd
    _run_batch(dev, sh.parents, sh.Ls, sh.p_match, Hq=sh.n_q_heads, Hkv=sh.n_kv_heads, d=sh.head_dim,
               D=sh.d_model, V=sh.vocab, seed=9, W=W, full_attention=False)


def test_batched_argument_errors(dev):
    bank = tv.Bank(4, 0)
    bid, _ = bank.add(synth.full_tree((2, 2)))
    k = torch.zeros((1, 2, 40, 128), dtype=torch.bfloat16, device=dev)
    k2 = torch.zeros((1, 4, 40, 128), dtype=torch.bfloat16, device=dev)
    q = torch.zeros((1, 7, 4, 128), dtype=torch.bfloat16, device=dev)
    d = torch.zeros(7, dtype=torch.int32, device=dev)
    mk = lambda kk: tv.Seq(bid, tv.KvCache(kk, kk, 3), q, d, torch.empty_like(q), tv.make_result(dev))  # noqa: E731
    h = torch.zeros((14, 64), dtype=torch.bfloat16, device=dev)
    W = torch.zeros((100, 64), dtype=torch.bfloat16, device=dev)
    o = torch.empty(14, dtype=torch.int32, device=dev)
    f = torch.empty(14, dtype=torch.float32, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(14, 1, 2, 4, 128, 100, 0), dev)
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.verify_step_batched(bank, [mk(k), mk(k2)], h, W, o, f, f, ws)  # kv head counts differ
    assert e.value.status == tv.TB_EINVAL
    with pytest.raises(tv.TreeVerifyError) as e:
        tv.verify_step_batched(bank, [mk(k)] * (tv.TB_MAX_BATCH + 1), h, W, o, f, f, ws)
    assert e.value.status == tv.TB_EINVAL
    bank.close()
