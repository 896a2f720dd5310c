"""Several host threads sharing one TopologyBank, each with its own stream,
cache, workspace and result block, calling verify_step concurrently.

Two step structures: a short attention that fits beside the LM head runs as
one chain on the caller's stream (each new thread's first call then encodes
its tensor maps before any other CUDA call of that thread); a longer one
forks the LM head onto the bank's helper stream, whose fork / join events are
shared and held under the bank's mutex, so the steps of different threads
never interleave their fork / join sequences.  Every step of every thread
must still match the fp64 oracle exactly (argmax, acceptance, path, bonus)
and within the attention tolerance, and the compacted caches must equal the
oracle's.
"""
import threading

import numpy as np
import pytest

import oracle
from helpers import STAT_TOL, bits, check_attention, make_case, to_dev
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


@pytest.mark.parametrize("d", [128, 64])
@pytest.mark.parametrize("structure,Hkv,L", [("chain", 2, 300), ("fork", 8, 3000)])
def test_threads_share_a_bank(dev, d, structure, Hkv, L):
    trees = [synth.full_tree((2, 2)), synth.bank_trees()[5], synth.bank_trees()[-1]]
    bank = tv.Bank(8, 0)
    ids = [bank.add(t)[0] for t in trees]
    n_threads, steps = 4, 12
    H, D, V = 8, 256, 1000
    workers = []
    for w in range(n_threads):
        j = w % len(trees)
        case = make_case(500 + 10 * w + d, trees[j], L, 1, H, Hkv, d, D, V, 0.7)
        N = case.N
        workers.append({
            "case": case, "id": ids[j], "N": N,
            "stream": torch.cuda.Stream(),
            "k": to_dev(case.k, dev), "v": to_dev(case.v, dev), "q": to_dev(case.q, dev),
            "h": to_dev(case.hidden, dev), "W": to_dev(case.W, dev),
            "drafts": to_dev(case.drafts.astype(np.int32), dev),
            "out": torch.empty((1, N, H, d), dtype=torch.bfloat16, device=dev),
            "am": torch.empty(N, dtype=torch.int32, device=dev),
            "t1": torch.empty(N, dtype=torch.float32, device=dev),
            "en": torch.empty(N, dtype=torch.float32, device=dev),
            "res": tv.make_result(dev),
            "ws": tv.make_workspace(tv.tb_workspace_size(N, 1, Hkv, H, d, V, 0), dev),
            "got": [], "error": None,
        })
    torch.cuda.synchronize()
    start = threading.Barrier(n_threads)

    def run(wk):
        try:
            s = wk["stream"]
            kv = tv.KvCache(wk["k"], wk["v"], L)
            start.wait()
            for t in range(steps):
                # the last step compacts the cache; the others leave it as it is
                flags = 0 if t == steps - 1 else tv.TB_NO_COMPACT
                tv.verify_step(bank, wk["id"], kv, wk["q"], wk["h"], wk["W"], wk["drafts"], wk["out"], wk["am"],
                               wk["t1"], wk["en"], wk["res"], wk["ws"], flags, s)
                s.synchronize()
                wk["got"].append((wk["out"].float().cpu().numpy(), wk["am"].cpu().numpy(),
                                  wk["en"].cpu().numpy(), tv.parse_result(wk["res"])))
        except Exception as e:  # reported by the main thread
            wk["error"] = e

    threads = [threading.Thread(target=run, args=(wk,)) for wk in workers]
    for th in threads:
        th.start()
    for th in threads:
        th.join(timeout=300)
    assert not any(th.is_alive() for th in threads), "a worker did not finish"
    for wk in workers:
        assert wk["error"] is None, wk["error"]
        c = wk["case"]
        ref_o = oracle.tree_attention(c.q[0], c.k[0], c.v[0], L, c.parent)
        ka, path, bonus = oracle.accept(c.parent, c.drafts, c.argmax)
        assert len(wk["got"]) == steps
        for t, (o, am, en, r) in enumerate(wk["got"]):
            check_attention(o[0], ref_o, f"step {t}")
            assert np.array_equal(am, c.argmax), f"step {t}"
            assert np.abs(en - c.entropy).max() <= STAT_TOL
            assert (r["accept_len"], r["path"], r["bonus_token"], r["new_L"], r["status"]) == \
                (ka, path, bonus, L + ka, 0), (t, r)
        assert np.array_equal(bits(wk["k"]), oracle.kv_compact(c.k, L, path))
        assert np.array_equal(bits(wk["v"]), oracle.kv_compact(c.v, L, path))
    bank.close()
