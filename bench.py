"""Benchmark of the per-step tree-verification pass on GB300.

Default workload: the long-context full decode step of a 7B Llama-shaped
model, batch 1: 32 layers of tree attention at 32 heads x 128 over a bf16 KV
cache of L=16384 per layer, a 64-node depth-5 draft tree, then the 4096 x
32000 bf16 LM head with argmax / top-1 / entropy, greedy acceptance and the
KV-cache update.  One step = one verify_step call through the C ABI.

Prints one JSON line (rank 0).  Metric: verify-steps/s (with tree-tokens/s
and the fraction of the HBM roofline: KV + LM-head bytes over the measured
copy bandwidth).  Inputs are seeded synthetic tensors of the model's shapes,
resident in HBM and larger than L2 (8.9 GB touched per step), so no L2 flush
is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config c4|c2|c1] [--impl ours|reference]

--impl reference times the fp64 CPU oracle (the reference arm of this
build) on the host cores on a bounded sample of the same workload,
extrapolated to a full step.
Under torchrun each rank runs an independent replica on its own GPU (weak
scaling); the step time is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2606_27550_gb300 import synth  # noqa: E402

FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_BYTES = 129 << 20  # GB300 L2
# the bank loop's L2 policy: the cache is compacted in place every step, so it cannot rotate
C3_L2 = ("inputs larger than L2 every step: the LM head (262 MB) streams through L2 between one step's cache "
         "reads (34-130 MB as L grows) and the next's")
NOMINAL_HBM_GBS = 8000.0  # nominal HBM3e bandwidth, for context beside the measured copy peak


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def workload(cfg: str, layers: int | None = None):
    sh = synth.SHAPES[cfg]()
    if layers:
        sh.n_layers = layers
    N = sh.N
    kv_bytes = sh.n_layers * 2 * (sh.L + N) * sh.n_kv_heads * sh.head_dim * 2
    w_bytes = sh.vocab * sh.d_model * 2
    flops = 2 * N * sh.d_model * sh.vocab + 4 * N * (sh.L + N) * sh.head_dim * sh.n_q_heads * sh.n_layers
    return sh, kv_bytes, w_bytes, flops


from paper_2606_27550_gb300.replicas import dist_info, job_throughput, max_over_ranks  # noqa: E402


# ----------------------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 100 ms while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for ln in out.strip().splitlines():
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[4:8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, x in enumerate(r) if x.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------------------- GPU arm


def traffic_from_profiles(kernel: str, workload: str = ""):
    """Per-launch DRAM bytes of `kernel` on `workload` from the committed ncu
    summary, if its source hash still matches the current kernel source (else
    None).  A record without a workload column matches any workload."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    for ln in open(path):
        f = ln.split()
        if len(f) >= 4 and f[0] == kernel and not ln.startswith("#") and (len(f) < 5 or f[4] == workload):
            return float(f[3]) if kernel_source_hash(f[1]) == f[2] else None
    return None


def kernel_source_hash(files: str) -> str:
    """sha256[:16] over the comma-separated csrc files a kernel is built from."""
    import hashlib

    h = hashlib.sha256()
    for name in files.split(","):
        src = os.path.join(ROOT, "paper_2606_27550_gb300", "csrc", name)
        if not os.path.exists(src):
            return ""
        h.update(open(src, "rb").read())
    return h.hexdigest()[:16]


def acceptance_label(args) -> str:
    if getattr(args, "accept", "greedy") == "typical":
        return "typical (T=0.7, eps=0.09, alpha=0.3)"
    if getattr(args, "accept", "greedy") == "sampled":
        return "speculative sampling (T=0.7; drafts drawn from a synthetic head distribution)"
    return "greedy"


def l2_plan(sh, kv_bytes: int, w_bytes: int):
    """(copies, bytes of one copy, description) of the L2 policy of run_gpu: when a step's
    cache, queries and hidden rows (and the LM head, when it is small too) fit in L2, the
    timed steps rotate over enough copies of them that a step's data was last read more
    than twice the L2 size of traffic earlier."""
    cache = sh.n_layers * sh.n_kv_heads * sh.L_cap * sh.head_dim * 2 * 2
    qh = sh.n_layers * sh.N * sh.n_q_heads * sh.head_dim * 2 + sh.N * sh.d_model * 2
    small = cache + qh + (w_bytes if w_bytes < L2_BYTES else 0)
    if small >= 2 * L2_BYTES:
        return 1, small, f"inputs larger than L2 ({(kv_bytes + w_bytes) / 1e9:.2f} GB read per step)"
    n = min(512, -(-2 * L2_BYTES // small))
    if w_bytes >= L2_BYTES:
        return n, small, (f"the timed steps rotate over {n} copies of the cache, queries and hidden rows "
                          f"({small / 1e6:.1f} MB each); the LM head of {w_bytes / 1e6:.0f} MB streams through L2 "
                          f"every step")
    return n, small, f"the timed steps rotate over {n} copies of every input ({small / 1e6:.2f} MB each)"


def workload_config(args, sh, kv_bytes: int, w_bytes: int) -> dict:
    """The `config` of the JSON line (both arms)."""
    return {"workload": sh.name, "layers": sh.n_layers, "q_heads": sh.n_q_heads, "kv_heads": sh.n_kv_heads,
            "head_dim": sh.head_dim, "L": sh.L, "tree_nodes": sh.N, "tree_depth": int(synth.depth_of(sh.parent).max()),
            "d_model": sh.d_model, "vocab": sh.vocab, "batch": 1, "l2": l2_plan(sh, kv_bytes, w_bytes)[2],
            "acceptance": acceptance_label(args), "rope": "in-kernel, theta 10000" if args.rope else "none"}


def run_gpu(args):
    import torch
    import torch.distributed as dist

    import paper_2606_27550_gb300 as tv
    from paper_2606_27550_gb300 import build as tvbuild

    world, rank, local = dist_info()
    tvbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    sh, kv_bytes, w_bytes, flops = workload(args.config, args.layers)
    N, L, H, Hkv, d, D, V, nl = (sh.N, sh.L, sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model, sh.vocab,
                                 sh.n_layers)
    seed = 1234 + rank
    bf = torch.bfloat16
    k = synth.device_normal_bf16_(torch.empty((nl, Hkv, sh.L_cap, d), dtype=bf, device=dev), seed + 1)
    v = synth.device_normal_bf16_(torch.empty((nl, Hkv, sh.L_cap, d), dtype=bf, device=dev), seed + 2)
    q = synth.device_normal_bf16_(torch.empty((nl, N, H, d), dtype=bf, device=dev), seed + 3)
    W = synth.device_normal_bf16_(torch.empty((V, D), dtype=bf, device=dev), seed + 4, std=sh.w_std)
    hidden = synth.device_normal_bf16_(torch.empty((N, D), dtype=bf, device=dev), seed + 5)

    bank = tv.Bank(16, local)
    bid, order = bank.add(sh.parent)
    # --rope: the queries and tree keys are pre-rotary and every call applies the rotary
    # embedding at L + depth (the tree slots are rotated in place again each step: timing only)
    kv = tv.KvCache(k, v, L, rope_theta=10000.0 if args.rope else 0.0)
    # L2 policy: when a step's cache, queries and hidden rows (and the LM head, when it is
    # small too) fit in L2, the timed steps rotate over enough copies of them that a step's
    # data was last read more than twice the L2 size of traffic earlier
    n_copies, _, _ = l2_plan(sh, kv_bytes, w_bytes)
    rot = [(kv, q, hidden, W)]
    for c in range(1, n_copies):
        kc, vc = torch.empty_like(k).copy_(k), torch.empty_like(v).copy_(v)
        rot.append((tv.KvCache(kc, vc, L, rope_theta=kv.rope_theta), q.clone(), hidden.clone(),
                    W.clone() if W.numel() * 2 < L2_BYTES else W))
    out = torch.empty((nl, N, H, d), dtype=bf, device=dev)
    am = torch.empty(N, dtype=torch.int32, device=dev)
    t1 = torch.empty(N, dtype=torch.float32, device=dev)
    en = torch.empty(N, dtype=torch.float32, device=dev)
    res = tv.make_result(dev)
    ws = tv.make_workspace(tv.tb_workspace_size(N, nl, Hkv, H, d, V, local), dev)
    stream = torch.cuda.current_stream()

    # drafts: the greedy token of each node's parent with probability p, from an untimed LM-head pass
    tv.lm_head_stats(hidden, W, am, t1, en, ws)
    torch.cuda.synchronize()
    drafts = torch.from_numpy(synth.gen_drafts(seed, sh.parent, am.cpu().numpy(), V, sh.p_match)).to(dev)

    typical = args.accept == "typical"
    sampled = args.accept == "sampled"
    lz, et, dl = (torch.empty(N, dtype=torch.float32, device=dev) for _ in range(3))
    if sampled:
        # untimed: draft distributions = the target sharpened plus noise (a head that mostly
        # agrees with the model), drafts drawn from them, seeded uniforms
        g = torch.Generator(device=dev)
        g.manual_seed(seed + 9)
        zf = (hidden.float() @ W.float().t()) / 0.7
        qd = torch.softmax(zf * 1.3 + 0.5 * torch.randn(zf.shape, generator=g, device=dev), dim=1).contiguous()
        par = torch.from_numpy(np.asarray(sh.parent, np.int64)).to(dev)
        drafts = torch.zeros(N, dtype=torch.int32, device=dev)
        drafts[1:] = torch.multinomial(qd[par[1:]], 1, generator=g).squeeze(1).int()
        unif = torch.rand(2 * N, generator=g, device=dev)
        lgs = torch.empty((N + 1, V), dtype=torch.float32, device=dev)
        del zf

    def step(qq=q, hh=hidden, dd=drafts, st=None, outs=None, kvx=kv, Wx=W):
        st = stream if st is None else st
        oam, ot1, oen, ores = (am, t1, en, res) if outs is None else outs
        if sampled:
            tv.verify_step_sampled(bank, bid, kvx, qq, hh, Wx, dd, qd, unif, 0.7, out, oam, ot1, oen, lgs, ores, ws,
                                   0, st)
        elif typical:
            tv.verify_step_typical(bank, bid, kvx, qq, hh, Wx, dd, out, oam, ot1, oen, ores, ws, *tv.PAPER_TYPICAL,
                                   0, st)
        else:
            tv.verify_step(bank, bid, kvx, qq, hh, Wx, dd, out, oam, ot1, oen, ores, ws, 0, st)

    def rstep(i):
        kvx, qq, hh, Wx = rot[i % n_copies]
        step(qq, hh, kvx=kvx, Wx=Wx)

    visible = os.environ.get("CUDA_VISIBLE_DEVICES")
    sampler = ClockSampler(visible.split(",")[local] if visible else str(local))
    sampler.start()
    for i in range(args.warmup):
        rstep(i)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n0 = tv.tb_launch_count()
    e0.record(stream)
    for i in range(args.steps):
        rstep(args.warmup + i)
    e1.record(stream)
    n_launch = tv.tb_launch_count() - n0
    torch.cuda.synchronize()
    elapsed_ms = e0.elapsed_time(e1)
    if world > 1:
        dist.barrier()
    elapsed_ms = max_over_ranks(elapsed_ms, dev)
    r = tv.parse_result(res)

    # per-kernel durations: the same work through the stage entry points, events between stages
    n_k = max(3, min(args.steps, 50))
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_k)]
    # keep the GPU busy while the host enqueues, so that the events bracket
    # device time only (no host launch gaps between stages)
    torch.cuda._sleep(200_000_000)
    nvtx = torch.cuda.nvtx
    for i in range(n_k):
        kvx, qq, hh, Wx = rot[i % n_copies]
        ev[i][0].record(stream)
        nvtx.range_push("lm_head")
        if typical or sampled:
            tv.lm_head_stats_typical(bank, bid, hh, Wx, tv.PAPER_TYPICAL[0], drafts, am, t1, en, lz, et, dl, ws,
                                     stream)
        else:
            tv.lm_head_stats(hh, Wx, am, t1, en, ws, stream)
        nvtx.range_pop()
        ev[i][1].record(stream)
        nvtx.range_push("tree_attention")
        tv.tree_attention(bank, bid, kvx, qq, out, ws, 0, nl, stream)
        nvtx.range_pop()
        ev[i][2].record(stream)
        nvtx.range_push("acceptance+compaction")
        if sampled:
            tv.spec_sample_accept(bank, bid, drafts, lgs[:N], lz, qd, unif, L, 0.7, lgs[N], res, stream)
        elif typical:
            tv.typical_accept(bank, bid, drafts, am, lz, et, dl, V, L, res, *tv.PAPER_TYPICAL, stream=stream)
        else:
            tv.greedy_accept(bank, bid, drafts, am, V, L, res, stream)
        tv.kv_compact(kvx, res, stream)
        nvtx.range_pop()
        ev[i][3].record(stream)
    torch.cuda.synchronize()
    t_lm = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    t_at = statistics.mean(e[1].elapsed_time(e[2]) for e in ev)
    t_ac = statistics.mean(e[2].elapsed_time(e[3]) for e in ev)

    # end to end: every step copies its inputs from pinned host memory and reads its result
    # back with a host synchronisation.  Inputs are double-buffered: step i + 1's copy runs on
    # a copy stream while step i computes (events keep a buffer from being overwritten while
    # a step still reads it).  The step's outputs (result, argmax, top-1, entropy) sit in one
    # device block, read back by one copy; each buffer's verify_step call and that copy are
    # captured once into a CUDA graph, so the host enqueues one replay per step, before it
    # queues the next step's upload.
    q_h = torch.empty(q.shape, dtype=bf, pin_memory=True).copy_(q)
    h_h = torch.empty(hidden.shape, dtype=bf, pin_memory=True).copy_(hidden)
    d_h = torch.empty(drafts.shape, dtype=torch.int32, pin_memory=True).copy_(drafts)
    RI = tv.RESULT_INTS
    blk = torch.zeros(RI + 3 * N, dtype=torch.int32, device=dev)
    outs_e = (blk[RI:RI + N], blk[RI + N:RI + 2 * N].view(torch.float32), blk[RI + 2 * N:].view(torch.float32),
              blk[:RI])
    blk_h = [torch.empty(blk.shape, dtype=torch.int32, pin_memory=True) for _ in range(2)]
    h2d = q_h.numel() * 2 + h_h.numel() * 2 + d_h.numel() * 4
    d2h = blk.numel() * 4
    bufs = [(q, hidden, drafts), (torch.empty_like(q), torch.empty_like(hidden), torch.empty_like(drafts))]
    copy_stream = torch.cuda.Stream()
    ev_copied = [torch.cuda.Event(), torch.cuda.Event()]
    ev_used = [torch.cuda.Event(), torch.cuda.Event()]

    def upload(b):
        copy_stream.wait_event(ev_used[b])  # the step that last read these buffers is done
        with torch.cuda.stream(copy_stream):
            bufs[b][0].copy_(q_h, non_blocking=True)
            bufs[b][1].copy_(h_h, non_blocking=True)
            bufs[b][2].copy_(d_h, non_blocking=True)
            ev_copied[b].record(copy_stream)

    n_e2e = max(3, min(args.steps, 50))
    graphs = []
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    for b in range(2):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            step(*bufs[b], st=cap, outs=outs_e)
            blk_h[b].copy_(blk, non_blocking=True)
        graphs.append(g)
    torch.cuda.synchronize()
    for b in range(2):
        ev_used[b].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t0 = time.perf_counter()
    upload(0)
    for i in range(n_e2e):
        b = i % 2
        stream.wait_event(ev_copied[b])
        graphs[b].replay()
        ev_used[b].record(stream)
        if i + 1 < n_e2e:
            upload(1 - b)
        stream.synchronize()
        _ = int(blk_h[b][0])  # the per-step host read of the accepted length
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)
    clocks = sampler.stop()

    if world > 1:
        dist.destroy_process_group()
    bank.close()
    if rank != 0:
        return

    k1_name = "k1_tree_attention_tc"
    peaks, peak_src = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    ms = elapsed_ms / args.steps
    value = job_throughput(args.steps, elapsed_ms / 1e3, world)
    at_gbs = kv_bytes / (t_at * 1e-3) / 1e9
    # the roofline object names the stage that takes longer: the attention (K/V
    # bytes) or the LM head (W and hidden-row bytes; its time includes the merge
    # kernel k2_lm_merge that follows it)
    wl_name = workload_config(args, sh, kv_bytes, w_bytes)["workload"]
    if t_lm > t_at:
        lm_bytes = w_bytes + N * D * 2
        lm_gbs = lm_bytes / (t_lm * 1e-3) / 1e9
        roof = {"kernel": "k2_lm_head", "bound": "hbm", "achieved": round(lm_gbs, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(lm_gbs / hbm, 4), "traffic": traffic_from_profiles("k2_lm_head", wl_name),
                "note": "the LM head only streams W; the peak is a copy (read + write); the time includes the "
                        "row merge kernel k2_lm_merge",
                "algorithmic_bytes": lm_bytes, "avg_launch_ms": round(t_lm, 4)}
    else:
        roof = {"kernel": k1_name, "bound": "hbm", "achieved": round(at_gbs, 1), "peak": hbm,
                "unit": "GB/s", "frac": round(at_gbs / hbm, 4),
                # the committed capture is of the 32-layer long-context launch (scaled from 4 layers)
                "traffic": traffic_from_profiles(k1_name) if (args.config == "c4" and nl == 32) else None,
                "note": "the kernel only reads; the peak is a copy (read + write), so frac can exceed 1",
                "algorithmic_bytes": kv_bytes, "avg_launch_ms": round(t_at, 4)}
    line = {
        "metric": "verify-steps/s",
        "value": round(value, 3),
        "unit": "verify-steps/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded normal bf16 K/V, queries, hidden rows; LM head N(0, 0.02^2)); "
                "drafts = parent greedy token with p, else uniform",
        "config": workload_config(args, sh, kv_bytes, w_bytes),
        "tree_tokens_per_s": round(value * N, 1),
        "hbm_roofline": {"bytes_per_step": kv_bytes + w_bytes,
                         "frac": round((kv_bytes + w_bytes) / (ms * 1e-3) / 1e9 / hbm, 4),
                         "peak_gbs": hbm, "peak_src": peak_src,
                         "frac_nominal": round((kv_bytes + w_bytes) / (ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS, 4),
                         "nominal_gbs": NOMINAL_HBM_GBS},
        "compute_roofline": {"flops_per_step": flops,
                             "t_ms": round(flops / (float(peaks.get("bf16_tflops_sustained", 1713.0)) * 1e12) * 1e3, 4),
                             "frac": round(flops / (float(peaks.get("bf16_tflops_sustained", 1713.0)) * 1e12)
                                           / (ms * 1e-3), 4),
                             "peak_tflops": float(peaks.get("bf16_tflops_sustained", 1713.0))},
        "roofline": roof,
        "kernels_ms": {"k2_lm_head": round(t_lm, 4), k1_name: round(t_at, 4),
                       "k3_accept_compact": round(t_ac, 4)},
        "lm_head_gbs": round(w_bytes / (t_lm * 1e-3) / 1e9, 1),
        "accept_len_last": r["accept_len"],
        "e2e": {"value": round(job_throughput(n_e2e, e2e_s, world), 3), "unit": "verify-steps/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": n_launch,
        "clocks": clocks,
    }
    if args.layers:
        line["config"]["layers_override"] = args.layers
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.config, budget_s=args.cpu_budget)
    print(json.dumps(line), flush=True)


def run_gpu_batched(args):
    """The ragged batch (verify_step_batched): 8 sequences, GQA 32/8 x 128,
    L ~ U[512, 8192], trees of 4-64 nodes, one LM head of 4096 x 128256."""
    import torch
    import torch.distributed as dist

    import paper_2606_27550_gb300 as tv
    from paper_2606_27550_gb300 import build as tvbuild

    world, rank, local = dist_info()
    tvbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    sh = synth.batch_c5(seed=5)
    Hq, Hkv, d, D, V = sh.n_q_heads, sh.n_kv_heads, sh.head_dim, sh.d_model, sh.vocab
    bf = torch.bfloat16
    seed = 4321 + rank
    bank = tv.Bank(16, local)
    W = synth.device_normal_bf16_(torch.empty((V, D), dtype=bf, device=dev), seed, std=sh.w_std)
    R = sum(sh.Ns)
    hidden = synth.device_normal_bf16_(torch.empty((R, D), dtype=bf, device=dev), seed + 1)
    am = torch.empty(R, dtype=torch.int32, device=dev)
    t1 = torch.empty(R, dtype=torch.float32, device=dev)
    en = torch.empty(R, dtype=torch.float32, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(R, 1, Hkv, Hq, d, V, local), dev)
    # drafts from an untimed LM-head pass (rows in chunks of 256)
    for r0 in range(0, R, 256):
        r1 = min(R, r0 + 256)
        tv.lm_head_stats(hidden[r0:r1], W, am[r0:r1], t1[r0:r1], en[r0:r1], ws)
    torch.cuda.synchronize()
    am_h = am.cpu().numpy()
    seqs, kv_bytes, r0 = [], 0, 0
    for b, (parent, L, pm) in enumerate(zip(sh.parents, sh.Ls, sh.p_match)):
        N = len(parent)
        bid, _ = bank.add(parent)
        k = synth.device_normal_bf16_(torch.empty((1, Hkv, L + N, d), dtype=bf, device=dev), seed + 10 + 2 * b)
        v = synth.device_normal_bf16_(torch.empty((1, Hkv, L + N, d), dtype=bf, device=dev), seed + 11 + 2 * b)
        q = synth.device_normal_bf16_(torch.empty((1, N, Hq, d), dtype=bf, device=dev), seed + 100 + b)
        drafts = torch.from_numpy(synth.gen_drafts(seed + b, parent, am_h[r0:r0 + N], V, pm)).to(dev)
        seqs.append(tv.Seq(bid, tv.KvCache(k, v, L), q, drafts, torch.empty((1, N, Hq, d), dtype=bf, device=dev),
                           tv.make_result(dev)))
        kv_bytes += 2 * (L + N) * Hkv * d * 2
        r0 += N
    w_bytes = V * D * 2
    flops = 2 * R * D * V + sum(4 * len(p) * (L + len(p)) * d * Hq for p, L in zip(sh.parents, sh.Ls))
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # KV (~0.1 GB) fits in L2: flush between steps
    stream = torch.cuda.current_stream()

    def step():
        if args.accept == "typical":
            tv.verify_step_batched_typical(bank, seqs, hidden, W, am, t1, en, ws, *tv.PAPER_TYPICAL, 0, stream)
        else:
            tv.verify_step_batched(bank, seqs, hidden, W, am, t1, en, ws, 0, stream)

    sampler = ClockSampler(os.environ.get("CUDA_VISIBLE_DEVICES", str(local)).split(",")[local]
                           if os.environ.get("CUDA_VISIBLE_DEVICES") else str(local))
    sampler.start()
    for _ in range(args.warmup):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    n_launch = 0
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        n0 = tv.tb_launch_count()
        step()
        n_launch += tv.tb_launch_count() - n0
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    elapsed_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in ev), dev)
    clocks = sampler.stop()
    if world > 1:
        dist.destroy_process_group()
    bank.close()
    if rank != 0:
        return
    peaks, peak_src = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    tflops = float(peaks.get("bf16_tflops_sustained", 1700.0))
    ms = elapsed_ms / args.steps
    value = job_throughput(args.steps, elapsed_ms / 1e3, world)
    t_mem = (kv_bytes + w_bytes) / (hbm * 1e9) * 1e3
    t_comp = flops / (tflops * 1e12) * 1e3
    line = {
        "metric": "verify-steps/s", "value": round(value, 3), "unit": "verify-steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded)",
        "config": {"workload": sh.name, "batch": len(sh.parents), "tree_nodes": sh.Ns, "L": sh.Ls, "q_heads": Hq,
                   "kv_heads": Hkv, "head_dim": d, "d_model": D, "vocab": V,
                   "l2": "256 MB flush before every step, outside the timed interval (the batch's KV fits in L2)",
                   "compaction": "included (every step)", "acceptance": acceptance_label(args)},
        "tree_tokens_per_s": round(value * R, 1),
        "roofline": {"bound": "max(hbm, tensor)", "t_mem_ms": round(t_mem, 4), "t_compute_ms": round(t_comp, 4),
                     "frac": round(max(t_mem, t_comp) / ms, 4), "bytes_per_step": kv_bytes + w_bytes,
                     "flops_per_step": flops, "peak_gbs": hbm, "peak_tflops_sustained": tflops, "peak_src": peak_src},
        "gpu_launches": n_launch,
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)


def run_gpu_bank_loop(args):
    """The bank-switching loop: 7B single-layer shapes, the 8-tree bank, L from
    2048 growing by accept_len, 1000 steps; each step's tree comes from the
    hysteretic step ladder (up below 1.5 nats, down above 2.5 nats) over a
    seeded AR(1) entropy trace; KV compaction every step; the host reads the
    step's result (new prefix length) once per step."""
    import torch

    import paper_2606_27550_gb300 as tv
    from paper_2606_27550_gb300 import build as tvbuild

    world, rank, local = dist_info()
    tvbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    sh = synth.shape_c3()
    steps = sh.extra["steps"] if args.steps == 200 else args.steps
    H, d, D, V, L0 = sh.n_q_heads, sh.head_dim, sh.d_model, sh.vocab, sh.L
    bf = torch.bfloat16
    seed = 777 + rank
    trees = synth.bank_trees()
    bank = tv.Bank(16, local)
    ids = [bank.add(t)[0] for t in trees]
    k = synth.device_normal_bf16_(torch.empty((1, H, sh.L_cap, d), dtype=bf, device=dev), seed)
    v = synth.device_normal_bf16_(torch.empty((1, H, sh.L_cap, d), dtype=bf, device=dev), seed + 1)
    W = synth.device_normal_bf16_(torch.empty((V, D), dtype=bf, device=dev), seed + 2, std=sh.w_std)
    pool = 16
    qs = synth.device_normal_bf16_(torch.empty((pool, 1, 64, H, d), dtype=bf, device=dev), seed + 3)
    hs = synth.device_normal_bf16_(torch.empty((pool, 64, D), dtype=bf, device=dev), seed + 4)
    am = torch.empty(64, dtype=torch.int32, device=dev)
    t1 = torch.empty(64, dtype=torch.float32, device=dev)
    en = torch.empty(64, dtype=torch.float32, device=dev)
    ws = tv.make_workspace(tv.tb_workspace_size(64, 1, H, H, d, V, local), dev)
    drafts = {}
    for i in range(pool):  # untimed: each pool entry's greedy tokens -> drafts for every bank tree
        tv.lm_head_stats(hs[i], W, am, t1, en, ws)
        a = am.cpu().numpy()
        for j, t in enumerate(trees):
            drafts[(i, j)] = torch.from_numpy(synth.gen_drafts(seed + 100 * i + j, t, a[:len(t)], V, sh.p_match)).to(dev)
    outs = [torch.empty((1, len(t), H, d), dtype=bf, device=dev) for t in trees]
    res = tv.make_result(dev)
    res_h = torch.empty(tv.RESULT_INTS, dtype=torch.int32, pin_memory=True)
    trace = synth.ar1_entropy_trace(0, steps + args.warmup, hmax=float(np.log(V)))
    stream = torch.cuda.current_stream()

    def loop(t_from, t_to, L, kix):
        toks = kv_b = 0
        accepted = []
        hist = [0] * len(trees)
        for t in range(t_from, t_to):
            kix = tv.tb_schedule_hysteretic_ladder(kix, len(trees), float(trace[t]), 1.5, 2.5)
            n = len(trees[kix])
            i = t % pool
            kv = tv.KvCache(k, v, L)
            tv.verify_step(bank, ids[kix], kv, qs[i][:, :n], hs[i][:n], W, drafts[(i, kix)], outs[kix], am[:n],
                           t1[:n], en[:n], res, ws, 0, stream)
            res_h.copy_(res, non_blocking=True)
            stream.synchronize()
            kv_b += 2 * (L + n) * H * d * 2
            toks += n
            hist[kix] += 1
            accepted.append(int(res_h[0]))
            L = int(res_h[2])
        return L, kix, toks, kv_b, accepted, hist

    if args.scheduled:
        return bank_loop_scheduled(args, tv, torch, dev, bank, ids, trees, k, v, W, qs, hs, drafts, am, t1, en, res,
                                   ws, trace, steps, L0, sh, rank, world)
    L, kix, *_ = loop(0, args.warmup, L0, 0)
    sampler = ClockSampler(os.environ.get("CUDA_VISIBLE_DEVICES", str(local)).split(",")[local]
                           if os.environ.get("CUDA_VISIBLE_DEVICES") else str(local))
    sampler.start()
    torch.cuda.synchronize()
    n0 = tv.tb_launch_count()
    t0 = time.perf_counter()
    L_end, _, toks, kv_b, accepted, hist = loop(args.warmup, args.warmup + steps, L, kix)
    el = time.perf_counter() - t0
    n_launch = tv.tb_launch_count() - n0
    clocks = sampler.stop()
    bank.close()
    if rank != 0:
        return
    peaks, peak_src = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    w_b = V * D * 2 * steps
    line = {
        "metric": "verify-steps/s", "value": round(steps / el, 3), "unit": "verify-steps/s", "n_gpus": world,
        "steps": steps, "warmup": args.warmup, "ms_per_step": round(el / steps * 1e3, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded), AR(1) entropy trace",
        "config": {"workload": sh.name, "bank_sizes": [len(t) for t in trees], "L_start": L, "L_end": L_end,
                   "policy": "hysteretic step ladder: up below 1.5 nats, down above 2.5 nats",
                   "host_read_per_step": True, "l2": C3_L2},
        "tree_tokens_per_s": round(toks / el, 1),
        "tau_mean_accept_len": round(float(np.mean(accepted)), 4),
        "tree_histogram": hist,
        "hbm_roofline": {"bytes": kv_b + w_b, "frac": round((kv_b + w_b) / el / 1e9 / hbm, 4), "peak_gbs": hbm,
                         "peak_src": peak_src},
        "gpu_launches": n_launch,
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)


def bank_loop_scheduled(args, tv, torch, dev, bank, ids, trees, k, v, W, qs, hs, drafts, am, t1, en, res, ws, trace,
                        steps, L0, sh, rank, world):
    """The bank-switching loop driven from the device (verify_step_scheduled):
    the tree and the prefix length of each step live in device memory and the
    acceptance kernel takes the ladder decision (trace feature, up below 1.5,
    down above 2.5), so G steps are captured into one CUDA graph and replayed
    with no host read between steps."""
    bf = torch.bfloat16
    H, d = sh.n_q_heads, sh.head_dim
    n_max = 64
    pool = qs.shape[0]
    G = 48  # steps per graph (a multiple of the input pool)
    tab = []
    for i in range(pool):
        t_ = torch.zeros((len(trees), n_max), dtype=torch.int32, device=dev)
        for j, t in enumerate(trees):
            t_[j, :len(t)] = drafts[(i, j)]
        tab.append(t_)
    trace_d = torch.from_numpy(np.asarray(trace, dtype=np.float32)).to(dev)
    pol = tv.make_policy(tv.TB_POLICY_HYSTERETIC_LADDER, tv.TB_FEATURE_TRACE, ids, a=1.5, b=2.5, trace=trace_d,
                         node_stride=n_max)
    state = tv.make_state(0, L0, dev)
    out = torch.empty((1, n_max, H, d), dtype=bf, device=dev)
    kv = tv.KvCache(k, v, 0)

    def sstep(t, s):
        i = t % pool
        tv.verify_step_scheduled(bank, pol, state, kv, qs[i], hs[i], W, tab[i], out, am, t1, en, res, ws, 0, s)

    stream = torch.cuda.current_stream()
    for t in range(max(args.warmup, 3)):
        sstep(t, stream)
    torch.cuda.synchronize()
    cs = torch.cuda.Stream()
    cs.wait_stream(stream)
    g = torch.cuda.CUDAGraph()
    n0 = tv.tb_launch_count()
    with torch.cuda.graph(g, stream=cs):
        for t in range(G):
            sstep(t, cs)
    per_graph = tv.tb_launch_count() - n0  # kernels in the graph, launched again by every replay
    n_rep = (steps + G - 1) // G
    state.copy_(tv.make_state(0, L0, dev))
    torch.cuda.synchronize()
    sampler = ClockSampler(os.environ.get("CUDA_VISIBLE_DEVICES", str(dev.index)).split(",")[dev.index]
                           if os.environ.get("CUDA_VISIBLE_DEVICES") else str(dev.index))
    sampler.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(n_rep):
        g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    el = e0.elapsed_time(e1) / 1e3
    clocks = sampler.stop()
    st = tv.parse_state(state)
    bank.close()
    if rank != 0:
        return
    done = n_rep * G
    peaks, peak_src = load_peaks()
    line = {
        "metric": "verify-steps/s", "value": round(done / el, 3), "unit": "verify-steps/s", "n_gpus": world,
        "steps": done, "warmup": max(args.warmup, 3), "ms_per_step": round(el / done * 1e3, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded), AR(1) entropy trace",
        "config": {"workload": sh.name + "-device-driven", "l2": C3_L2, "bank_sizes": [len(t) for t in trees],
                   "L_start": L0,
                   "L_end": st["L"], "policy": "hysteretic step ladder on the device: up below 1.5, down above 2.5",
                   "host_read_per_step": False, "cuda_graph_steps": G},
        "tau_mean_accept_len": round((st["L"] - L0) / done, 4),
        "gpu_launches": per_graph * n_rep,
        "clocks": clocks,
        "hbm_roofline": {"peak_gbs": float(peaks["hbm_gbs"]), "peak_src": peak_src},
    }
    print(json.dumps(line), flush=True)


def expected_accept_len(parent, p_match: float) -> float:
    """E[accept_len] when every edge matches independently with probability
    p_match (the synthetic draft model: a node copies its parent's greedy token
    with probability p_match).  With f_u(k) = P(the deepest fully matched path
    below an accepted node u is >= k edges long), f_u(0) = 1 and
    f_u(k) = 1 - prod over children c of (1 - p f_c(k - 1)); then
    E[accept_len] = 1 + sum_{k >= 1} f_root(k)."""
    parent = list(parent)
    n = len(parent)
    kids = [[] for _ in range(n)]
    for i in range(1, n):
        kids[parent[i]].append(i)
    depth_max = int(synth.depth_of(parent).max())
    f = [[1.0] + [0.0] * depth_max for _ in range(n)]
    for u in range(n - 1, -1, -1):  # parent[i] < i: children before parents
        for k in range(1, depth_max + 1):
            miss = 1.0
            for c in kids[u]:
                miss *= 1.0 - p_match * f[c][k - 1]
            f[u][k] = 1.0 - miss
    return 1.0 + sum(f[0][1:])


def run_gpu_sweep(args):
    """Verify cost against tree size over the 8-tree bank (the kernel-side
    counterpart of the paper's throughput frontier, Sec. 3.2): for each tree,
    the device time of one verify_step at the 7B single-layer shape (L=2048)
    and at the long-context shape (32 layers, L=16384), with the expected
    accept length of the synthetic draft model at several match rates and the
    resulting accepted tokens per second."""
    import torch

    import paper_2606_27550_gb300 as tv
    from paper_2606_27550_gb300 import build as tvbuild

    world, rank, local = dist_info()
    tvbuild.build()
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    bf = torch.bfloat16
    trees = synth.bank_trees()
    bank = tv.Bank(16, local)
    ids = [bank.add(t)[0] for t in trees]
    ps = (0.5, 0.6, 0.7, 0.8, 0.9)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    rows = []
    n_launch = 0
    shapes = {"7b-1layer-L2048": (1, 2048), "7b-32layer-L16384": (32, 16384)}
    visible = os.environ.get("CUDA_VISIBLE_DEVICES")
    sampler = ClockSampler(visible.split(",")[local] if visible else str(local))
    sampler.start()
    for sname, (nl, L) in shapes.items():
        H, d, D, V = 32, 128, 4096, 32000
        seed = 99 + nl
        k = synth.device_normal_bf16_(torch.empty((nl, H, L + 64, d), dtype=bf, device=dev), seed)
        v = synth.device_normal_bf16_(torch.empty((nl, H, L + 64, d), dtype=bf, device=dev), seed + 1)
        W = synth.device_normal_bf16_(torch.empty((V, D), dtype=bf, device=dev), seed + 2, std=0.02)
        q = synth.device_normal_bf16_(torch.empty((nl, 64, H, d), dtype=bf, device=dev), seed + 3)
        hid = synth.device_normal_bf16_(torch.empty((64, D), dtype=bf, device=dev), seed + 4)
        am = torch.empty(64, dtype=torch.int32, device=dev)
        t1 = torch.empty(64, dtype=torch.float32, device=dev)
        en = torch.empty(64, dtype=torch.float32, device=dev)
        ws = tv.make_workspace(tv.tb_workspace_size(64, nl, H, H, d, V, local), dev)
        res = tv.make_result(dev)
        drafts = torch.zeros(64, dtype=torch.int32, device=dev)
        for j, t in enumerate(trees):
            n = len(t)
            qn = q[:, :n].contiguous()
            out = torch.empty((nl, n, H, d), dtype=bf, device=dev)
            kv = tv.KvCache(k, v, L)
            n_steps = max(10, min(args.steps, 100))
            for _ in range(args.warmup):
                tv.verify_step(bank, ids[j], kv, qn, hid[:n], W, drafts[:n], out, am[:n], t1[:n], en[:n], res, ws,
                               0, stream)
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                  for _ in range(n_steps)]
            for i in range(n_steps):
                flush.zero_()
                ev[i][0].record(stream)
                n0 = tv.tb_launch_count()
                tv.verify_step(bank, ids[j], kv, qn, hid[:n], W, drafts[:n], out, am[:n], t1[:n], en[:n], res, ws,
                               0, stream)
                n_launch += tv.tb_launch_count() - n0
                ev[i][1].record(stream)
            torch.cuda.synchronize()
            ms = statistics.median(a.elapsed_time(b) for a, b in ev)
            taus = {str(pm): round(expected_accept_len(t, pm), 4) for pm in ps}
            rows.append({"shape": sname, "tree_nodes": n, "tree_depth": int(synth.depth_of(t).max()),
                         "ms_per_step": round(ms, 4),
                         "accepted_tokens_per_s": {pm: round(tau / (ms * 1e-3), 1) for pm, tau in taus.items()},
                         "expected_accept_len": taus})
        del k, v, W, q, hid, ws
        torch.cuda.empty_cache()
    clocks = sampler.stop()
    bank.close()
    if rank != 0:
        return
    best = {}
    for sname in shapes:
        for pm in ps:
            cand = [r for r in rows if r["shape"] == sname]
            top = max(cand, key=lambda r: r["accepted_tokens_per_s"][str(pm)])
            best[f"{sname} p={pm}"] = top["tree_nodes"]
    c4_64 = [r for r in rows if r["shape"] == "7b-32layer-L16384" and r["tree_nodes"] == 64][0]
    line = {
        "metric": "verify-steps/s", "value": round(1e3 / c4_64["ms_per_step"], 3), "unit": "verify-steps/s",
        "n_gpus": 1, "steps": max(10, min(args.steps, 100)), "warmup": args.warmup,
        "ms_per_step": c4_64["ms_per_step"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded); accept lengths from the independent-match draft model",
        "config": {"workload": "bank sweep: 8 trees x {7B 1 layer L=2048, 7B 32 layers L=16384}",
                   "l2": "256 MB flush before every timed step, outside the timed interval",
                   "compaction": "included (every step)"},
        "sweep": rows,
        "throughput_optimal_tree": best,
        "gpu_launches": n_launch,
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- CPU oracle (reference arm)


def cpu_sample_step(cfg: str, attn_units: int, vocab_slices: int, seed: int = 0):
    """Runs the fp64 oracle on `attn_units` (layer, kv head) attention units and
    `vocab_slices` 1/32 vocab slices of the LM head plus acceptance; returns
    (extrapolated seconds of one full step, sample description)."""
    import oracle

    sh, _, _, _ = workload(cfg)
    N, L, d, D, V = sh.N, sh.L, sh.head_dim, sh.d_model, sh.vocab
    g = synth.rng(seed, 99)
    units_total = sh.n_layers * sh.n_kv_heads
    group = sh.n_q_heads // sh.n_kv_heads
    k = synth.normal_bf16(g, (1, L + N, d))
    v = synth.normal_bf16(g, (1, L + N, d))
    q = synth.normal_bf16(g, (N, group, d))
    slice_rows = (V + 31) // 32
    Wslice = synth.normal_bf16(g, (slice_rows, D), sh.w_std)
    hidden = synth.normal_bf16(g, (N, D))
    t0 = time.perf_counter()
    for _ in range(attn_units):
        oracle.tree_attention(q, k, v, L, sh.parent)
    t_attn = (time.perf_counter() - t0) / attn_units
    t0 = time.perf_counter()
    for _ in range(vocab_slices):
        am, _, _, _ = oracle.lm_head(hidden, Wslice)
    t_lm = (time.perf_counter() - t0) / vocab_slices
    t0 = time.perf_counter()
    drafts = synth.gen_drafts(seed, sh.parent, am, slice_rows, sh.p_match)
    oracle.accept(sh.parent, drafts, am)
    t_acc = time.perf_counter() - t0
    full = t_attn * units_total + t_lm * 32 + t_acc
    sample = (f"{attn_units} of {units_total} (layer, kv head) attention units ({N} nodes x {group} q heads x "
              f"{L + N} keys x d {d}) and {vocab_slices} of 32 vocab slices ({slice_rows} x {D}) of the LM head "
              f"for {N} rows, plus acceptance; time extrapolated to one full step")
    return full, sample, t_attn + t_lm, t_attn * attn_units + t_lm * vocab_slices + t_acc


def cpu_model() -> str:
    try:
        for ln in open("/proc/cpuinfo"):
            key = ln.split(":")[0].strip().lower()
            if key in ("model name", "cpu model", "hardware"):
                return ln.split(":", 1)[1].strip()
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    import platform

    return platform.processor() or platform.machine()


def sample_units(cfg: str, budget_s: float) -> int:
    """Attention units of a CPU sample that takes about budget_s (a probe times one unit
    and one vocab slice), at most the whole step."""
    _, _, probe, _ = cpu_sample_step(cfg, 1, 1)
    sh, _, _, _ = workload(cfg)
    return int(max(1, min(sh.n_layers * sh.n_kv_heads, budget_s / max(probe, 1e-6))))


def cpu_baseline(cfg: str, budget_s: float = 20.0):
    """The oracle timed on this host's cores on a bounded sample of the workload (all
    cores, and one thread on a smaller sample)."""
    import oracle

    oracle.build()
    n = sample_units(cfg, budget_s)
    full, sample, _, _ = cpu_sample_step(cfg, n, min(n, 32), seed=1)
    cores = oracle.num_threads()
    prev = oracle.set_num_threads(1)
    try:
        full1, sample1, _, _ = cpu_sample_step(cfg, 1, 1, seed=2)
    finally:
        oracle.set_num_threads(prev)
    return {"value": round(1.0 / full, 6), "unit": "verify-steps/s", "cores": cores, "kind": "oracle",
            "sample": sample, "s_per_full_step": round(full, 3),
            "single_thread": {"value": round(1.0 / full1, 7), "s_per_full_step": round(full1, 2), "sample": sample1},
            "nproc": os.cpu_count(), "cpu_model": cpu_model()}


def run_reference(args):
    import oracle

    world, rank, _ = dist_info()
    if rank != 0:
        return
    oracle.build()
    sh, _, _, _ = workload(args.config)
    # each step: a sample of as many attention units as the run's time budget allows
    # (args.cpu_budget x 6 seconds over warm-up and timed steps), extrapolated to a full step
    n = sample_units(args.config, args.cpu_budget * 6.0 / (args.warmup + args.steps))
    for i in range(args.warmup):
        cpu_sample_step(args.config, n, min(n, 32), seed=i)
    times, measured = [], []
    sample = ""
    for i in range(args.steps):
        full, sample, _, took = cpu_sample_step(args.config, n, min(n, 32), seed=100 + i)
        times.append(full)
        measured.append(took)
    mean = statistics.mean(times)
    value = 1.0 / mean
    line = {
        "impl": "reference",
        "metric": "verify-steps/s",
        "value": round(value, 6),
        "unit": "verify-steps/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(mean * 1e3, 3),
        "ms_per_step_kind": "extrapolated: each step times a sample of the workload and scales it to one full step",
        "measured_s_per_step": round(statistics.mean(measured), 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic (seeded)",
        "config": workload_config(args, sh, *workload(args.config)[1:3]),
        "cpu_baseline": {"value": round(value, 6), "unit": "verify-steps/s", "cores": oracle.num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 6), "unit": "verify-steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", default="c4", choices=["c1", "c2", "c3", "c4", "c5", "sweep"])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=None, help="override the layer count (smaller profiling cases)")
    ap.add_argument("--cpu-budget", type=float, default=20.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--rope", action="store_true",
                    help="c1/c2/c4: pre-rotary inputs, rotary embedding applied by the library")
    ap.add_argument("--scheduled", action="store_true",
                    help="c3 only: the device-driven loop (tree and L on the device, CUDA-graph replay)")
    ap.add_argument("--accept", default="greedy", choices=["greedy", "typical", "sampled"],
                    help="verification rule: greedy (default), typical acceptance at T=0.7, eps=0.09, alpha=0.3, "
                         "or speculative sampling at T=0.7")
    args = ap.parse_args(argv)
    if args.accept != "greedy" and (args.impl == "reference" or args.config in ("c3", "sweep")):
        ap.error("--accept typical / sampled apply to the GPU arm of c1, c2, c4 and c5")
    if args.accept == "sampled" and args.config == "c5":
        ap.error("--accept sampled runs one sequence per step (c1, c2, c4)")
    if args.scheduled and (args.config != "c3" or args.impl == "reference"):
        ap.error("--scheduled applies to the GPU arm of c3")
    if args.impl == "reference" and args.config == "sweep":
        ap.error("the sweep has no reference arm")
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    elif args.config == "c5":
        run_gpu_batched(args)
    elif args.config == "c3":
        run_gpu_bank_loop(args)
    elif args.config == "sweep":
        run_gpu_sweep(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
