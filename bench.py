#!/usr/bin/env python3
"""Draft+verify decoding step of tri-mode decoding on one GB300, at the 8B shape.

One step = the whole path on one batch of synthetic input:
  diffusion-draft block attention (bidirectional in-block) over the paged KV
  cache, top-k unmasking of the draft confidences, AR-verify block attention
  (causal in-block), and longest-prefix acceptance. Each block-attention pass
  is the attention kernel plus, when the KV range is split, the combine.

Workload: batch 1, 32 query / 8 KV heads, head_dim 128, 4096-token prefix in
16-token pages under a random page permutation, block of 16 (the 8B decoder
shape). Every pass reads its own KV pool from a rotation of pools larger than
three times L2, so each pass streams its KV from HBM as it would with the other
layers of a model running between two passes of the same layer.

Output: one JSON line (rank 0). value = KV GB/s over the whole step
(algorithmic KV bytes of both passes / step time); steps_per_s alongside.

--impl reference times the fp64 CPU oracle on the host cores instead (the
slow reference program this path is checked against), on a bounded sample of
the same workload per step.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import platform
import os
import re
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_05722_gb300 import workloads as W  # noqa: E402

METRIC = "block-attn KV GB/s (% of GB300 HBM peak); draft+verify steps/sec at 8B shape"
WORKLOAD = W.HEADLINE
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
TRAFFIC_NOTE = os.path.join(ROOT, "profiles", "block_attn_8b_b1_L4096_bl16.md")
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2607_05722_gb300", "csrc", f)
                  for f in ("block_attn_tc.cuh", "nld_internal.cuh", "nld_api.cu")]


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30000)
    ap.add_argument("--warmup", type=int, default=300)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--pools", type=int, default=32, help="rotating KV pools (cold-L2 rotation)")
    ap.add_argument("--splits", type=int, default=0, help="KV splits (0 = automatic)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--headline-only", action="store_true", help="skip the other named workloads")
    ap.add_argument("--only-workload", default=None,
                    help="time only this named workload (device-drawn inputs), e.g. for a profiler")
    ap.add_argument("--workload-batch", type=int, default=None, help="batch override for --only-workload")
    ap.add_argument("--split-sweep", action="store_true",
                    help="with --only-workload: also time a verify pass for explicit split counts 1..64")
    ap.add_argument("--only-section", default=None, choices=["decisions", "logits", "kv_commit", "quadss"],
                    help="time only this section of the report (e.g. for a profiler)")
    ap.add_argument("--no-prefix-ready", action="store_true",
                    help="do not let attention stream prefix KV before its dependency wait")
    ap.add_argument("--seed", type=int, default=0)
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def hbm_peak():
    try:
        with open(PEAKS_PATH) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash():
    h = hashlib.sha256()
    for p in KERNEL_SOURCES:
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic():
    """DRAM bytes per launch of the attention kernel from a committed ncu
    summary, when it was taken on the current kernel source; else None."""
    try:
        text = open(TRAFFIC_NOTE).read()
    except OSError:
        return None
    m_src = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]{16})", text)
    m_tr = re.search(r"dram_bytes_per_launch:\s*([0-9]+)", text)
    if not m_src or not m_tr or m_src.group(1) != kernel_source_hash():
        return None
    return int(m_tr.group(1))


# ---------------------------------------------------------------------------
# clock sampling during the timed region
# ---------------------------------------------------------------------------

CLOCK_FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    def __init__(self, device_index: int):
        self.proc = None
        self.path = None
        try:
            fd, self.path = tempfile.mkstemp(prefix="nld_clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={CLOCK_FIELDS}", "--format=csv,noheader,nounits", "-lms", "50",
                 "-i", str(device_index)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        """Median SM clock and throttle reasons of samples inside [t0, t1] (host
        time); falls back to all samples while the GPU was busy."""
        if self.path is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "note": "nvidia-smi unavailable"}
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts, float(parts[2]), float(parts[3]), parts[6:10]))
            except (ValueError, IndexError):
                continue
        os.unlink(self.path)
        inside = [r for r in rows if t0 - 0.05 <= r[0] <= t1 + 0.05]
        note = "samples inside the timed region"
        if not inside:
            inside = rows
            note = "timed region shorter than the sampling period: all samples of the run"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "note": "no samples"}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in inside for j, v in enumerate(r[3]) if v.lower() == "active"})
        return {"sm_mhz": float(np.median([r[1] for r in inside])), "sm_max_mhz": max(r[2] for r in inside),
                "reasons": reasons, "samples": len(inside), "note": note}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def run_only_workload(args, local):
    """Time one named workload's step (for profilers); prints one JSON line."""
    import torch

    from paper_2607_05722_gb300 import build as nld_build
    from paper_2607_05722_gb300 import nld

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    nld_build.build()
    nld.lib()
    peak, _ = hbm_peak()
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    stream = torch.cuda.Stream(device=dev)
    res = run_workloads(torch, nld, dev, stream, peak, l2, only=args.only_workload, batch=args.workload_batch,
                        sweep_splits=args.split_sweep)
    print(json.dumps({"workload": args.only_workload, "batch": args.workload_batch, **res[args.only_workload]}))


def run_only_section(args, local):
    """Time one auxiliary section of the report alone; prints one JSON line."""
    import torch

    from paper_2607_05722_gb300 import build as nld_build
    from paper_2607_05722_gb300 import nld

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    nld_build.build()
    nld.lib()
    peak, _ = hbm_peak()
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    stream = torch.cuda.Stream(device=dev)
    fn = {"decisions": lambda: run_decisions(torch, nld, dev, stream),
          "logits": lambda: run_logits(torch, nld, dev, stream, peak, l2),
          "kv_commit": lambda: run_kv_commit(torch, nld, dev, stream),
          "quadss": lambda: run_quadss(torch, nld, dev, stream, peak, l2)}[args.only_section]
    print(json.dumps({"section": args.only_section, **fn()}))


# ---------------------------------------------------------------------------
# multi-GPU host logic (weak scaling: one rank per GPU, each on its own
# sequences; the timing reduce is the only collective)
# ---------------------------------------------------------------------------

def rank_seed(base_seed: int, rank: int) -> int:
    """Seed of a rank's workload: every rank draws its own sequences."""
    return base_seed + rank


def max_over_ranks(value: float, world: int, device=None) -> float:
    """The job's time is its slowest rank's: the max over the ranks."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_kv_gbs(kv_bytes_per_pass: int, passes: int, world: int, ms_per_step: float) -> float:
    """Whole-job KV GB/s: every rank's passes over its own KV per step time."""
    return passes * kv_bytes_per_pass * world / (ms_per_step * 1e-3) / 1e9


def run_ours(args, world, rank, local):
    import torch
    import torch.distributed as dist

    from paper_2607_05722_gb300 import build as nld_build
    from paper_2607_05722_gb300 import nld

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    nld_build.build()
    nld.lib()

    wl = W.make_workload(WORKLOAD, seed=rank_seed(args.seed, rank))
    c = wl.attn
    kv = c.kv
    B, bl, Hq, Hkv, D = c.batch, c.block_len, c.num_q_heads, c.num_kv_heads, c.head_dim
    kv_bytes = c.kv_bytes_per_pass()
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    npool = pool_count(kv_bytes, l2, args.pools)

    def dev_bf16(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)

    k0, v0 = dev_bf16(kv.k_bits), dev_bf16(kv.v_bits)
    pools = [(k0, v0)] + [(k0.clone(), v0.clone()) for _ in range(npool - 1)]
    table = torch.from_numpy(kv.page_table).to(dev)
    prefix = torch.from_numpy(kv.prefix_lens).to(dev)
    q_d, q_v = dev_bf16(c.q_draft_bits), dev_bf16(c.q_verify_bits)
    # The page table, prefix lengths and prefix KV are not written by the
    # kernels of the step, so each attention pass may start streaming its
    # prefix before waiting on the previous kernel (NLD_ATTN_PREFIX_READY).
    params = nld.make_params(B, Hq, Hkv, D, c.page_size, kv.num_pages, kv.max_pages, args.splits, 0.0,
                             0 if args.no_prefix_ready else nld.NLD_ATTN_PREFIX_READY)
    splits = nld.nld_block_attn_num_splits(params, bl)
    ws = torch.zeros(max(nld.nld_block_attn_workspace_size(params, bl), 16), dtype=torch.uint8, device=dev)
    out_d = torch.empty((B, bl, Hq, D), dtype=torch.bfloat16, device=dev)
    out_v = torch.empty_like(out_d)
    lse_d = torch.empty((B, Hq, bl), dtype=torch.float32, device=dev)
    lse_v = torch.empty_like(lse_d)
    draft = torch.from_numpy(wl.draft_ids).to(dev)
    verify = torch.from_numpy(wl.verify_ids).to(dev)
    conf = torch.from_numpy(wl.conf[0]).to(dev)
    k_unmask = wl.unmask_k[0]
    acc = torch.empty((B,), dtype=torch.int32, device=dev)
    pos = torch.empty((B, k_unmask), dtype=torch.int32, device=dev)
    nsel = torch.empty((B,), dtype=torch.int32, device=dev)
    attn_kernels = nld.nld_block_attn_kernels(params, bl)  # 1: unsplit or cluster-merged; 2: + combine
    launches_per_step = 2 * attn_kernels + 2

    def step(i, kd=None, vd=None, kvv=None, vv=None):
        kd, vd = (kd, vd) if kd is not None else pools[(2 * i) % npool]
        kvv, vv = (kvv, vv) if kvv is not None else pools[(2 * i + 1) % npool]
        nld.nld_block_attn(params, q_d, kd, vd, table, prefix, bl, nld.NLD_MODE_DIFFUSION, out_d, lse_d, ws)
        nld.nld_unmask(conf, k_unmask, pos, nsel)
        nld.nld_block_attn(params, q_v, kvv, vv, table, prefix, bl, nld.NLD_MODE_VERIFY, out_v, lse_v, ws)
        nld.nld_accept(draft, verify, acc)

    # eager run once (also loads per-device state before capture)
    step(0)
    torch.cuda.synchronize()

    chunk = 256
    stream = torch.cuda.Stream(device=dev)

    def capture(nsteps, offset=0):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(g, stream=stream):
                for i in range(nsteps):
                    step(offset + i)
        return g

    g_main = capture(chunk)
    reps, rem = divmod(args.steps, chunk)
    g_rem = capture(rem, offset=reps * chunk) if rem else None
    wreps, wrem = divmod(max(args.warmup, 3), chunk)
    g_wrem = capture(wrem) if wrem else None
    torch.cuda.synchronize()

    sampler = ClockSampler(local) if rank == 0 else None
    time.sleep(0.3 if sampler else 0.0)
    # warm-up steps (untimed)
    with torch.cuda.stream(stream):
        for _ in range(wreps):
            g_main.replay()
        if g_wrem is not None:
            g_wrem.replay()
    torch.cuda.synchronize()

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_host0 = time.time()
    with torch.cuda.stream(stream):
        ev0.record(stream)
        for _ in range(reps):
            g_main.replay()
        if g_rem is not None:
            g_rem.replay()
        ev1.record(stream)
    torch.cuda.synchronize()
    t_host1 = time.time()
    if world > 1:
        dist.barrier()
    ms = max_over_ranks(ev0.elapsed_time(ev1), world, dev)
    clocks = None
    if sampler is not None:
        time.sleep(0.1)
        sampler.stop()
        clocks = sampler.summary(t_host0, t_host1)

    # ---- per-launch duration of the attention kernel (CUDA events on its stream) ----
    # (a) a CUDA graph of back-to-back attention launches, each on its own cold
    #     KV pool, alternating modes: events around the replays / launches;
    # (b) the same launches one by one, each bracketed by its own events.
    nker = 2 * npool
    views = nld.workspace_views(params, bl, ws)

    def attn_launch(j, strm=None):
        # the attention kernel alone: the whole call when it launches one
        # kernel, else the partials entry (the combine is timed apart)
        kp, vp = pools[j % npool]
        mode = nld.NLD_MODE_VERIFY if j % 2 else nld.NLD_MODE_DIFFUSION
        fn = nld.nld_block_attn if attn_kernels == 1 else nld.nld_block_attn_partials
        fn(params, q_v if j % 2 else q_d, kp, vp, table, prefix, bl, mode, out_v, lse_v, ws, stream=strm)

    g_attn = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        with torch.cuda.graph(g_attn, stream=stream):
            for j in range(nker):
                attn_launch(j)
    g_comb = None
    if views is not None and attn_kernels == 2:
        g_comb = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(g_comb, stream=stream):
                for j in range(nker):
                    nld.nld_split_kv_combine(views[0], views[1], out_v, lse_v)
    krep = 20
    with torch.cuda.stream(stream):
        g_attn.replay()
        torch.cuda.synchronize()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(krep):
            g_attn.replay()
        a1.record(stream)
        if g_comb is not None:
            c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            c0.record(stream)
            for _ in range(krep):
                g_comb.replay()
            c1.record(stream)
    torch.cuda.synchronize()
    attn_ms = a0.elapsed_time(a1) / (krep * nker)
    comb_ms = c0.elapsed_time(c1) / (krep * nker) if g_comb is not None else 0.0

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nker)]
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(60e6))  # queue the launches behind a busy GPU so no host gap enters a bracket
        for j in range(nker):
            evs[j][0].record(stream)
            attn_launch(j, stream)
            evs[j][1].record(stream)
    torch.cuda.synchronize()
    attn_iso_ms = float(np.mean([x.elapsed_time(y) for x, y in evs]))

    # ---- warm step: both passes of every step read one KV pool (16 MiB, so it
    #      stays in L2), as when the verify pass rereads the prefix the draft
    #      pass has just read; reported beside the cold step, not as the value ----
    warm_ms = time_graph(torch, stream, lambda i: step(0, k0, v0, k0, v0), 64, 10)

    # ---- end to end through the API with host buffers ----
    e2e_params = nld.make_params(B, Hq, Hkv, D, c.page_size, kv.num_pages, kv.max_pages, args.splits, 0.0, 0)
    e2e = run_e2e(args, torch, nld, dev, stream, wl, e2e_params, splits, kv_bytes, world)

    if world > 1:
        dist.barrier()
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    peak, peak_kind = hbm_peak()
    ms_step = ms / args.steps
    value = job_kv_gbs(kv_bytes, 2, world, ms_step)
    attn_gbs = kv_bytes / (attn_ms * 1e-3) / 1e9
    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": headline_config(wl, npool, l2, splits, attn_kernels, not args.no_prefix_ready),
        "steps_per_s": round(1e3 / ms_step, 1) * world,
        "pct_of_hbm_peak": round(100.0 * value / world / peak, 2),
        "clocks": clocks,
        "e2e": e2e,
        "warm_step": {"ms_per_step": round(warm_ms, 6), "kv_gbs": round(2 * kv_bytes / (warm_ms * 1e-3) / 1e9, 1),
                      "note": "both passes of every step read one KV pool (L2-resident): the verify pass "
                              "rereads the prefix the draft pass has just read; the value above is the cold step"},
        "gpu_launches": launches_per_step * args.steps,
        "roofline": {
            "kernel": "block_attn_tc_kernel (attention; split partials when the plan has several)",
            "bound": "hbm",
            "achieved": round(attn_gbs, 1),
            "peak": peak,
            "peak_kind": f"{peak_kind} hbm_gbs (burst copy)",
            "unit": "GB/s",
            "frac": round(attn_gbs / peak, 4),
            "traffic": recorded_traffic(),
            "algorithmic_bytes_per_launch": kv_bytes,
            "avg_launch_us": round(attn_ms * 1e3, 3),
            "timing": "CUDA graph of back-to-back launches on rotating cold KV pools; events around replays",
            "isolated_launch_us": round(attn_iso_ms * 1e3, 3),
            "combine_avg_launch_us": round(comb_ms * 1e3, 3),
        },
    }
    if not args.headline_only:
        line["workloads"] = run_workloads(torch, nld, dev, stream, peak, l2)
        line["decisions"] = run_decisions(torch, nld, dev, stream)
        line["logits_argmax"] = run_logits(torch, nld, dev, stream, peak, l2)
        line["kv_commit"] = run_kv_commit(torch, nld, dev, stream)
        line["quadss_pass"] = run_quadss(torch, nld, dev, stream, peak, l2)
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, budget_s=12.0)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_e2e(args, torch, nld, dev, stream, wl, params, splits, kv_bytes, world):
    """The same step through the API with every input copied in from pinned
    host memory and the results read back, inside the timed region. Inputs
    are double-buffered as a serving loop would: while step i computes on one
    device set, the copy stream brings step i+1's inputs into the other; the
    small inputs travel packed in one copy and the results in one read-back."""
    c = wl.attn
    kv = c.kv
    B, bl, Hq, D = c.batch, c.block_len, c.num_q_heads, c.head_dim
    kk = wl.unmask_k[0]

    def pinned(a):
        return torch.from_numpy(np.ascontiguousarray(a)).pin_memory()

    # host side: K and V pools, then the small inputs packed (16-byte aligned)
    small = [("q_d", c.q_draft_bits.view(np.int16)), ("q_v", c.q_verify_bits.view(np.int16)),
             ("table", kv.page_table), ("prefix", kv.prefix_lens), ("draft", wl.draft_ids),
             ("verify", wl.verify_ids), ("conf", wl.conf[0])]
    offs, off = {}, 0
    for name, a in small:
        offs[name] = (off, a)
        off += (a.nbytes + 15) // 16 * 16
    h_small = torch.zeros(off, dtype=torch.uint8).pin_memory()
    for name, (o, a) in offs.items():
        h_small[o:o + a.nbytes].copy_(torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1)))
    h_k, h_v = pinned(kv.k_bits.view(np.int16)), pinned(kv.v_bits.view(np.int16))
    out_bytes = 2 * B * bl * Hq * D * 2 + B * 4 + B * kk * 4

    def device_set():
        ds = {"k": torch.empty(h_k.shape, dtype=h_k.dtype, device=dev),
              "v": torch.empty(h_v.shape, dtype=h_v.dtype, device=dev),
              "small": torch.empty(off, dtype=torch.uint8, device=dev),
              "out": torch.empty(out_bytes, dtype=torch.uint8, device=dev)}
        for name, (o, a) in offs.items():
            dt = {np.dtype(np.int16): torch.int16, np.dtype(np.int32): torch.int32,
                  np.dtype(np.float32): torch.float32}[a.dtype]
            ds[name] = ds["small"][o:o + a.nbytes].view(dt).view(a.shape)
        o = 0
        for name, n, dt, shape in (("out_d", B * bl * Hq * D * 2, torch.bfloat16, (B, bl, Hq, D)),
                                   ("out_v", B * bl * Hq * D * 2, torch.bfloat16, (B, bl, Hq, D)),
                                   ("acc", B * 4, torch.int32, (B,)), ("pos", B * kk * 4, torch.int32, (B, kk))):
            ds[name] = ds["out"][o:o + n].view(dt).view(shape)
            o += n
        return ds

    sets = [device_set(), device_set()]
    h_out = torch.empty(out_bytes, dtype=torch.uint8).pin_memory()
    ws = torch.zeros(max(nld.nld_block_attn_workspace_size(params, bl), 16), dtype=torch.uint8, device=dev)
    nsel = torch.empty((B,), dtype=torch.int32, device=dev)
    copy_stream = torch.cuda.Stream(device=dev)

    def bf(t):
        return t.view(torch.bfloat16)

    def copy_into(ds):
        ds["k"].copy_(h_k, non_blocking=True)
        ds["v"].copy_(h_v, non_blocking=True)
        ds["small"].copy_(h_small, non_blocking=True)

    def compute(ds):
        nld.nld_block_attn(params, bf(ds["q_d"]), bf(ds["k"]), bf(ds["v"]), ds["table"], ds["prefix"], bl,
                           nld.NLD_MODE_DIFFUSION, ds["out_d"], None, ws)
        nld.nld_unmask(ds["conf"], kk, ds["pos"], nsel)
        nld.nld_block_attn(params, bf(ds["q_v"]), bf(ds["k"]), bf(ds["v"]), ds["table"], ds["prefix"], bl,
                           nld.NLD_MODE_VERIFY, ds["out_v"], None, ws)
        nld.nld_accept(ds["draft"], ds["verify"], ds["acc"])
        h_out.copy_(ds["out"], non_blocking=True)

    def step(cur, nxt):
        # compute on `cur` while the copy stream fills `nxt`; join before the next step
        main = torch.cuda.current_stream(dev)
        fork = torch.cuda.Event()
        fork.record(main)
        copy_stream.wait_event(fork)
        with torch.cuda.stream(copy_stream):
            copy_into(nxt)
        done = torch.cuda.Event()
        done.record(copy_stream)
        compute(cur)
        main.wait_event(done)

    nsteps = max(2, min(args.steps, 3000)) // 2 * 2
    with torch.cuda.stream(stream):
        copy_into(sets[0])
        for _ in range(2):
            step(sets[0], sets[1])
            step(sets[1], sets[0])
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step(sets[0], sets[1])
            step(sets[1], sets[0])
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(nsteps // 2):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / nsteps
    h2d = int(h_k.numel() * h_k.element_size() + h_v.numel() * h_v.element_size() + h_small.numel())
    d2h = int(h_out.numel())
    return {"value": round(2 * kv_bytes * world / (ms * 1e-3) / 1e9, 2), "unit": "GB/s",
            "ms_per_step": ms, "steps": nsteps, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "note": "every input (the whole K/V pool, queries, page table, lengths, ids, confidences) copied "
                    "from pinned host memory each step and the results read back, in a CUDA graph; inputs "
                    "double-buffered so that the next step's copy overlaps this step's kernels"}


# ---------------------------------------------------------------------------
# the other named workloads (each with its own step sequence)
# ---------------------------------------------------------------------------

def time_graph(torch, stream, body, nsteps, reps):
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        body(0)  # eager once (per-device setup outside the capture)
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=stream):
            for i in range(nsteps):
                body(i)
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / (reps * nsteps)


def run_quadss(torch, nld, dev, stream, peak, l2):
    """One quadratic self-speculation pass (Sec. 3 variant: drafting and
    verification in one forward with the structured mask) at the 8B shape
    (B=1, 32/8 heads, D=128, 4096-token prefix) for k = 3 and 5 (13 and 31
    block slots), next to a verify pass of the same block length: us per
    pass and KV GB/s over rotating cold pools."""
    res = {}
    gen = torch.Generator(device=dev)
    gen.manual_seed(17)
    B, Hq, Hkv, D, P, L = 1, 32, 8, 128, 16, 4096
    for k in (3, 5):
        bl = 1 + k + k * k
        pages = (L + bl + P - 1) // P
        kvb = (L + bl) * Hkv * D * 2 * 2
        npool = int(max(2, np.ceil(3 * l2 / kvb)))
        pools = [(torch.randn((pages, Hkv, P, D), generator=gen, device=dev).to(torch.bfloat16),
                  torch.randn((pages, Hkv, P, D), generator=gen, device=dev).to(torch.bfloat16)) for _ in range(npool)]
        table = torch.randperm(pages, generator=gen, device=dev).to(torch.int32).view(1, pages)
        prefix = torch.full((B,), L, dtype=torch.int32, device=dev)
        q = torch.randn((B, bl, Hq, D), generator=gen, device=dev).to(torch.bfloat16)
        out = torch.empty_like(q)
        p = nld.make_params(B, Hq, Hkv, D, P, pages, pages, 0, 0.0, 0)
        ws = torch.zeros(max(16, nld.nld_block_attn_workspace_size(p, bl)), dtype=torch.uint8, device=dev)
        bm = torch.from_numpy(nld.nld_quadss_block_mask(k).view(np.int32)).to(dev)
        masked = lambda i: nld.nld_block_attn_masked(p, q, pools[i % npool][0], pools[i % npool][1], table, prefix, bl,
                                                     bm, out, None, ws)
        verify = lambda i: nld.nld_block_attn(p, q, pools[i % npool][0], pools[i % npool][1], table, prefix, bl,
                                              nld.NLD_MODE_VERIFY, out, None, ws)
        us_m = time_graph(torch, stream, masked, 2 * npool, 10) * 1e3
        us_v = time_graph(torch, stream, verify, 2 * npool, 10) * 1e3
        res[f"k{k}_bl{bl}"] = {"quadss_us_per_pass": round(us_m, 3), "verify_us_per_pass": round(us_v, 3),
                               "quadss_kv_gbs": round(kvb / (us_m * 1e-6) / 1e9, 1),
                               "quadss_pct_of_hbm_peak": round(100 * kvb / (us_m * 1e-6) / 1e9 / peak, 2),
                               "kv_bytes_per_pass": kvb}
        del pools
    res["timing"] = "CUDA graph of back-to-back passes over rotating cold KV pools (attention + combine)"
    return res


def run_kv_commit(torch, nld, dev, stream):
    """nld_kv_commit of one verify step's accepted rows (counts from the accept
    rule's typical length, advance) at the 8B shape (B=1, bl=16) and for 128
    sequences (bl=8): us per call; bytes moved = 2 x (read + write) of the
    committed K/V rows."""
    res = {}
    gen = torch.Generator(device=dev)
    gen.manual_seed(13)
    for B, bl in ((1, 16), (128, 8)):
        Hkv, D, P = 8, 128, 16
        L = 4096
        pages = (L + bl + P - 1) // P
        num_pages = B * pages
        kp = torch.zeros((num_pages, Hkv, P, D), dtype=torch.bfloat16, device=dev)
        vp = torch.zeros_like(kp)
        table = torch.arange(num_pages, dtype=torch.int32, device=dev).view(B, pages)
        prefix = torch.full((B,), L, dtype=torch.int32, device=dev)
        k_new = torch.randn((B, bl, Hkv, D), generator=gen, device=dev).to(torch.bfloat16)
        v_new = torch.randn_like(k_new)
        counts = torch.full((B,), bl, dtype=torch.int32, device=dev)
        p = nld.make_params(B, 4 * Hkv, Hkv, D, P, num_pages, pages, 0, 0.0, 0)
        us = time_graph(torch, stream, lambda i: nld.nld_kv_commit(p, k_new, v_new, counts, table, prefix, bl, False,
                                                                   kp, vp), 64, 10) * 1e3
        moved = 2 * 2 * B * bl * Hkv * D * 2
        res[f"b{B}_bl{bl}"] = {"us_per_call": round(us, 3), "gbs_moved": round(moved / (us * 1e-6) / 1e9, 1)}
    res["timing"] = "CUDA graph of 64 back-to-back calls (no advance, so every call writes the same slots)"
    return res


def run_logits(torch, nld, dev, stream, peak, l2):
    """nld_logits_argmax over a 131072-token vocabulary for the positions of
    one step: 16 (8B shape, one diffusion block), 512 (14B shape, 16 x 32) and
    1024 (128 sequences x 8 verify positions). Logits bytes read / time, cold:
    each call reads its own buffer from a rotation past 3x L2."""
    V = 131072
    res = {}
    gen = torch.Generator(device=dev)
    gen.manual_seed(11)
    for rows in (16, 512, 1024):
        nbytes = rows * V * 2
        nbuf = int(max(1, np.ceil(3 * l2 / nbytes)))
        bufs = [(torch.randn((rows, V), generator=gen, device=dev) * 3).to(torch.bfloat16) for _ in range(nbuf)]
        ids = torch.empty((rows,), dtype=torch.int32, device=dev)
        conf = torch.empty((rows,), dtype=torch.float32, device=dev)
        ncall = max(nbuf, 8)
        us = time_graph(torch, stream, lambda i: nld.nld_logits_argmax(bufs[i % nbuf], ids, conf), ncall, 10) * 1e3
        gbs = nbytes / (us * 1e-6) / 1e9
        res[f"rows{rows}_v{V}"] = {"us_per_call": round(us, 3), "logits_gbs": round(gbs, 1),
                                   "pct_of_hbm_peak": round(100 * gbs / peak, 2), "buffers": nbuf}
        if rows <= 512:
            # the ensemble verifier reads two logits rows per position (AR and diffusion)
            npair = max(1, nbuf // 2)
            us_e = time_graph(torch, stream, lambda i: nld.nld_logits_ensemble_argmax(
                bufs[(2 * i) % (2 * npair)], bufs[(2 * i + 1) % (2 * npair)], 0.5, ids, conf), max(npair, 8), 10) * 1e3
            gbs_e = 2 * nbytes / (us_e * 1e-6) / 1e9
            res[f"ensemble_rows{rows}_v{V}"] = {"us_per_call": round(us_e, 3), "logits_gbs": round(gbs_e, 1),
                                               "pct_of_hbm_peak": round(100 * gbs_e / peak, 2)}
        del bufs
    res["timing"] = "CUDA graph of back-to-back calls over rotating buffers, events around 10 replays"
    return res


def run_decisions(torch, nld, dev, stream):
    """Each token-decision kernel alone (latency-bound: a few hundred bytes per
    sequence), as a CUDA graph of back-to-back calls: us per call at B = 1 and
    B = 128 sequences of n = 32 positions."""
    res = {}
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    for B in (1, 128):
        n = 32
        conf = torch.rand((B, n), generator=gen, device=dev)
        ids_a = torch.randint(0, 131072, (B, n), generator=gen, device=dev, dtype=torch.int32)
        ids_b = torch.where(torch.rand((B, n), generator=gen, device=dev) < 0.7, ids_a, ids_a + 1)
        pos_k = torch.empty((B, 8), dtype=torch.int32, device=dev)
        pos_n = torch.empty((B, n), dtype=torch.int32, device=dev)
        nsel = torch.empty((B,), dtype=torch.int32, device=dev)
        acc = torch.empty((B,), dtype=torch.int32, device=dev)
        calls = {
            "accept": lambda i: nld.nld_accept(ids_a, ids_b, acc),
            "unmask_top8": lambda i: nld.nld_unmask(conf, 8, pos_k, nsel),
            "unmask_threshold_0.9": lambda i: nld.nld_unmask_threshold(conf, 0.9, pos_n, nsel),
            "greedy_accept": lambda i: nld.nld_greedy_accept(ids_a, ids_b, conf, pos_n, nsel),
        }
        res[f"b{B}_n{n}_us_per_call"] = {k: round(time_graph(torch, stream, f, 256, 10) * 1e3, 3)
                                          for k, f in calls.items()}
    res["timing"] = "CUDA graph of 256 back-to-back calls (PDL), events around 10 replays"
    return res


SWEEP_SPLITS = (1, 2, 4, 8, 12, 14, 16, 17, 18, 19, 20, 24, 32, 48, 64)


def split_sweep(torch, nld, stream, w, pools, out, lse, peak):
    """Verify-pass time over explicit KV split counts, two ways: the default
    plan (pieces of 2/4/8 dividing S merge as thread-block clusters) and
    every piece its own partial merged by the combine kernel
    (NLD_ATTN_NO_CLUSTER). `partial_bytes` = S x B x Hq x bl x (2 D + 4) (bf16 rows, fp32 lse),
    written once by the attention kernel and read once by the combine."""
    B, bl, Hq, Hkv, D = w["batch"], w["bl"], w["hq"], w["hkv"], w["d"]
    kvb = w["kv_bytes_per_pass"]
    variants = (("clusters", 0), ("no_cluster", nld.NLD_ATTN_NO_CLUSTER))
    sweep = {}
    for vname, vflags in variants:
        curve = {}
        for S in SWEEP_SPLITS:
            pS = nld.make_params(B, Hq, Hkv, D, w["page"], w["num_pages"], w["max_pages"], S, 0.0,
                                 nld.NLD_ATTN_PREFIX_READY | vflags)
            plan = nld.nld_block_attn_plan(pS, bl, torch.cuda.get_device_properties(0).multi_processor_count)
            wsS = torch.zeros(max(nld.nld_block_attn_workspace_size(pS, bl), 16), dtype=torch.uint8,
                              device=out.device)

            def one(i, pS=pS, wsS=wsS):
                kp, vp = pools[i % len(pools)]
                nld.nld_block_attn(pS, w["q_verify"], kp, vp, w["page_table"], w["prefix_lens"], bl,
                                   nld.NLD_MODE_VERIFY, out, lse, wsS)
            msS = time_graph(torch, stream, one, 16, reps=8)
            parts = nld.nld_block_attn_num_splits(pS, bl)
            gbs = kvb / (msS * 1e-3) / 1e9
            curve[str(S)] = {"us_per_pass": round(msS * 1e3, 2), "kv_gbs": round(gbs, 1),
                             "pct_of_hbm_peak": round(100 * gbs / peak, 2), "pieces": plan["splits"],
                             "cluster": plan["cluster"], "kv_partials": parts,
                             "kernels": nld.nld_block_attn_kernels(pS, bl),
                             "partial_bytes": (parts * B * Hq * bl * (2 * D + 4)) if parts > 1 else 0}
            del wsS
        sweep[vname] = curve
    return sweep


def run_workloads(torch, nld, dev, stream, peak, l2, only=None, batch=None, sweep_splits=False):
    """Each named workload's step (its attention passes, then its decisions),
    inputs drawn on the device, pools rotated past L2 where the KV is smaller
    than three times L2."""
    res = {}
    for name in W.WORKLOADS:
        if (only is None and name == WORKLOAD) or (only is not None and name != only):
            continue
        w = W.make_device_workload(name, seed=0, device=dev, batch=batch)
        B, bl, Hq, Hkv, D = w["batch"], w["bl"], w["hq"], w["hkv"], w["d"]
        kvb = w["kv_bytes_per_pass"]
        npool = int(min(64, max(1, np.ceil(3 * l2 / kvb))))
        pools = [(w["k"], w["v"])] + [(w["k"].clone(), w["v"].clone()) for _ in range(npool - 1)]
        params = nld.make_params(B, Hq, Hkv, D, w["page"], w["num_pages"], w["max_pages"], 0, 0.0,
                                 nld.NLD_ATTN_PREFIX_READY)
        parts = nld.nld_block_attn_num_splits(params, bl)
        ws = torch.zeros(max(nld.nld_block_attn_workspace_size(params, bl), 16), dtype=torch.uint8, device=dev)
        out = torch.empty((B, bl, Hq, D), dtype=torch.bfloat16, device=dev)
        lse = torch.empty((B, Hq, bl), dtype=torch.float32, device=dev)
        acc = torch.empty((B,), dtype=torch.int32, device=dev)
        kk = max(w["unmask_k"])
        pos = torch.empty((B, kk), dtype=torch.int32, device=dev)
        nsel = torch.empty((B,), dtype=torch.int32, device=dev)
        seq = w["steps"]
        npass = sum(1 for s_ in seq if s_ in ("diffusion", "verify"))
        counter = {"p": 0}

        def step(i, seq=seq, pools=pools, params=params):
            for s_ in seq:
                if s_ in ("diffusion", "verify"):
                    kp, vp = pools[counter["p"] % len(pools)]
                    counter["p"] += 1
                    mode = nld.NLD_MODE_DIFFUSION if s_ == "diffusion" else nld.NLD_MODE_VERIFY
                    q = w["q_draft"] if s_ == "diffusion" else w["q_verify"]
                    nld.nld_block_attn(params, q, kp, vp, w["page_table"], w["prefix_lens"], bl, mode, out, lse, ws)
                elif s_ == "accept":
                    nld.nld_accept(w["draft_ids"], w["verify_ids"], acc)
                elif s_ == "unmask":
                    nld.nld_unmask(w["conf"][0], kk, pos, nsel)

        nsteps = max(1, min(64, 512 // max(1, len(seq))))
        ms = time_graph(torch, stream, step, nsteps, reps=8)
        gbs = npass * kvb / (ms * 1e-3) / 1e9
        entry = {"step": " + ".join(seq), "ms_per_step": round(ms, 5), "kv_gbs": round(gbs, 1),
                 "pct_of_hbm_peak": round(100 * gbs / peak, 2), "steps_per_s": round(1e3 / ms, 1),
                 "kv_bytes_per_pass": kvb, "kv_partials": parts,
                 "l2": ("cold: %d rotating pools" % npool) if npool * kvb >= 3 * l2 else
                       "warm: KV fits in L2 (%d pools, launch-bound shape)" % npool}
        if (name.startswith("long") and only is None) or sweep_splits:
            entry["verify_pass_split_sweep"] = split_sweep(torch, nld, stream, w, pools, out, lse, peak)
        res[name] = entry
        del pools, w
        torch.cuda.empty_cache()
    return res


# ---------------------------------------------------------------------------
# CPU oracle timings
# ---------------------------------------------------------------------------

def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo), for the baseline records."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                name = line.split(":", 1)[1].strip()
                if name and not name.isdigit():
                    return name
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu model", "hardware")):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


def headline_config(wl, npool, l2, splits, attn_kernels, prefix_ready):
    """The config dict of the headline workload, shared by both arms."""
    c = wl.attn
    kv_bytes = c.kv_bytes_per_pass()
    return {
        "workload": WORKLOAD,
        "batch_per_gpu": c.batch, "q_heads": c.num_q_heads, "kv_heads": c.num_kv_heads, "head_dim": c.head_dim,
        "prefix": int(c.kv.prefix_lens[0]), "block_len": c.block_len, "page_size": c.page_size,
        "page_order": "random permutation", "kv_partials": splits, "attn_kernels_per_pass": attn_kernels,
        "split_merge": "combine kernel" if attn_kernels == 2 else "none (one partial per row)",
        "unmask_k": wl.unmask_k[0], "prefix_ready_flag": prefix_ready,
        "step": "diffusion attention + unmask + verify attention + accept (one attention layer)",
        "l2": f"cold: each pass reads its own KV pool from a rotation of {npool} pools "
              f"({npool * kv_bytes / 2**20:.0f} MiB > 3x L2 {l2 / 2**20:.0f} MiB)",
        "timing": "CUDA graph of the steps, CUDA events on the launching stream",
    }


def pool_count(kv_bytes, l2, pools_arg):
    npool = max(pools_arg, 2)
    if npool * kv_bytes < 3 * l2:
        npool = int(np.ceil(3 * l2 / kv_bytes)) + 1
    return npool + npool % 2


def oracle_step(orc, wl, rows=None):
    """One draft+verify step on the oracle: both passes (all rows, or the
    given (b, i, h) rows), unmask and accept."""
    c = wl.attn
    kv = c.kv
    for mode, qb in ((W.MODE_DIFFUSION, c.q_draft_bits), (W.MODE_VERIFY, c.q_verify_bits)):
        if rows is None:
            orc.block_attn(qb, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens, c.num_q_heads, c.num_kv_heads,
                           c.block_len, mode, c.scale)
        else:
            orc.block_attn_rows(qb, kv.k_bits, kv.v_bits, kv.page_table, kv.prefix_lens, c.num_q_heads,
                                c.num_kv_heads, c.block_len, mode, c.scale, rows)
        if mode == W.MODE_DIFFUSION:
            orc.unmask(wl.conf[0], wl.unmask_k[0])
    orc.accept(wl.draft_ids, wl.verify_ids)


def cpu_baseline(wl, budget_s: float):
    import oracle
    orc = oracle.load()
    kv_bytes = wl.attn.kv_bytes_per_pass()
    n = 0
    t0 = time.perf_counter()
    while True:
        oracle_step(orc, wl)
        n += 1
        if time.perf_counter() - t0 > budget_s or n >= 50:
            break
    dt = time.perf_counter() - t0
    return {"value": round(2 * kv_bytes * n / dt / 1e9, 4), "unit": "GB/s", "cores": orc.max_threads(),
            "cpu_model": cpu_model(), "kind": "oracle", "steps_per_s": round(n / dt, 3),
            "sample": f"{n} full draft+verify steps (every row of both passes, unmask, accept) of {WORKLOAD}, "
                      f"fp64, OpenMP over (sequence, query head)"}


def reference_config(args, wl):
    """The GPU arm's config dict for the same workload: the split plan from
    the host-only plan query for this machine's GPU (no device work), the pool
    rotation from its L2 size."""
    from paper_2607_05722_gb300 import build as nld_build
    from paper_2607_05722_gb300 import nld
    nld_build.build()  # the host-only plan query lives in the library (no kernel runs)
    c = wl.attn
    sms, l2 = 152, 129 << 20
    try:
        import torch
        if torch.cuda.is_available():
            prop = torch.cuda.get_device_properties(0)
            sms, l2 = prop.multi_processor_count, prop.L2_cache_size
    except Exception:  # noqa: BLE001 - the plan falls back to the GB300 figures
        pass
    prefix_ready = not args.no_prefix_ready
    params = nld.make_params(c.batch, c.num_q_heads, c.num_kv_heads, c.head_dim, c.page_size, c.kv.num_pages,
                             c.kv.max_pages, args.splits, 0.0, nld.NLD_ATTN_PREFIX_READY if prefix_ready else 0)
    plan = nld.nld_block_attn_plan(params, c.block_len, sms)
    kernels = 2 if plan["partials"] > 1 else 1
    npool = pool_count(c.kv_bytes_per_pass(), l2, args.pools)
    return headline_config(wl, npool, l2, plan["partials"], kernels, prefix_ready)


def run_reference(args, world, rank):
    if rank != 0:
        return
    import oracle
    orc = oracle.load()
    wl = W.make_workload(WORKLOAD, seed=args.seed)
    c = wl.attn
    kv_bytes = c.kv_bytes_per_pass()
    total_rows = c.batch * c.block_len * c.num_q_heads
    rng = np.random.default_rng(7)
    all_rows = np.array([(b, i, h) for b in range(c.batch) for i in range(c.block_len)
                         for h in range(c.num_q_heads)], dtype=np.int32)
    # calibrate the per-row cost, then size each step's sample so the run stays
    # within about two minutes
    probe = all_rows[rng.permutation(total_rows)[:64]]
    t0 = time.perf_counter()
    oracle_step(orc, wl, probe)
    per_row = (time.perf_counter() - t0) / (2 * len(probe))
    budget = 120.0 / max(1, args.steps + args.warmup)
    nrows = int(np.clip(budget / (2 * per_row), 1, total_rows))
    sample = all_rows[rng.permutation(total_rows)[:nrows]]
    for _ in range(args.warmup):
        oracle_step(orc, wl, sample)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(orc, wl, sample)
    dt = time.perf_counter() - t0
    frac = nrows / total_rows
    value = 2 * kv_bytes * frac * args.steps / dt / 1e9
    desc = (f"{nrows} of {total_rows} query rows of both passes per step (+ unmask, accept), {WORKLOAD}, "
            f"fp64 oracle, OpenMP over rows")
    line = {
        "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3 / frac, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": reference_config(args, wl),
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": orc.max_threads(),
                         "cpu_model": cpu_model(), "kind": "oracle", "sample": desc},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    world, rank, local = dist_env()
    if args.gpus != world and world > 1:
        print(f"--gpus {args.gpus} but WORLD_SIZE {world}", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args, world, rank)
        return
    if args.only_workload is not None:
        run_only_workload(args, local)
        return
    if args.only_section is not None:
        run_only_section(args, local)
        return
    run_ours(args, world, rank, local)


if __name__ == "__main__":
    main()
