"""Benchmark of the RhymeFlow asynchronous step core on GB300.

A "step" is one asynchronous denoising step of the trajectory, all five
library calls (compaction, Eq. 3 projection of the latents, Eq. 3 projection of
the skipped frames' keys and values from the rolling cache, active-query
attention, Euler update) over the workload's synthetic inputs resident in HBM.  Timed step k is
schedule step s = k mod S, so K = S steps is one whole trajectory.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config long]
    python bench.py --impl reference ...   # the CPU oracle on the host cores

value        attention TFLOP/s of the whole step core (algorithmic FLOPs
             4 * active_rows * F*N * d * H summed over the timed steps, divided
             by the device time of the timed steps), summed over ranks
roofline     rf_attn alone: its algorithmic FLOPs per launch / its average launch
             time (CUDA events around each launch on the launching stream)
e2e          the same metric with every step's inputs copied from pinned host
             memory and its outputs read back, inside the timed region
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "rf_attn TFLOP/s (% BF16 peak); step-core ms vs all-frames-active on 1 GB300"
UNIT = "TFLOP/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM traffic of rf_attn launches measured with ncu (dram__bytes_read.sum +
# dram__bytes_write.sum), per workload.  A figure is reported only while the kernel source
# still has the hash it was measured with.
ATTN_TRAFFIC = {
    "small": {"code_sha256_rf_attn_cu": "70d6f3611b001ebc671ab73df654848676226a2001c8d47726bc16900d557f9a",
              "bytes_per_launch": 190560333,
              "launch": "average over the 20 launches of one trajectory of the small workload "
                        "(10 with all 13 frames active, 10 with the 4 keyframes)"},
    "long": {"code_sha256_rf_attn_cu": "70d6f3611b001ebc671ab73df654848676226a2001c8d47726bc16900d557f9a",
             "bytes_per_launch": 5118625213,
             "launch": "average over the 50 launches of one trajectory of the long workload "
                       "(21 with all 33 frames active, 29 with the 6 keyframes)"},
}


def _env_rank():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def _code_sha(path):
    """sha256 of a C++/CUDA source with its // comments and blank lines removed: counters
    recorded for a kernel stay attached to it while only comments change.  (The source holds
    no "//" inside string literals.)"""
    lines = []
    for line in open(path, encoding="utf-8"):
        code = line.split("//", 1)[0].rstrip()
        if code:
            lines.append(code)
    return hashlib.sha256("\n".join(lines).encode()).hexdigest()


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) != 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for _, _, flags in rows for n, fl in zip(names, flags)
                          if fl.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows)}


def combine_ranks(ms_local: float, flops_local: float, dist=None, device="cpu"):
    """Whole-job throughput of N replicas: the slowest rank's time (all ranks start together
    after a barrier) and every rank's FLOPs.  Returns (max_ms, total_flops, TFLOP/s)."""
    import torch
    t = torch.tensor([ms_local, flops_local], dtype=torch.float64, device=device)
    if dist is not None and dist.is_initialized() and dist.get_world_size() > 1:
        ms_t = t[:1].clone()
        fl_t = t[1:].clone()
        dist.all_reduce(ms_t, op=dist.ReduceOp.MAX)
        dist.all_reduce(fl_t, op=dist.ReduceOp.SUM)
        t = torch.cat([ms_t, fl_t])
    max_ms, total = float(t[0].item()), float(t[1].item())
    return max_ms, total, total / (max_ms * 1e-3) / 1e12


def _gpu_index(local_rank):
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [x.strip() for x in vis.split(",")]
        if local_rank < len(ids) and ids[local_rank].isdigit():
            return int(ids[local_rank])
    return local_rank


# ---------------------------------------------------------------------------
# The GPU arm
# ---------------------------------------------------------------------------
def run_gpu(args):
    import torch
    import workloads as wl
    import paper_2606_06309_gb300 as rf
    from paper_2606_06309_gb300.stepcore import StepCore, upload_plan

    rank, world, local = _env_rank()
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    rf.load()
    dev = torch.device("cuda", local)
    w = wl.get(args.config)
    E = w.N * w.C
    S = w.S
    plan = upload_plan(w.F, w.S, w.is_key, w.stride, w.T_w, dev)
    core = StepCore(w.F, w.N, E, w.H, w.d, plan, dev)
    core.set_state(wl.latents(w, device=dev))
    Q, K, V = wl.qkv(w, device=dev)
    core.set_kv_cache(K, V)
    O = torch.empty_like(Q)
    vel = [wl.velocity(w, s, device=dev) for s in range(S)]
    stream = torch.cuda.current_stream(dev)
    mask_host = plan.host["mask"]
    A_per_step = mask_host.sum(axis=1)
    flops_step = [4 * int(A_per_step[s]) * w.N * w.S_tok * w.d * w.H for s in range(S)]

    # all-frames-active comparison plan (mask = 1, every frame one step)
    plan_all = upload_plan(w.F, w.S, [1] * w.F, [1] * S, 0, dev)
    core_all = StepCore(w.F, w.N, E, w.H, w.d, plan_all, dev)
    core_all.set_state(wl.latents(w, device=dev))
    core_all.set_kv_cache(K, V)
    flops_all = 4 * w.F * w.N * w.S_tok * w.d * w.H

    def barrier():
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
            torch.cuda.synchronize()

    def timed(c, K_steps, W_steps, per_launch=False):
        for k in range(W_steps):
            c.run(k % S, vel[k % S], O, Q, K, V, w.softmax_scale)
        barrier()
        ev = [] if per_launch else None
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for k in range(K_steps):
            s = k % S
            c.compact(s)
            c.project(s)
            c.project_kv(s, K, V)
            if per_launch:
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record(stream)
                c.attn(O, Q, K, V, w.softmax_scale)
                b.record(stream)
                ev.append((s, a, b))
            else:
                c.attn(O, Q, K, V, w.softmax_scale)
            c.step(s, vel[s])
        t1.record(stream)
        barrier()
        ms = t0.elapsed_time(t1)
        return ms, ev

    K_steps, W_steps = args.steps, args.warmup
    with ClockSampler(_gpu_index(local)) as clk:
        ms, _ = timed(core, K_steps, W_steps)
    clocks = clk.summary()
    # slowest rank's time, every rank's work
    ms, total_flops, value = combine_ranks(
        ms, float(sum(flops_step[k % S] for k in range(K_steps))), dist, dev)

    # per-launch attention timing for the roofline (separate pass, same work)
    _, ev = timed(core, K_steps, 0, per_launch=True)
    launch_ms = [a.elapsed_time(b) for _, a, b in ev]
    attn_ms_total = sum(launch_ms)
    attn_flops_total = sum(flops_step[s] for s, _, _ in ev)
    achieved = attn_flops_total / (attn_ms_total * 1e-3) / 1e12
    per_launch_flops = attn_flops_total / len(ev)
    # all-frames-active comparison, same number of steps
    ms_all, _ = timed(core_all, K_steps, min(W_steps, 3))
    # the step core's five launches, each timed on its own over one trajectory (the latent-width
    # kernels are launch-bound, so their microseconds are reported, not GB/s)
    parts = {"rf_schedule_compact": [], "rf_project": [], "rf_project_kv": [], "rf_attn": [],
             "rf_step": []}
    for k in range(S):
        calls = (("rf_schedule_compact", lambda: core.compact(k)),
                 ("rf_project", lambda: core.project(k)),
                 ("rf_project_kv", lambda: core.project_kv(k, K, V)),
                 ("rf_attn", lambda: core.attn(O, Q, K, V, w.softmax_scale)),
                 ("rf_step", lambda: core.step(k, vel[k])))
        for name, fn in calls:
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            parts[name].append((a, b))
    barrier()
    breakdown_us = {n: round(1000 * statistics.mean(a.elapsed_time(b) for a, b in v), 2)
                    for n, v in parts.items()}
    # per schedule step: attention launch time against the all-active launch
    _, ev_all = timed(core_all, S, 3, per_launch=True)
    attn_all_ms = statistics.mean(a.elapsed_time(b) for _, a, b in ev_all)
    by_step = {}
    for (s_, _, _), t in zip(ev, launch_ms):
        by_step.setdefault(s_, []).append(t)
    per_step_ms = [statistics.mean(by_step[s_]) if s_ in by_step else None for s_ in range(S)]
    per_step = {
        "attn_ms": [round(t, 5) if t is not None else None for t in per_step_ms],
        "attn_ms_all_active": round(attn_all_ms, 5),
        "attn_speedup": [round(attn_all_ms / t, 3) if t else None for t in per_step_ms],
        "ideal_attn_speedup": [round(w.F / int(A_per_step[s_]), 3) if A_per_step[s_] else None
                               for s_ in range(S)],
    }
    # the same trajectory replayed from one CUDA graph (launch overhead removed)
    graph_ms = None
    try:
        g = core.capture_trajectory(vel, O, Q, K, V, w.softmax_scale)
        reps = max(1, K_steps // S)
        g.replay()
        barrier()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        barrier()
        graph_ms = a.elapsed_time(b) / (reps * S)
        del g
    except RuntimeError as e:  # report, never hide: the eager numbers above stand
        graph_ms = f"capture failed: {e}"

    # end to end through the public API with host buffers
    e2e = run_e2e(args, w, core, plan, Q, K, V, vel, flops_step, stream, barrier, dist, world)

    peaks, peak_src = _peaks()
    traffic = None
    attn_src = os.path.join(ROOT, "paper_2606_06309_gb300", "csrc", "rf_attn.cu")
    tr = ATTN_TRAFFIC.get(args.config)
    if tr is not None and tr["code_sha256_rf_attn_cu"] == _code_sha(attn_src):
        traffic = tr["bytes_per_launch"]
    bw = run_bandwidth(w, dev, peaks) if not args.no_bandwidth else None
    sweep = run_sweep(w, dev, Q, K, V, O, vel, max(3, min(K_steps, 10))) if w.sweep else None
    block = run_block_mask(w, dev, Q, K, V, O, plan, core) if not args.no_bandwidth else None
    status = int(core.status.item()) | int(core_all.status.item())

    out = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": K_steps, "warmup": W_steps, "ms_per_step": round(ms / K_steps, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {
            "workload": _workload_name(w),
            "keyframes": list(w.keyframes), "stride": f"{w.stride[0]}..{w.stride[-1]}",
            "active_frames_per_step_avg": float(A_per_step.mean()),
            "l2": _l2_note(3 * Q.numel() * 2, dev),
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "peak_source": peak_src,
        },
        "step_core_ms": round(ms / K_steps, 5),
        "step_core_ms_all_active": round(ms_all / K_steps, 5),
        "step_core_ms_cuda_graph": round(graph_ms, 5) if isinstance(graph_ms, float) else graph_ms,
        "speedup_vs_all_active": round(ms_all / ms, 4),
        "ideal_speedup_vs_all_active": round(K_steps * flops_all /
                                             sum(flops_step[k % S] for k in range(K_steps)), 4),
        "per_step": per_step,
        "step_core_breakdown_us": breakdown_us,
        "roofline": {
            "bound": "tensor", "kernel": "rf_attn", "achieved": round(achieved, 2),
            "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
            "frac": round(achieved / peaks["bf16_tflops"], 4),
            "frac_of_sustained": round(achieved / peaks["bf16_tflops_sustained"], 4),
            "traffic": traffic,
            "traffic_launch": tr["launch"] if traffic is not None else None,
            "flops_per_launch": per_launch_flops,
            "avg_launch_ms": round(attn_ms_total / len(ev), 5),
        },
        "bandwidth_kernels": bw,
        "active_fraction_sweep": sweep,
        "combined_block_mask": block,
        "e2e": e2e,
        "gpu_launches": core.launches_per_step * K_steps,
        "clocks": clocks,
        "device_status": status,
    }
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(w, budget_s=args.cpu_budget)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(out), flush=True)


def _l2_note(qkv_bytes, dev):
    """How the timed steps relate to L2: every workload but the smallest streams Q/K/V from
    HBM; the smallest fits in L2 and is timed warm (it is a parity case, not a bench line)."""
    import torch
    l2 = getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0) or 129 * 2 ** 20
    if qkv_bytes > l2:
        return f"inputs larger than L2: Q/K/V {qkv_bytes / 1e6:.0f} MB, L2 {l2 / 1e6:.0f} MB"
    return (f"inputs fit in L2 (Q/K/V {qkv_bytes / 1e6:.2f} MB, L2 {l2 / 1e6:.0f} MB): timed "
            "warm, not flushed")


def run_e2e(args, w, core, plan, Q, K, V, vel, flops_step, stream, barrier, dist, world):
    """End to end through the library's host-fed pipeline (rf_pipeline_step: one C-ABI call
    per step, host pointers in and out).  Every step copies the active frames' Q, K and V rows
    and the velocity from pinned host memory and reads the attention output's active rows,
    the latent context and the latent store back, with the copies of neighbouring steps
    overlapped with compute (two copy streams, three device buffer sets)."""
    import torch
    from paper_2606_06309_gb300.stepcore import HostPipeline
    S = w.S
    hQ, hK, hV = (x.cpu().pin_memory() for x in (Q, K, V))
    hv = [v.cpu().pin_memory() for v in vel]
    hO = torch.empty(Q.shape, dtype=Q.dtype).pin_memory()
    hz = torch.empty(core.z2.shape, dtype=core.z2.dtype).pin_memory()
    hc = torch.empty(core.ctx.shape, dtype=core.ctx.dtype).pin_memory()
    pipe = HostPipeline(core, w.S_tok, hK, hV, Q.device)
    K_steps = max(1, min(args.steps, args.e2e_steps))
    for k in range(3):
        pipe.step(k % S, hQ, hK, hV, hv[k % S], hO, hz, w.softmax_scale, hctx=hc)
    barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(pipe.h2d)
    for k in range(K_steps):
        pipe.step(k % S, hQ, hK, hV, hv[k % S], hO, hz, w.softmax_scale, hctx=hc)
    t1.record(pipe.d2h)
    barrier()
    ms, flops, _ = combine_ranks(t0.elapsed_time(t1),
                                 float(sum(flops_step[k % S] for k in range(K_steps))), dist,
                                 Q.device)
    h2d, d2h = pipe.bytes_per_step(last=K_steps)
    status = pipe.sync()
    pipe.close()
    # this machine's host->device copy rate (pinned, 256 MB, after the timed region): the step's
    # input copies take h2d / rate, which bounds the e2e figure where it exceeds the compute
    src = torch.empty(64 * 2 ** 20, dtype=torch.float32).pin_memory()
    dst = torch.empty_like(src, device=Q.device)
    dst.copy_(src, non_blocking=True)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(5):
        dst.copy_(src, non_blocking=True)
    b.record()
    torch.cuda.synchronize()
    h2d_gbs = 5 * src.numel() * 4 / (a.elapsed_time(b) * 1e-3) / 1e9
    del src, dst
    return {"value": round(flops / (ms * 1e-3) / 1e12, 3), "unit": UNIT, "steps": K_steps,
            "ms_per_step": round(ms / K_steps, 5), "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "api": "rf_pipeline_step", "device_status": status,
            "h2d_gbs_measured": round(h2d_gbs, 1),
            "h2d_ms_per_step_at_that_rate": round(h2d / (h2d_gbs * 1e9) * 1e3, 4),
            "overlap": "three buffer sets: H2D of steps k+1, k+2 and D2H of earlier steps "
                       "overlap the compute of step k",
            "copied": "in: active frames' Q, K and V rows, the velocity (skipped frames' keys "
                      "and values are projected from the device-resident cache); out: active "
                      "frames' O rows, the latent context, the latent store (bytes averaged "
                      "over the timed steps)"}


def _bw_sets(w, dev, R):
    """R independent input sets of the stress shape: latent store, velocity, context, K/V rows
    and K/V caches (set 0 seeded; the others copies of it)."""
    import torch
    import workloads as wl
    F, E, D = w.F, w.N * w.H * w.d, w.H * w.d
    z2 = torch.empty(2, F, E, device=dev)
    z2[0].copy_(wl.hidden_latents(w, 0, device=dev))
    z2[1].copy_(wl.hidden_latents(w, 1, device=dev))
    g = torch.Generator(device=dev).manual_seed(w.seed)
    base = {"z2": z2, "v": wl.hidden_latents(w, 2, device=dev),
            "ctx": torch.empty(F, E, device=dev),
            "K": torch.randn(F * w.N, D, generator=g, device=dev).to(torch.bfloat16),
            "V": torch.randn(F * w.N, D, generator=g, device=dev).to(torch.bfloat16),
            "Kc": torch.randn(2, F, w.N, D, generator=g, device=dev).to(torch.bfloat16),
            "Vc": torch.randn(2, F, w.N, D, generator=g, device=dev).to(torch.bfloat16)}
    return [base] + [{k: x.clone() for k, x in base.items()} for _ in range(R - 1)]


def run_bandwidth(w, dev, peaks):
    """rf_project, rf_project_kv and rf_step at the hidden-width stress shape (C = H*d fp32, the
    width of the per-layer rolling cache) on the keyframe-only step (the most skipped frames),
    and rf_step on the all-active step too.  Each kernel is timed two ways:
      back to back  R launches in a row over R distinct input sets, R chosen so that the other
                    R - 1 launches move more than twice L2's size between two uses of a set (so
                    every launch reads cold inputs); time per launch = the interval / R, median
                    of 7 repetitions.  The headline: the step core issues its kernels back to
                    back as well.
      single        one launch after a 256 MB write that flushes L2, median of 10; this includes
                    the launch latency between the two events."""
    import math
    import torch
    import workloads as wl
    import paper_2606_06309_gb300 as rf
    F, E, D = w.F, w.N * w.H * w.d, w.H * w.d
    p = rf.rf_plan_build(w.F, w.S, w.is_key, w.stride, w.T_w)
    s = _keyframe_step(p["mask"])
    A, A0 = int(p["mask"][s].sum()), int(p["mask"][0].sum())
    l2 = getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0) or 129 * 2 ** 20
    set_bytes = (5 * F * E) * 4 + 6 * F * w.N * D * 2
    read_min = 8 * A * E                               # the smallest launch: rf_step, step s
    R = 1 + math.ceil(2 * l2 / read_min)
    free = torch.cuda.mem_get_info(dev)[0]
    if set_bytes > 0.5 * free:
        return None
    R = max(1, min(R, 8, int(0.5 * free // set_bytes)))
    sets = _bw_sets(w, dev, R)

    def plan_row(step):
        row = {k: torch.from_numpy(p[k][step]).to(dev) for k in ("mask", "alpha", "beta",
                                                                 "cur_slot", "dt")}
        row["act"] = torch.zeros(F, dtype=torch.int32, device=dev)
        row["skp"] = torch.zeros(F, dtype=torch.int32, device=dev)
        row["cnt"] = torch.zeros(2, dtype=torch.int32, device=dev)
        rf.rf_schedule_compact(row["mask"], F, w.N, row["act"], row["skp"], None, row["cnt"])
        return row

    ps, p0 = plan_row(s), plan_row(0)
    kernels = (
        ("rf_project_kv", lambda b: rf.rf_project_kv(
            b["K"], b["V"], D, b["Kc"], b["Vc"], ps["cur_slot"], ps["alpha"], ps["beta"],
            ps["act"], ps["skp"], ps["cnt"], F, w.N, D), 2 * (6 * (F - A) + 4 * A) * w.N * D, s, A,
         f"K and V bf16 [{F * w.N}][{D}] + caches [2][{F}][{w.N}][{D}]"),
        ("rf_project", lambda b: rf.rf_project(b["ctx"], b["z2"], ps["cur_slot"], ps["alpha"],
                                               ps["beta"], F, E), (12 * (F - A) + 8 * A) * E, s, A,
         None),
        ("rf_step", lambda b: rf.rf_step(b["z2"], ps["cur_slot"], b["v"], ps["dt"], ps["act"],
                                         ps["cnt"], F, E), 12 * A * E, s, A, None),
        ("rf_step_all_active", lambda b: rf.rf_step(b["z2"], p0["cur_slot"], b["v"], p0["dt"],
                                                    p0["act"], p0["cnt"], F, E), 12 * A0 * E, 0,
         A0, None))
    flush = torch.empty(256 * 1024 * 1024 // 4, device=dev)
    res = {}
    for name, fn, nbytes, step, nact, shape in kernels:
        for b in sets:                                  # warm-up, every set
            fn(b)
        torch.cuda.synchronize()
        b2b = []
        for rep in range(7):
            flush.fill_(rep)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            for st in sets:
                fn(st)
            b.record()
            torch.cuda.synchronize()
            b2b.append(a.elapsed_time(b) / R)
        single = []
        for rep in range(10):
            flush.fill_(rep)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            fn(sets[0])
            b.record()
            torch.cuda.synchronize()
            single.append(a.elapsed_time(b))
        ms, ms1 = statistics.median(b2b), statistics.median(single)
        gbs, gbs1 = nbytes / (ms * 1e-3) / 1e9, nbytes / (ms1 * 1e-3) / 1e9
        res[name] = {"GB/s": round(gbs, 1), "frac": round(gbs / peaks["hbm_gbs"], 4),
                     "peak": peaks["hbm_gbs"], "ms": round(ms, 4), "bytes": nbytes,
                     "timing": f"back to back over {R} input sets",
                     "single_launch": {"GB/s": round(gbs1, 1),
                                       "frac": round(gbs1 / peaks["hbm_gbs"], 4),
                                       "ms": round(ms1, 4)},
                     "shape": (shape or f"F={F} x E={E} fp32 (C = H*d = {D})")
                              + f", step {step}, A={nact}"}
    # Denominators.  The measured peak is a copy (one read, one write per element); kernels that
    # read more than they write can exceed it.  Two library kernels with other read:write mixes,
    # timed the same way over 1 GiB fp32 operands, and the nominal HBM3e rate give context.
    nominal = 7900.0
    for v in res.values():
        v["frac_of_nominal_7900"] = round(v["GB/s"] / nominal, 4)
    n = 2 ** 28
    xa = torch.randn(n, device=dev)
    xb = torch.randn(n, device=dev)
    xc = torch.empty(n, device=dev)
    refs = {"torch_add_2_reads_1_write": (lambda: torch.add(xa, xb, out=xc), 12 * n),
            "torch_sum_read_only": (lambda: xa.sum(), 4 * n)}
    ref_out = {}
    for name, (fn, nbytes) in refs.items():
        for _ in range(3):
            fn()
        ts = []
        for rep in range(7):
            flush.fill_(rep)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        ms = statistics.median(ts)
        gbs = nbytes / (ms * 1e-3) / 1e9
        ref_out[name] = {"GB/s": round(gbs, 1), "frac": round(gbs / peaks["hbm_gbs"], 4),
                         "frac_of_nominal_7900": round(gbs / nominal, 4), "bytes": nbytes}
    res["library_references"] = ref_out
    del xa, xb, xc
    z2 = sets[0]["z2"]
    del sets
    # keyframe selection's inner products: proxies at latent width (where Algorithm 1 runs)
    # and at the hidden-width stress shape
    G = torch.empty(F, F, dtype=torch.float64, device=dev)
    for label, P in (("rf_frame_gram_latent", wl.latents(w, device=dev)), ("rf_frame_gram", z2[0])):
        times = []
        for rep in range(13):
            flush.fill_(rep)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            rf.rf_frame_gram(P, G)
            b.record()
            torch.cuda.synchronize()
            if rep >= 3:
                times.append(a.elapsed_time(b))
        ms = statistics.median(times)
        nbytes = P.numel() * 4
        res[label] = {"GB/s": round(nbytes / (ms * 1e-3) / 1e9, 1),
                      "frac": round(nbytes / (ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4),
                      "peak": peaks["hbm_gbs"], "ms": round(ms, 4), "bytes": nbytes,
                      "shape": f"F={F} proxies x E={P.shape[1]} fp32 -> [{F}][{F}] fp64"}
    del z2, flush
    torch.cuda.empty_cache()
    return res


def _keyframe_step(mask):
    """The first schedule step with the fewest active frames (the keyframes only, once the
    other frames skip)."""
    a = mask.sum(axis=1)
    return int(a.argmin())


def run_block_mask(w, dev, Q, K, V, O, plan, core, reps=10):
    """Frame mask x token block mask (the paper's combined mask): attention of a step with a
    synthetic banded block mask (query block qb may attend to key blocks |qb - kb| <= band,
    about a quarter of all blocks) next to the same step unmasked, at the all-active step 0 and
    at the keyframe-only step.  FLOPs count allowed (query row, key) pairs only."""
    import numpy as np
    import torch
    import paper_2606_06309_gb300 as rf
    nb = (w.S_tok + 127) // 128
    band = max(1, nb // 8)
    qb, kb = np.meshgrid(np.arange(nb), np.arange(nb), indexing="ij")
    bm = np.broadcast_to((np.abs(qb - kb) <= band).astype(np.uint8), (w.H, nb, nb)).copy()
    bm_d = torch.from_numpy(bm).to(dev)
    out = {"band_blocks": band, "density": round(float(bm[0].mean()), 4), "steps": {}}
    key_len = np.array([min(128, w.S_tok - 128 * k) for k in range(nb)])
    for s in sorted({0, _keyframe_step(plan.host["mask"])}):
        core.compact(s)
        mask = plan.host["mask"][s]
        rows = np.array([f * w.N + p for f in range(w.F) if mask[f] for p in range(w.N)])
        allowed_keys = (bm[0][rows // 128] * key_len[None, :]).sum()
        flops = 4 * int(allowed_keys) * w.d * w.H
        res = {}
        for label, fn in (
                ("unmasked", lambda: rf.rf_attn(O, None, Q, K, V, Q.stride(0), O.stride(0), w.F,
                                                w.N, w.H, w.d, core.active, core.counts,
                                                w.softmax_scale, core.workspace, core.status)),
                ("block_masked", lambda: rf.rf_attn_block_masked(
                    O, None, Q, K, V, Q.stride(0), O.stride(0), w.F, w.N, w.H, w.d, core.active,
                    core.counts, w.softmax_scale, bm_d, core.workspace, core.status))):
            for _ in range(3):
                fn()
            torch.cuda.synchronize()
            ts = []
            for _ in range(reps):
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record()
                fn()
                b.record()
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(b))
            res[label] = statistics.median(ts)
        out["steps"][str(s)] = {
            "active_frames": int(mask.sum()), "unmasked_ms": round(res["unmasked"], 4),
            "block_masked_ms": round(res["block_masked"], 4),
            "speedup": round(res["unmasked"] / res["block_masked"], 3),
            "ideal_speedup": round(4 * len(rows) * w.S_tok * w.d * w.H / flops, 3),
            "masked_tflops": round(flops / (res["block_masked"] * 1e-3) / 1e12, 1)}
    return out


def run_sweep(w, dev, Q, K, V, O, vel, steps):
    """Step core with a fixed active-frame mask for each active fraction of the workload
    (frames {floor(i*F/A)}), against the all-frames-active step."""
    import numpy as np
    import torch
    import workloads as wl
    from paper_2606_06309_gb300.stepcore import Plan, StepCore
    E = w.N * w.C
    out = {"fractions": [], "active_frames": [], "step_core_ms": [], "attn_tflops": []}
    for frac, mask in zip(w.sweep, wl.sweep_masks(w.F, w.sweep)):
        m = np.tile(np.asarray(mask, np.uint8), (w.S, 1))
        alpha = np.where(m == 1, 1.0, 0.5).astype(np.float32)
        host = {"mask": m, "alpha": alpha, "beta": (1 - alpha).astype(np.float32),
                "dt": np.where(m == 1, -1.0 / w.S, 0.0).astype(np.float32),
                "cur_slot": np.zeros_like(m)}
        t = {k: torch.from_numpy(v).to(dev) for k, v in host.items()}
        plan = Plan(t["mask"], t["alpha"], t["beta"], t["dt"], t["cur_slot"], host)
        core = StepCore(w.F, w.N, E, w.H, w.d, plan, dev)
        core.set_kv_cache(K, V)
        for k in range(3):
            core.run(k % w.S, vel[k % w.S], O, Q, K, V, w.softmax_scale)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        for k in range(steps):
            core.run(k % w.S, vel[k % w.S], O, Q, K, V, w.softmax_scale)
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        A = int(sum(mask))
        out["fractions"].append(frac)
        out["active_frames"].append(A)
        out["step_core_ms"].append(round(ms, 4))
        out["attn_tflops"].append(round(4 * A * w.N * w.S_tok * w.d * w.H / (ms * 1e-3) / 1e12, 1))
        assert core.status.item() == 0
    dense = out["step_core_ms"][out["fractions"].index(1.0)] if 1.0 in out["fractions"] else None
    if dense:
        out["speedup_vs_all_active"] = [round(dense / x, 3) for x in out["step_core_ms"]]
        out["ideal_speedup"] = [round(w.F / A, 3) for A in out["active_frames"]]
    return out


# ---------------------------------------------------------------------------
# CPU oracle (baseline leg and the reference arm)
# ---------------------------------------------------------------------------
def _cpu_model():
    """The host CPU as /proc/cpuinfo names it (on aarch64: implementer and part codes)."""
    info = {}
    try:
        for line in open("/proc/cpuinfo", encoding="utf-8"):
            k, _, v = line.partition(":")
            k = k.strip().lower()
            if k in ("model name", "cpu implementer", "cpu part") and k not in info:
                info[k] = v.strip()
    except OSError:
        pass
    import platform
    if "model name" in info:
        return info["model name"]
    parts = [f"{k} {info[k]}" for k in ("cpu implementer", "cpu part") if k in info]
    return platform.machine() + (" (" + ", ".join(parts) + ")" if parts else "")


class _OracleSample:
    """One step of the fp64 oracle on a bounded sample, inputs prepared once: the schedule,
    projection and Euler update for every frame at latent width, and attention for sampled
    active query rows of sampled heads (all keys)."""

    def __init__(self, w, s=0):
        import numpy as np
        import oracle
        import workloads as wl
        self.w, self.s = w, s
        # the same seeded inputs, widened to fp64 once: the oracle takes fp64 arrays as they are
        self.Q, self.K, self.V = (oracle.to_f64(x) for x in wl.qkv(w))
        self.plan = oracle.schedule(w.F, w.S, w.is_key, w.stride, w.T_w)
        mask = self.plan["mask"][s]
        self.rows_all = np.array([f * w.N + p for f in range(w.F) if mask[f]
                                  for p in range(w.N)])
        self.z = wl.latents(w).double().numpy()
        self.v = wl.velocity(w, s).double().numpy()
        self.rng = np.random.default_rng(0)

    def run(self, n_rows, n_heads=None):
        """(algorithmic attention FLOPs, seconds) of one sample step with n_rows query rows of
        n_heads heads (all heads if None)."""
        import oracle
        w, s = self.w, self.s
        n = int(min(max(1, n_rows), len(self.rows_all)))
        nh = w.H if n_heads is None else int(min(max(1, n_heads), w.H))
        rows = self.rng.choice(self.rows_all, size=n, replace=False)
        heads = None if nh == w.H else sorted(self.rng.choice(w.H, size=nh, replace=False))
        t0 = time.perf_counter()
        oracle.compact(self.plan["mask"][s], w.N)
        oracle.project(self.z, self.z, self.plan["alpha"][s])
        oracle.euler(self.z, self.v, self.plan["dt"][s])
        oracle.attention(self.Q, self.K, self.V, rows, w.softmax_scale, heads)
        return oracle.flops_attn(n, w.S_tok, w.d, nh), time.perf_counter() - t0

    def describe(self, flops, n_heads=None):
        w = self.w
        hs = f"{w.H} heads" if n_heads in (None, w.H) else f"{n_heads} sampled heads of {w.H}"
        return (f"step {self.s} of {w.name}: full schedule/projection/Euler at latent width plus "
                f"attention of sampled active rows x {hs} x {w.S_tok} keys (fp64 numpy, inputs "
                f"widened once; {flops / 1e12:.4f} TFLOP)")


def cpu_baseline(w, budget_s=15.0):
    """The fp64 oracle as it stands, timed on the host cores: sample steps with a doubling
    number of attention rows until the budget is spent.  Throughput is the samples'
    algorithmic attention FLOPs per second."""
    smp = _OracleSample(w)
    n, flops, elapsed = 64, 0, 0.0
    while True:
        f, t = smp.run(n)
        flops += f
        elapsed += t
        if elapsed >= budget_s or n >= len(smp.rows_all):
            break
        n *= 2
    return {"value": round(flops / elapsed / 1e12, 6), "unit": UNIT, "cores": os.cpu_count(),
            "cpu": _cpu_model(), "kind": "oracle", "seconds": round(elapsed, 2),
            "sample": smp.describe(flops)}


def run_reference(args):
    """The reference arm: the oracle as it stands on the host cores.  Every step (warm-up
    included) is one sample step of the same workload; the numbers of sampled heads and
    attention rows are set once, from a calibration sample (64 rows of one head), so that the
    whole run takes about two minutes whatever --steps and --warmup are."""
    rank, world, _ = _env_rank()
    if rank != 0:
        return
    import workloads as wl
    w = wl.get(args.config)
    smp = _OracleSample(w)
    f0, t1 = smp.run(64, 1)                            # calibration (not counted)
    per_step = min(20.0, 120.0 / max(1, args.steps + args.warmup))
    n_heads = max(1, min(w.H, int(per_step / max(t1, 1e-6))))
    n_rows = max(1, min(len(smp.rows_all), int(64 * per_step / max(n_heads * t1, 1e-6))))
    flops, secs = 0, 0.0
    for k in range(args.warmup + args.steps):
        f, t = smp.run(n_rows, n_heads)
        if k >= args.warmup:
            flops += f
            secs += t
    value = round(flops / secs / 1e12, 6)
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(1000 * secs / max(1, args.steps), 3), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": _workload_name(w)},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(),
                            "cpu": _cpu_model(), "kind": "oracle",
                            "sample": f"{n_rows} attention rows per step; "
                                      + smp.describe(flops, n_heads)},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def _workload_name(w):
    return (f"{w.name}: {w.F} latent frames x {w.N} tokens, {w.H} heads x {w.d}, latent {w.C} "
            f"ch, {w.S} flow-matching steps")


def run_attn_shape(args):
    """rf_attn alone at a given shape F,N,H,d with every frame active, random bf16 inputs
    resident on the device and the split-KV workspace: the median launch time and TFLOP/s
    (4 * F*N * F*N * d * H per launch).  A small fixed command for shapes outside the
    workloads and for profiling one kernel."""
    import torch
    import paper_2606_06309_gb300 as rf
    F, N, H, d = (int(x) for x in args.attn_shape.split(","))
    rf.load()
    dev = torch.device("cuda", 0)
    S_tok = F * N
    g = torch.Generator(device=dev).manual_seed(0)
    Q, K, V = (torch.randn(S_tok, H, d, generator=g, device=dev).to(torch.bfloat16)
               for _ in range(3))
    O = torch.empty_like(Q)
    ws = torch.zeros((rf.rf_attn_workspace_bytes(d) + 3) // 4, dtype=torch.int32, device=dev)
    act = torch.zeros(F, dtype=torch.int32, device=dev)
    skp = torch.zeros_like(act)
    cnt = torch.zeros(2, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rf.rf_schedule_compact(torch.ones(F, dtype=torch.uint8, device=dev), F, N, act, skp, None,
                           cnt)
    scale = 1.0 / math.sqrt(d)
    times = []
    for _ in range(args.launches):
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        rf.rf_attn(O, None, Q, K, V, Q.stride(0), O.stride(0), F, N, H, d, act, cnt, scale, ws,
                   status)
        t1.record()
        torch.cuda.synchronize()
        times.append(t0.elapsed_time(t1))
    ms = statistics.median(times[min(2, len(times) - 1):])
    flops = 4 * S_tok * S_tok * d * H
    st = int(status.item())
    print(json.dumps({"attn_shape": {"F": F, "N": N, "H": H, "d": d}, "launches": args.launches,
                      "median_ms": round(ms, 5), "tflops": round(flops / ms / 1e9, 1),
                      "device_status": st}), flush=True)
    if st != 0:
        raise SystemExit(1)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default: two whole trajectories of the workload)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="long",
                    help="workload: tiny, small, mid, large or long (the largest, the default)")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-bandwidth", action="store_true")
    ap.add_argument("--bandwidth-only", action="store_true",
                    help="only the bandwidth-kernel leg (for profiling); prints its JSON")
    ap.add_argument("--attn-shape", default=None, metavar="F,N,H,D",
                    help="only rf_attn at this shape, every frame active (for profiling)")
    ap.add_argument("--launches", type=int, default=10, help="launches for --attn-shape")
    args = ap.parse_args()
    if args.steps is None:
        import workloads as wl
        args.steps = 2 * wl.get(args.config).S
    if args.warmup < 3 and args.impl != "reference":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    elif args.attn_shape:
        run_attn_shape(args)
    elif args.bandwidth_only:
        import torch
        import workloads as wl
        import paper_2606_06309_gb300 as rf
        rf.load()
        peaks, _ = _peaks()
        print(json.dumps(run_bandwidth(wl.get(args.config), torch.device("cuda", 0), peaks)))
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
