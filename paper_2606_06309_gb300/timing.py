"""Time rf_attn on random bf16 inputs of a given shape (all frames active).

    python -m paper_2606_06309_gb300.timing --F 13 --N 1560 --H 24 --d 64 --launches 5

Prints the median launch time and the attention TFLOP/s (4 * F*N * F*N * d * H FLOPs per
launch).  Inputs stay resident on the device; the split-KV workspace is used.  Useful for
shapes outside the benchmark's workloads and as a small, fixed command to profile.
"""
import argparse
import math
import statistics

import torch

from . import load, rf_attn, rf_attn_workspace_bytes, rf_schedule_compact


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--F", type=int, default=13)
    ap.add_argument("--N", type=int, default=1560)
    ap.add_argument("--H", type=int, default=12)
    ap.add_argument("--d", type=int, default=128, choices=(64, 128))
    ap.add_argument("--launches", type=int, default=10)
    ap.add_argument("--seed", type=int, default=0)
    a = ap.parse_args()
    load()
    dev = torch.device("cuda", 0)
    S_tok = a.F * a.N
    g = torch.Generator(device=dev).manual_seed(a.seed)
    Q, K, V = (torch.randn(S_tok, a.H, a.d, generator=g, device=dev).to(torch.bfloat16)
               for _ in range(3))
    O = torch.empty_like(Q)
    ws = torch.zeros((rf_attn_workspace_bytes(a.d) + 3) // 4, dtype=torch.int32, device=dev)
    act = torch.zeros(a.F, dtype=torch.int32, device=dev)
    skp = torch.zeros_like(act)
    cnt = torch.zeros(2, dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rf_schedule_compact(torch.ones(a.F, dtype=torch.uint8, device=dev), a.F, a.N, act, skp, None,
                        cnt)
    scale = 1.0 / math.sqrt(a.d)
    times = []
    for _ in range(a.launches):
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        rf_attn(O, None, Q, K, V, Q.stride(0), O.stride(0), a.F, a.N, a.H, a.d, act, cnt, scale,
                ws, status)
        t1.record()
        torch.cuda.synchronize()
        times.append(t0.elapsed_time(t1))
    ms = statistics.median(times[min(2, len(times) - 1):])
    flops = 4 * S_tok * S_tok * a.d * a.H
    print(f"F={a.F} N={a.N} H={a.H} d={a.d}: {ms:.4f} ms, {flops / ms / 1e9:.1f} TFLOP/s, "
          f"status {int(status.item())}")
    if int(status.item()) != 0:
        raise SystemExit(1)


if __name__ == "__main__":
    main()
