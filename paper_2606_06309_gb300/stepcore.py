"""Device state and the four-call sequence of one asynchronous denoising step.

One step s of Algorithm 2 on the device, all on one CUDA stream, no host
synchronisation:

  1. rf_schedule_compact(mask[s])  -> active / skipped frame lists, token list, counts
  2. rf_project(...)               -> full-sequence context at sigma_s (Eq. 3)
  3. rf_attn(...)                  -> active queries x all keys (Q/K/V supplied by the
                                      caller; the DiT projections that would produce them
                                      from the context are outside this library)
  4. rf_step(...)                  -> Euler update of the active frames (two-slot store)

The plan (masks, Eq. 3 weights, step sizes, slot bits) comes from the host
planner rf_plan_build and is uploaded once.  PyTorch only allocates memory.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

from . import (rf_attn, rf_attn_workspace_bytes, rf_plan_build, rf_project, rf_schedule_compact,
               rf_step)


@dataclass
class Plan:
    mask: torch.Tensor      # [S, F] uint8
    alpha: torch.Tensor     # [S, F] fp32
    beta: torch.Tensor      # [S, F] fp32
    dt: torch.Tensor        # [S, F] fp32
    cur_slot: torch.Tensor  # [S, F] uint8
    host: dict


def upload_plan(F, S, is_key, stride, T_w, device, sigma=None) -> Plan:
    h = rf_plan_build(F, S, is_key, stride, T_w, sigma)
    t = {k: torch.from_numpy(v).to(device) for k, v in h.items()}
    return Plan(t["mask"], t["alpha"], t["beta"], t["dt"], t["cur_slot"], h)


class StepCore:
    """Buffers for F frames of N tokens, E latent elements per frame, H heads of dim d."""

    def __init__(self, F: int, N: int, E: int, H: int, d: int, plan: Plan, device="cuda",
                 token_list: bool = True, split_kv: bool = True):
        self.F, self.N, self.E, self.H, self.d = F, N, E, H, d
        self.plan = plan
        dev = torch.device(device)
        self.active = torch.zeros(F, dtype=torch.int32, device=dev)
        self.skipped = torch.zeros(F, dtype=torch.int32, device=dev)
        self.token_idx = torch.zeros(F * N, dtype=torch.int32, device=dev) if token_list else None
        self.counts = torch.zeros(2, dtype=torch.int32, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.z2 = torch.zeros(2, F, E, dtype=torch.float32, device=dev)
        self.ctx = torch.zeros(F, E, dtype=torch.float32, device=dev)
        # split-KV workspace for rf_attn: zero-filled once, left zeroed by every call
        self.workspace = None
        if split_kv:
            nbytes = rf_attn_workspace_bytes(d)
            self.workspace = torch.zeros((nbytes + 3) // 4, dtype=torch.int32, device=dev)

    def set_state(self, z0: torch.Tensor):
        self.z2[0].copy_(z0)
        self.z2[1].copy_(z0)

    def current(self, s: int) -> torch.Tensor:
        """State of every frame when step s begins (s = S: the final state)."""
        S = self.plan.mask.shape[0]
        if s < S:
            slot = self.plan.cur_slot[s].long()
        else:  # after the last step: flip the slots of the frames active at S-1
            slot = (self.plan.cur_slot[S - 1] ^ self.plan.mask[S - 1]).long()
        idx = torch.arange(self.F, device=slot.device)
        return self.z2[slot, idx]

    def compact(self, s: int, stream=None):
        rf_schedule_compact(self.plan.mask[s], self.F, self.N, self.active, self.skipped,
                            self.token_idx, self.counts, stream)

    def project(self, s: int, stream=None):
        rf_project(self.ctx, self.z2, self.plan.cur_slot[s], self.plan.alpha[s],
                   self.plan.beta[s], self.F, self.E, stream)

    def attn(self, O, Q, K, V, scale: float, lse: Optional[torch.Tensor] = None, stream=None):
        rf_attn(O, lse, Q, K, V, Q.stride(0), O.stride(0), self.F, self.N, self.H, self.d,
                self.active, self.counts, scale, self.workspace, self.status, stream)

    def step(self, s: int, v: torch.Tensor, stream=None):
        rf_step(self.z2, self.plan.cur_slot[s], v, self.plan.dt[s], self.active, self.counts,
                self.F, self.E, stream)

    def run(self, s: int, v, O, Q, K, V, scale: float, lse=None, stream=None):
        self.compact(s, stream)
        self.project(s, stream)
        self.attn(O, Q, K, V, scale, lse, stream)
        self.step(s, v, stream)

    def capture_trajectory(self, vels, O, Q, K, V, scale: float, steps=None):
        """Record steps 0..S-1 (4 launches each) into one CUDA graph and return it.

        Nothing in the step core synchronises the host (counts stay on the device), so the
        whole trajectory replays with one launch.  Every call is made once eagerly first, so
        one-time host set-up (kernel attributes, entry points) happens outside the capture.
        Replaying advances the latent store exactly as the eager steps would.
        """
        S = self.plan.mask.shape[0] if steps is None else steps
        self.run(0, vels[0], O, Q, K, V, scale)  # warm-up outside the capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for s in range(S):
                self.run(s, vels[s], O, Q, K, V, scale)
        return g


class HostPipeline:
    """Step-core steps fed from pinned host memory, with the copies hidden behind compute.

    Each step copies host -> device what the step reads: the query rows of the frames active
    at that step (the attention reads no other query row), all of K and V (every query attends
    to every key), and the velocity.  It copies device -> host what the step writes: the
    active frames' rows of the attention output (no other row is written) and a snapshot of
    the two-slot latent store.  Rows of consecutive active frames move in one copy each.
    `depth` device buffer sets and two copy streams (one per direction, so both copy engines
    work) let the input copies of the next depth-1 steps and the read-back of earlier steps
    run during the compute of step k.  Events order the three streams; nothing synchronises
    the host.  Three sets, not two: steps differ in cost (all frames active, then only the
    keyframes), and with two sets the inputs of a heavy step could only be copied during the
    short light step before it (0.84 ms of copies against 0.5 ms of compute on 13 x 1560
    tokens).
    """

    def __init__(self, core: StepCore, S_tok: int, device="cuda", depth: int = 3):
        dev = torch.device(device)
        self.core = core
        self.N = S_tok // core.F
        self.depth = depth
        self.compute = torch.cuda.current_stream(dev)
        self.h2d = torch.cuda.Stream(dev)
        self.d2h = torch.cuda.Stream(dev)
        H, d, F, E = core.H, core.d, core.F, core.E
        self.buf = []
        for _ in range(depth):
            self.buf.append({
                "Q": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "K": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "V": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "v": torch.empty(F, E, dtype=torch.float32, device=dev),
                "O": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "z": torch.empty(2, F, E, dtype=torch.float32, device=dev),
            })
        ev = lambda: [torch.cuda.Event() for _ in range(depth)]
        self.loaded = ev()     # inputs of buffer b are on the device
        self.consumed = ev()   # compute finished with buffer b (inputs read, outputs ready)
        self.drained = ev()    # outputs of buffer b are back on the host
        self.k = 0
        self.moved = []                # (host->device, device->host) bytes of each step

    def active_runs(self, s: int):
        """[f0, f1) ranges of consecutive frames active at schedule step s."""
        m = self.core.plan.host["mask"][s]
        runs, f, F = [], 0, len(m)
        while f < F:
            if m[f]:
                g = f
                while g < F and m[g]:
                    g += 1
                runs.append((f, g))
                f = g
            else:
                f += 1
        return runs

    def step(self, s: int, hQ, hK, hV, hv, hO, hz, scale: float):
        """Enqueue schedule step s: inputs from pinned host tensors hQ, hK, hV (bf16
        [S_tok, H, d]) and hv (fp32 [F, E]); results into pinned hO (bf16; the active frames'
        rows) and hz (fp32 [2, F, E]).  Returns immediately."""
        b = self.k % self.depth
        B = self.buf[b]
        N = self.N
        rows = [(f0 * N, f1 * N) for f0, f1 in self.active_runs(s)]
        first_use = self.k < self.depth
        with torch.cuda.stream(self.h2d):
            if not first_use:
                self.h2d.wait_event(self.consumed[b])   # step k-depth has read these inputs
            for r0, r1 in rows:
                B["Q"][r0:r1].copy_(hQ[r0:r1], non_blocking=True)
            B["K"].copy_(hK, non_blocking=True)
            B["V"].copy_(hV, non_blocking=True)
            B["v"].copy_(hv, non_blocking=True)
            self.loaded[b].record(self.h2d)
        self.compute.wait_event(self.loaded[b])
        if not first_use:
            self.compute.wait_event(self.drained[b])    # step k-depth's outputs are on the host
        self.core.run(s, B["v"], B["O"], B["Q"], B["K"], B["V"], scale, stream=self.compute)
        B["z"].copy_(self.core.z2, non_blocking=True)
        self.consumed[b].record(self.compute)
        with torch.cuda.stream(self.d2h):
            self.d2h.wait_event(self.consumed[b])
            for r0, r1 in rows:
                hO[r0:r1].copy_(B["O"][r0:r1], non_blocking=True)
            hz.copy_(B["z"], non_blocking=True)
            self.drained[b].record(self.d2h)
        self.k += 1
        nbytes = lambda t: t.numel() * t.element_size()
        row_q = nbytes(B["Q"][0])
        act = sum(r1 - r0 for r0, r1 in rows)
        self.moved.append((act * row_q + nbytes(B["K"]) + nbytes(B["V"]) + nbytes(B["v"]),
                           act * row_q + nbytes(B["z"])))

    def bytes_per_step(self, last: Optional[int] = None):
        """Average (host->device, device->host) bytes of the last `last` steps (all steps if
        None)."""
        moved = self.moved if last is None else self.moved[-last:]
        n = max(1, len(moved))
        return (int(round(sum(m[0] for m in moved) / n)), int(round(sum(m[1] for m in moved) / n)))
