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

    Each step's inputs (Q, K, V and the velocity) are copied host -> device and its results
    (the attention output O and a snapshot of the two-slot latent store) device -> host.  Two
    device buffer sets and two copy streams (one per direction, so both copy engines work)
    overlap the input copy of step k+1 and the read-back of step k-1 with the compute of
    step k.  Events order the three streams; nothing synchronises the host.
    """

    def __init__(self, core: StepCore, S_tok: int, device="cuda"):
        dev = torch.device(device)
        self.core = core
        self.compute = torch.cuda.current_stream(dev)
        self.h2d = torch.cuda.Stream(dev)
        self.d2h = torch.cuda.Stream(dev)
        H, d, F, E = core.H, core.d, core.F, core.E
        self.buf = []
        for _ in range(2):
            self.buf.append({
                "Q": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "K": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "V": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "v": torch.empty(F, E, dtype=torch.float32, device=dev),
                "O": torch.empty(S_tok, H, d, dtype=torch.bfloat16, device=dev),
                "z": torch.empty(2, F, E, dtype=torch.float32, device=dev),
            })
        ev = lambda: torch.cuda.Event()
        self.loaded = [ev(), ev()]     # inputs of buffer b are on the device
        self.consumed = [ev(), ev()]   # compute finished with buffer b (inputs read, outputs ready)
        self.drained = [ev(), ev()]    # outputs of buffer b are back on the host
        self.k = 0

    def step(self, s: int, hQ, hK, hV, hv, hO, hz, scale: float):
        """Enqueue schedule step s: inputs from pinned host tensors hQ, hK, hV (bf16
        [S_tok, H, d]) and hv (fp32 [F, E]); results into pinned hO (bf16) and hz (fp32
        [2, F, E]).  Returns immediately."""
        b = self.k % 2
        B = self.buf[b]
        first_use = self.k < 2
        with torch.cuda.stream(self.h2d):
            if not first_use:
                self.h2d.wait_event(self.consumed[b])   # step k-2 has read these inputs
            B["Q"].copy_(hQ, non_blocking=True)
            B["K"].copy_(hK, non_blocking=True)
            B["V"].copy_(hV, non_blocking=True)
            B["v"].copy_(hv, non_blocking=True)
            self.loaded[b].record(self.h2d)
        self.compute.wait_event(self.loaded[b])
        if not first_use:
            self.compute.wait_event(self.drained[b])    # step k-2's outputs are on the host
        self.core.run(s, B["v"], B["O"], B["Q"], B["K"], B["V"], scale, stream=self.compute)
        B["z"].copy_(self.core.z2, non_blocking=True)
        self.consumed[b].record(self.compute)
        with torch.cuda.stream(self.d2h):
            self.d2h.wait_event(self.consumed[b])
            hO.copy_(B["O"], non_blocking=True)
            hz.copy_(B["z"], non_blocking=True)
            self.drained[b].record(self.d2h)
        self.k += 1

    def bytes_per_step(self):
        B = self.buf[0]
        h2d = sum(B[n].numel() * B[n].element_size() for n in ("Q", "K", "V", "v"))
        d2h = sum(B[n].numel() * B[n].element_size() for n in ("O", "z"))
        return h2d, d2h
