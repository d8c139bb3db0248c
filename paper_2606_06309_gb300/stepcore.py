"""Device state and the five-call sequence of one asynchronous denoising step.

One step s of Algorithm 2 on the device, all on one CUDA stream, no host
synchronisation:

  1. rf_schedule_compact(mask[s])  -> active / skipped frame lists, token list, counts
  2. rf_project(...)               -> full-sequence latent context at sigma_s (Eq. 3)
  3. rf_project_kv(...)            -> keys and values of the skipped frames: Eq. 3 over the
                                      rolling cache of Appendix B.2; the active frames' fresh
                                      rows shifted into the cache
  4. rf_attn(...)                  -> active queries x all keys (the active frames' Q/K/V
                                      rows supplied by the caller; the DiT projections that
                                      would produce them are outside this library)
  5. rf_step(...)                  -> Euler update of the active frames (two-slot store)

The plan (masks, Eq. 3 weights, step sizes, slot bits) comes from the host
planner rf_plan_build and is uploaded once.  PyTorch only allocates memory.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Optional

import torch

from . import (rf_attn, rf_attn_workspace_bytes, rf_pipeline_bytes, rf_pipeline_create,
               rf_pipeline_destroy, rf_pipeline_step, rf_pipeline_sync, rf_plan_build, rf_project,
               rf_project_kv, rf_schedule_compact, rf_step)


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
    """Buffers for F frames of N tokens, E latent elements per frame, H heads of dim d.

    With kv_cache (the default) the step core holds the rolling key/value cache (bf16
    [2, F, N, H*d] each) and run() fills the skipped frames' rows of K and V from it before
    the attention; set_kv_cache() gives the cache its initial contents."""

    def __init__(self, F: int, N: int, E: int, H: int, d: int, plan: Plan, device="cuda",
                 token_list: bool = True, split_kv: bool = True, kv_cache: bool = True):
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
        self.Kc = self.Vc = None
        if kv_cache:
            self.Kc = torch.zeros(2, F, N, H * d, dtype=torch.bfloat16, device=dev)
            self.Vc = torch.zeros_like(self.Kc)
        # split-KV workspace for rf_attn: zero-filled once, left zeroed by every call
        self.workspace = None
        if split_kv:
            nbytes = rf_attn_workspace_bytes(d)
            self.workspace = torch.zeros((nbytes + 3) // 4, dtype=torch.int32, device=dev)

    def set_state(self, z0: torch.Tensor):
        self.z2[0].copy_(z0)
        self.z2[1].copy_(z0)

    def set_kv_cache(self, K0: torch.Tensor, V0: torch.Tensor):
        """Both cache slots of every frame hold the keys and values K0, V0 ([F*N, H, d]): a frame
        projected before its second update gets them back (alpha weights two equal states)."""
        D = self.H * self.d
        for c, X in ((self.Kc, K0), (self.Vc, V0)):
            x = X.reshape(self.F, self.N, D)
            c[0].copy_(x)
            c[1].copy_(x)

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

    def project_kv(self, s: int, K, V, stream=None):
        rf_project_kv(K, V, K.stride(0), self.Kc, self.Vc, self.plan.cur_slot[s],
                      self.plan.alpha[s], self.plan.beta[s], self.active, self.skipped,
                      self.counts, self.F, self.N, self.H * self.d, stream)

    def attn(self, O, Q, K, V, scale: float, lse: Optional[torch.Tensor] = None, stream=None):
        rf_attn(O, lse, Q, K, V, Q.stride(0), O.stride(0), self.F, self.N, self.H, self.d,
                self.active, self.counts, scale, self.workspace, self.status, stream)

    def step(self, s: int, v: torch.Tensor, stream=None):
        rf_step(self.z2, self.plan.cur_slot[s], v, self.plan.dt[s], self.active, self.counts,
                self.F, self.E, stream)

    def run(self, s: int, v, O, Q, K, V, scale: float, lse=None, stream=None):
        """Step s.  Q, K, V hold the active frames' fresh rows; with the cache, the skipped
        frames' rows of K and V are overwritten with their projection before the attention."""
        self.compact(s, stream)
        self.project(s, stream)
        if self.Kc is not None:
            self.project_kv(s, K, V, stream)
        self.attn(O, Q, K, V, scale, lse, stream)
        self.step(s, v, stream)

    @property
    def launches_per_step(self) -> int:
        return 5 if self.Kc is not None else 4

    def capture_trajectory(self, vels, O, Q, K, V, scale: float, steps=None):
        """Record steps 0..S-1 (all launches of each) into one CUDA graph and return it.

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

    A thin wrapper of the library's native pipeline (``rf_pipeline_*``), which owns the plan,
    the two-slot latent store, the rolling key/value cache and `depth` device buffer sets.  Each
    step copies host -> device what it reads: the fresh query, key and value rows of the frames
    active at that step, and the velocity (the skipped frames' keys and values are projected
    from the device-resident cache).  It copies device -> host what it writes: the active
    frames' rows of the attention output, the latent context and a snapshot of the latent
    store.  Three streams (compute, host->device, device->host) are ordered by events, so the
    input copies of the next depth-1 steps and the read-back of earlier steps run during the
    compute of step k; nothing synchronises the host.  Three sets, not two: steps differ in
    cost (all frames active, then only the keyframes), and with two sets the inputs of a heavy
    step could only be copied during the short light step before it.

    The pipeline starts from `core`'s plan and current latent store, and from the initial keys
    and values K0, V0 (host tensors); it does not change `core`.
    """

    def __init__(self, core: StepCore, S_tok: int, K0, V0, device="cuda", depth: int = 3):
        dev = torch.device(device)
        self.core = core
        self.N = S_tok // core.F
        self.depth = depth
        self.compute = torch.cuda.current_stream(dev)
        self.h2d = torch.cuda.Stream(dev)
        self.d2h = torch.cuda.Stream(dev)
        torch.cuda.synchronize(dev)  # the core's latent store is read below
        self.handle = rf_pipeline_create(core.F, self.N, core.H, core.d, core.E, core.plan.host,
                                         core.z2, K0, V0, depth, self.compute, self.h2d,
                                         self.d2h)
        self._marks = []  # (steps, h2d bytes, d2h bytes) after each step

    def step(self, s: int, hQ, hK, hV, hv, hO, hz, scale: float, hctx=None):
        """Enqueue schedule step s: inputs from pinned host tensors hQ, hK, hV (bf16
        [S_tok, H, d], contiguous rows; the active frames' rows are read) and hv (fp32 [F, E]);
        results into pinned hO (bf16; the active frames' rows), hz (fp32 [2, F, E]) and, if
        given, hctx (fp32 [F, E], the Eq. 3 context).  Returns immediately."""
        rf_pipeline_step(self.handle, s, hQ, hK, hV, hv, hO, hz, hctx, scale)
        self._marks.append(rf_pipeline_bytes(self.handle))

    def sync(self) -> int:
        """Wait for every enqueued step; returns the device status word."""
        return rf_pipeline_sync(self.handle)

    def bytes_per_step(self, last: Optional[int] = None):
        """Average (host->device, device->host) bytes of the last `last` steps (all steps if
        None)."""
        if not self._marks:
            return 0, 0
        n = len(self._marks) if last is None else min(last, len(self._marks))
        end = self._marks[-1]
        start = self._marks[-n - 1] if n < len(self._marks) else (0, 0, 0)
        steps = end[0] - start[0]
        return (int(round((end[1] - start[1]) / steps)), int(round((end[2] - start[2]) / steps)))

    def close(self):
        if getattr(self, "handle", None):
            rf_pipeline_destroy(self.handle)
            self.handle = None

    def __del__(self):
        self.close()
