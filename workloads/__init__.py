"""Synthetic workloads and seeded input generators.

This module is shared by the tests, the benchmark and the CPU oracle's callers.
It holds the workload shapes (frames, tokens, heads, head dim, latent channels,
flow-matching steps, keyframe set, per-step skip stride) and seeded random
inputs.  It deliberately contains none of the method's arithmetic: no active-set
rule, no projection weights, no attention and no flow update.

The shapes follow video-DiT latents: F latent frames of N = h*w spatial tokens
each, attention with H heads of head dim d over all F*N tokens, and a latent of
C channels per token.  The paper's own Wan 2.1 workload is 21 latent frames of
3600 tokens, 12 heads of dim 128 and 50 steps (Table "Wan2.1 Model
Configuration", Appendix B.1); its prompts, videos and weights are replaced here
by seeded Gaussian data of the same shapes.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional, Sequence, Tuple

import torch

__all__ = [
    "Workload", "WORKLOADS", "get", "progressive_stride",
    "qkv", "latents", "velocity", "hidden_latents", "sweep_masks",
]


def progressive_stride(S: int, k: int) -> Tuple[int, ...]:
    """Skip stride growing from 1 to k over S steps in k equal segments.

    stride[s] = 1 + floor(k*s/S).  The stride-1 segment plays the role of the
    synchronous warm-up; the last segment uses stride k.
    """
    return tuple(1 + (k * s) // S for s in range(S))


@dataclass(frozen=True)
class Workload:
    name: str
    F: int              # latent frames
    N: int              # tokens per frame
    H: int              # attention heads
    d: int              # head dim
    C: int              # latent channels
    S: int              # flow-matching steps (sigma uniform 1 -> 0)
    keyframes: Tuple[int, ...]
    stride: Tuple[int, ...]   # per-step skip stride for non-keyframes (len S)
    T_w: int            # synchronous warm-up steps
    seed: int
    heavy_frac: float = 0.0   # fraction of tokens drawn with std 2 (shared by Q, K, V)
    sweep: Tuple[float, ...] = field(default=())  # active-frame fractions to sweep

    @property
    def S_tok(self) -> int:
        return self.F * self.N

    @property
    def is_key(self) -> Tuple[int, ...]:
        ks = set(self.keyframes)
        return tuple(1 if f in ks else 0 for f in range(self.F))

    @property
    def softmax_scale(self) -> float:
        return 1.0 / (self.d ** 0.5)


WORKLOADS = {
    # 4 frames x 8x8 tokens, 2 heads x 64; keyframes {0,3}; 4 steps; non-keyframes
    # active on steps {0,2} only (stride 2).
    "tiny": Workload("tiny", F=4, N=64, H=2, d=64, C=16, S=4, keyframes=(0, 3),
                     stride=(2, 2, 2, 2), T_w=0, seed=0),
    # 13 frames x 30x52 tokens, 12 heads x 128; keyframes every 4th frame plus the
    # last; 20 steps; non-keyframes skip every other step.
    "small": Workload("small", F=13, N=1560, H=12, d=128, C=16, S=20,
                      keyframes=(0, 4, 8, 12), stride=(2,) * 20, T_w=0, seed=1),
    # 21 frames x 1560 tokens, 12 heads; keyframes 0,5,10,15,20; 50 steps;
    # progressive stride 1 -> 4.
    "mid": Workload("mid", F=21, N=1560, H=12, d=128, C=16, S=50,
                    keyframes=(0, 5, 10, 15, 20), stride=progressive_stride(50, 4),
                    T_w=0, seed=2),
    # 21 frames x 45x80 tokens, 40 heads; keyframes 0,4,...,20; 50 steps;
    # progressive stride 1 -> 4; 10% of tokens with std 2.
    "large": Workload("large", F=21, N=3600, H=40, d=128, C=16, S=50,
                      keyframes=(0, 4, 8, 12, 16, 20), stride=progressive_stride(50, 4),
                      T_w=0, seed=3, heavy_frac=0.1),
    # 33 frames x 3600 tokens, 24 heads; keyframes every 7th frame plus the last;
    # 50 steps; progressive stride 1 -> 6; active-fraction sweep.
    "long": Workload("long", F=33, N=3600, H=24, d=128, C=16, S=50,
                     keyframes=(0, 7, 14, 21, 28, 32), stride=progressive_stride(50, 6),
                     T_w=0, seed=4, sweep=(0.15, 0.3, 0.6, 1.0)),
}


def get(name: str) -> Workload:
    return WORKLOADS[name]


# ---------------------------------------------------------------------------
# Seeded generators.  Each tensor comes from its own stream: a torch Generator
# seeded with (workload seed, stream id, step).  Device generation is used for
# large shapes; the tests copy the needed slices back to the host.
# ---------------------------------------------------------------------------
_STREAM = {"q": 1, "k": 2, "v": 3, "z": 4, "vel": 5, "heavy": 6, "hid": 7}


def _gen(seed: int, stream: str, step: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + _STREAM[stream] * 10_007 + step) & 0x7FFF_FFFF_FFFF)
    return g


def qkv(w: Workload, device="cpu", row_stride: Optional[int] = None):
    """bf16 Q, K, V of shape [S_tok, H, d] (token-major, heads interleaved).

    Values ~ N(0,1) rounded to bf16 (round to nearest even).  With heavy_frac > 0
    a seeded per-token Bernoulli mask, shared by Q, K and V and all heads, scales
    those tokens by 2 (variance 4).  If row_stride > H*d the tensors are views
    into wider rows ([S_tok, row_stride] storage).
    """
    shape = (w.S_tok, w.H, w.d)
    out = []
    heavy = None
    if w.heavy_frac > 0:
        gh = _gen(w.seed, "heavy", 0, device)
        heavy = torch.rand(w.S_tok, generator=gh, device=device) < w.heavy_frac
    for name in ("q", "k", "v"):
        g = _gen(w.seed, name, 0, device)
        if row_stride is None or row_stride == w.H * w.d:
            x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
            if heavy is not None:
                x[heavy] *= 2.0
            out.append(x.to(torch.bfloat16))
        else:
            base = torch.randn((w.S_tok, row_stride), generator=g, device=device,
                               dtype=torch.float32)
            if heavy is not None:
                base[heavy] *= 2.0
            base = base.to(torch.bfloat16)
            out.append(base[:, : w.H * w.d].view(w.S_tok, w.H, w.d))
    return tuple(out)


def latents(w: Workload, C: Optional[int] = None, device="cpu") -> torch.Tensor:
    """Initial noise latent z_1 ~ N(0,1), fp32 [F, N*C]."""
    C = w.C if C is None else C
    g = _gen(w.seed, "z", 0, device)
    return torch.randn((w.F, w.N * C), generator=g, device=device, dtype=torch.float32)


def velocity(w: Workload, step: int, C: Optional[int] = None, device="cpu") -> torch.Tensor:
    """Synthetic velocity for flow-matching step `step`, fp32 [F, N*C] ~ N(0,1)."""
    C = w.C if C is None else C
    g = _gen(w.seed, "vel", step, device)
    return torch.randn((w.F, w.N * C), generator=g, device=device, dtype=torch.float32)


def hidden_latents(w: Workload, slot: int, device="cpu") -> torch.Tensor:
    """Hidden-width state fp32 [F, N*H*d] for the bandwidth-kernel stress shape."""
    g = _gen(w.seed, "hid", slot, device)
    return torch.randn((w.F, w.N * w.H * w.d), generator=g, device=device, dtype=torch.float32)


def sweep_masks(F: int, fracs: Sequence[float]):
    """Active-frame masks with A = round(frac*F) frames spread evenly:
    active = {floor(i*F/A) : i < A}."""
    masks = []
    for fr in fracs:
        A = max(1, int(round(fr * F)))
        m = [0] * F
        for i in range(A):
            m[(i * F) // A] = 1
        masks.append(tuple(m))
    return masks
