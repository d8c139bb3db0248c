"""Tolerances for comparing the bf16 attention kernel with the fp64 oracle.

Max-abs 2e-2 and mean-abs 2e-3 are the stated bounds for bf16 attention
outputs.  They are loose next to |O| ~ 0.01-0.1 for N(0,1) data, so three
tighter checks are added: relative Frobenius error <= 1e-2, |delta LSE| <= 1e-3,
and (in the planted-key tests) O(1)-scale outputs.  The arithmetic that sets
them: the kernel rounds O to bf16 (relative 2^-9 ~ 2e-3), rounds the
probabilities to bf16 before the PV product (relative 2^-9 per term, averaging
down over thousands of keys, but not on rows dominated by a few keys),
accumulates in fp32 and evaluates exp2 with the hardware approximation
(relative ~2^-22).

The max-abs bound is 2e-2 plus the rounding of the stored output itself:
|g - o| <= 2e-2 + ulp_bf16(|o|) / 2 where |o| >= 1, and exactly 2e-2 below 1.
bf16 keeps 8 significant bits, so the nearest bf16 value to an output in
[2^e, 2^(e+1)) can be 2^(e-8) away from it: 0.0078 in [2, 4), 0.0156 in [4, 8).
Outputs of that size occur where a few large keys dominate a row (the tokens
with std 2 of the 21 x 3600-token workload).  Nothing else is scaled with |o|.
"""
import numpy as np

MAX_ABS = 2e-2
MEAN_ABS = 2e-3
REL_FRO = 1e-2
LSE_ABS = 1e-3


def half_ulp_bf16(x):
    """Half the spacing of bf16 values at |x| (8 significant bits): 2^(floor(log2|x|) - 8)."""
    a = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.maximum(a, np.finfo(np.float64).tiny)))
    return np.exp2(e - 8.0)


def max_abs_bound(o_ref):
    """Per-element max-abs bound: 2e-2, plus half a bf16 ulp of |o| where |o| >= 1."""
    r = np.abs(np.asarray(o_ref, dtype=np.float64))
    return MAX_ABS + np.where(r >= 1.0, half_ulp_bf16(r), 0.0)


def compare(o_gpu, o_ref, lse_gpu=None, lse_ref=None, label=""):
    g = np.asarray(o_gpu, dtype=np.float64)
    r = np.asarray(o_ref, dtype=np.float64)
    assert g.shape == r.shape, (g.shape, r.shape)
    assert np.isfinite(g).all(), f"{label}: non-finite output"
    err = np.abs(g - r)
    rel = np.linalg.norm(g - r) / max(np.linalg.norm(r), 1e-30)
    ratio = err / max_abs_bound(r)
    i = np.unravel_index(np.argmax(ratio), ratio.shape)
    msg = (f"{label}: max-abs {err.max():.3e} (absolute bound {MAX_ABS:g}), worst against the "
           f"per-element bound {ratio[i]:.2f} (gpu {g[i]:.5f}, oracle {r[i]:.5f}) "
           f"mean {err.mean():.3e} relF {rel:.3e}")
    assert ratio.max() <= 1.0, msg
    assert err.mean() <= MEAN_ABS, msg
    assert rel <= REL_FRO, msg
    out = {"max": float(err.max()), "worst_ratio": float(ratio.max()),
           "mean": float(err.mean()), "rel": float(rel)}
    if lse_gpu is not None:
        dl = np.abs(np.asarray(lse_gpu, np.float64) - np.asarray(lse_ref, np.float64)).max()
        assert dl <= LSE_ABS, f"{label}: lse {dl:.3e}"
        out["lse"] = float(dl)
    print(msg)
    return out
