"""CPU checks of the attention tolerance itself (tests/attn_check.py)."""
import numpy as np
import torch

from attn_check import MAX_ABS, compare, half_ulp_bf16, max_abs_bound


def test_half_ulp_is_the_bf16_rounding_bound():
    """Round-to-nearest bf16 moves x by at most half_ulp_bf16(x), and that bound is reached
    (x halfway between two bf16 neighbours)."""
    rng = np.random.default_rng(0)
    # fp32 inputs: torch rounds float64 to bf16 through fp32, which would round twice
    x = (rng.standard_normal(200_000) * np.exp2(rng.integers(-6, 6, 200_000))).astype(np.float32)
    r = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    x = x.astype(np.float64)
    assert (np.abs(r - x) <= half_ulp_bf16(x) * (1 + 1e-12)).all()
    # 4.234375 lies halfway between the bf16 values 4.21875 and 4.25
    assert half_ulp_bf16(4.234375) == 0.015625
    assert half_ulp_bf16(3.99) == 0.0078125
    assert half_ulp_bf16(1.0) == 2.0 ** -8


def test_bound_is_absolute_below_one():
    o = np.array([0.0, 0.5, 0.999, 1.0, 4.25, -8.5])
    b = max_abs_bound(o)
    assert (b[:3] == MAX_ABS).all()
    np.testing.assert_allclose(b[3:], MAX_ABS + np.array([2 ** -8, 2 ** -6, 2 ** -5]))


def test_compare_rejects_what_the_scaled_bound_let_through():
    """An error of 0.05 at |o| = 3.9 was inside the old 2e-2 * max(1, |o|) = 0.078; the bound
    now allows 0.0278 there."""
    o = np.full((4, 2, 8), 0.01)
    o[0, 0, 0] = 3.9
    g = o.copy()
    g[0, 0, 0] += 0.05
    try:
        compare(g, o, label="planted")
    except AssertionError:
        pass
    else:
        raise AssertionError("a 0.05 error at 3.9 passed")
    g[0, 0, 0] = 3.9 + 0.027
    compare(g, o, label="inside")
