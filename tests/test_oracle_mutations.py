"""The oracle's pins catch plausible mistakes (CPU only).

Each mutant below is the oracle with one plausible mistake planted: a dropped term, a wrong
sign or index, a transposed or swapped operand.  With the mutant patched in, at least one
pin of tests/test_oracle_pins.py must fail; the real oracle passes them all.
"""

import numpy as np
import pytest

import oracle
import oracle.rf_oracle as ro
import test_oracle_pins as pins

# pin calls (parametrized pins with one representative argument set)
PIN_CALLS = [
    (pins.test_tiny_active_pattern, {}),
    (pins.test_tiny_worked_example_alpha_dt, {}),
    (pins.test_every_trajectory_reaches_zero, {"name": "mid"}),
    (pins.test_warmup_all_active, {}),
    (pins.test_matches_algorithm2_rule_constant_stride, {"n": 3, "T_w": 8, "T": 50}),
    (pins.test_eq2_two_level_stride_paper_defaults, {}),
    (pins.test_attention_flop_count_matches_printed_example, {}),
    (pins.test_flop_example_step_counts, {}),
    (pins.test_skip_count_identity, {"n": 3}),
    (pins.test_last_jump_clamped_to_sigma_zero, {}),
    (pins.test_compact_brute_force, {"seed": 1}),
    (pins.test_compact_edges, {}),
    (pins.test_projection_endpoints_exact, {}),
    (pins.test_projection_straight_line_exact, {}),
    (pins.test_projection_weight_limits, {}),
    (pins.test_sampler_constant_velocity, {}),
    (pins.test_euler_identity_and_linear, {}),
    (pins.test_attention_brute_force_tiny, {}),
    (pins.test_attention_all_active_equals_sdpa, {}),
    (pins.test_attention_rows_sum_to_one, {}),
    (pins.test_attention_equal_keys_gives_mean, {}),
    (pins.test_attention_planted_key, {}),
    (pins.test_keyframes_identical_frames, {}),
    (pins.test_keyframes_budget_and_orthogonal, {}),
    (pins.test_keyframes_dynamic_threshold_hand_worked, {}),
    (pins.test_keyframes_threshold_direction, {}),
    (pins.test_kv_cache_endpoints_and_store, {}),
    (pins.test_kv_cache_commutes_with_affine_map, {}),
    (pins.test_block_masked_attention_matches_sdpa_with_mask, {}),
    (pins.test_block_masked_attention_all_allowed_is_dense_and_empty_rows_zero, {}),
]


# the unmutated functions, captured before any test patches the module
ORIG = {name: getattr(ro, name) for name in
        ("project", "euler", "attention", "schedule", "compact", "keyframe_select",
         "project_kv_cache", "attention_block_masked")}


def _failures():
    """Number of pins whose assertions fail.  Any other exception is an error of this test:
    a pin must catch the mistake by checking a value, not by crashing."""
    n = 0
    for fn, kw in PIN_CALLS:
        try:
            fn(**kw)
        except AssertionError:
            n += 1
    return n


def test_real_oracle_passes_every_pin():
    assert _failures() == 0


# ---- mutants: each replaces one oracle function with a copy holding one mistake ----------
def _project_swapped(z_start, z_end, alpha):
    a = np.asarray(alpha, dtype=np.float64)[:, None]
    return a * ro.to_f64(z_start) + (1.0 - a) * ro.to_f64(z_end)     # weights swapped


def _project_dropped(z_start, z_end, alpha):
    a = np.asarray(alpha, dtype=np.float64)[:, None]
    return ro.to_f64(z_start) + a * ro.to_f64(z_end)                  # (1 - alpha) dropped


def _euler_sign(z, v, dt):
    return ro.to_f64(z) - np.asarray(dt, dtype=np.float64)[:, None] * ro.to_f64(v)


def _attention_kv_swapped(Q, K, V, rows, scale, heads=None, chunk=256):
    return ORIG['attention'](Q, V, K, rows, scale, heads, chunk)   # K and V swapped


def _attention_no_scale(Q, K, V, rows, scale, heads=None, chunk=256):
    return ORIG['attention'](Q, K, V, rows, 1.0, heads, chunk)     # scale ignored


def _attention_lse_no_log(Q, K, V, rows, scale, heads=None, chunk=256):
    O, L = ORIG['attention'](Q, K, V, rows, scale, heads, chunk)
    Kf, Qf = ro.to_f64(K), ro.to_f64(Q)
    rows = np.asarray(rows)
    hs = list(range(Kf.shape[1])) if heads is None else list(heads)
    for hi, h in enumerate(hs):
        s = scale * (Qf[rows, h, :] @ Kf[:, h, :].T)
        L[hi] = s.max(axis=1)                                          # LSE without + ln l
    return O, L


def _attention_transposed_rows(Q, K, V, rows, scale, heads=None, chunk=256):
    O, L = ORIG['attention'](Q, K, V, rows, scale, heads, chunk)
    return O[::-1].copy(), L[:, ::-1].copy()                          # rows out of order


def _schedule_dt_sign(*a, **k):
    p = ORIG['schedule'](*a, **k)
    p["dt"] = -p["dt"]
    return p


def _schedule_due_off_by_one(F, S, is_key, stride, T_w, sigma=None):
    return ORIG['schedule'](F, S, is_key, [n + 1 for n in stride], T_w, sigma)


def _schedule_alpha_flipped(*a, **k):
    p = ORIG['schedule'](*a, **k)
    sk = p["mask"] == 0
    p["alpha"][sk] = 1.0 - p["alpha"][sk]
    p["beta"][sk] = 1.0 - p["beta"][sk]
    return p


def _compact_token_shift(mask, N):
    a, s, t, c = ORIG['compact'](mask, N)
    return a, s, t + 1, c                                              # f*N + p + 1


def _keyframe_direction(proxies, M, tau, dtau, delta_up, delta_down):
    return ORIG['keyframe_select'](proxies, M, tau, -dtau, delta_up, delta_down)


def _kv_slots_swapped(KV, cache, cur_slot, alpha, mask):
    return ORIG['project_kv_cache'](KV, cache, 1 - np.asarray(cur_slot), alpha, mask)


def _block_mask_transposed(Q, K, V, rows, scale, block_mask, block=128, heads=None):
    bm = np.swapaxes(np.asarray(block_mask), 1, 2)                   # [h][kb][qb]
    return ORIG['attention_block_masked'](Q, K, V, rows, scale, bm, block, heads)


MUTANTS = {
    "project: weights swapped": ("project", _project_swapped),
    "project: (1 - alpha) dropped": ("project", _project_dropped),
    "euler: sign of the step": ("euler", _euler_sign),
    "attention: K and V swapped": ("attention", _attention_kv_swapped),
    "attention: softmax scale ignored": ("attention", _attention_no_scale),
    "attention: LSE without ln l": ("attention", _attention_lse_no_log),
    "attention: rows out of order": ("attention", _attention_transposed_rows),
    "schedule: sign of dt": ("schedule", _schedule_dt_sign),
    "schedule: stride off by one": ("schedule", _schedule_due_off_by_one),
    "schedule: alpha and 1 - alpha exchanged": ("schedule", _schedule_alpha_flipped),
    "compact: token index off by one": ("compact", _compact_token_shift),
    "keyframe_select: threshold step direction": ("keyframe_select", _keyframe_direction),
    "project_kv_cache: slots exchanged": ("project_kv_cache", _kv_slots_swapped),
    "attention_block_masked: mask transposed": ("attention_block_masked", _block_mask_transposed),
}


@pytest.mark.parametrize("label", list(MUTANTS))
def test_mutant_fails_some_pin(monkeypatch, label):
    name, fn = MUTANTS[label]
    monkeypatch.setattr(ro, name, fn)        # functions that call it inside the module
    monkeypatch.setattr(oracle, name, fn)    # the package name the pins use
    assert _failures() >= 1, f"no pin caught: {label}"
