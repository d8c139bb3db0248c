"""Pins of the CPU oracle to things other than itself (CPU only).

Each test checks the oracle against a value the paper prints, a closed form, an
invariant, a library routine, or a brute force on a tiny input.  Together they
are chosen so that a dropped term, a wrong sign, index or slot, or a transposed
operand in the oracle fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# Schedule (Algorithm 2, Eq. 2)
# --------------------------------------------------------------------------
def _plan(w, **kw):
    args = dict(F=w.F, S=w.S, is_key=w.is_key, stride=w.stride, T_w=w.T_w)
    args.update(kw)
    return oracle.schedule(**args)


def test_tiny_active_pattern():
    """The tiny workload: keyframes 0 and 3 on every step, non-keyframes 1 and 2
    active on steps {0, 2} only."""
    p = _plan(wl.get("tiny"))
    m = p["mask"]
    assert m[:, 0].tolist() == [1, 1, 1, 1]
    assert m[:, 3].tolist() == [1, 1, 1, 1]
    assert m[:, 1].tolist() == [1, 0, 1, 0]
    assert m[:, 2].tolist() == [1, 0, 1, 0]


def test_tiny_worked_example_alpha_dt():
    """sigma = 1, .75, .5, .25, 0.  Non-keyframes jump 1 -> .5 at step 0 and
    .5 -> 0 at step 2 (dt = -0.5); at steps 1 and 3 they are projected with
    alpha = (1-.75)/(1-.5) = (.5-.25)/(.5-0) = 0.5 (Eq. 3).  Keyframes dt = -.25."""
    p = _plan(wl.get("tiny"))
    assert p["dt"][:, 0].tolist() == [-0.25] * 4
    assert p["dt"][:, 1].tolist() == [-0.5, 0.0, -0.5, 0.0]
    assert p["alpha"][1, 1] == 0.5 and p["alpha"][3, 2] == 0.5
    assert p["alpha"][1, 0] == 1.0 and p["beta"][1, 0] == 0.0
    # slot bookkeeping: an active frame writes its new state to the other slot
    assert p["cur_slot"][:, 0].tolist() == [0, 1, 0, 1]
    assert p["cur_slot"][:, 1].tolist() == [0, 1, 1, 0]


def test_eq2_two_level_stride_paper_defaults():
    """Eq. 2 with the paper's defaults (T = 50, T_w = 8, T_mid = T/2, n_small = 2,
    n_large = 3), worked by hand with the due-step reading: a non-keyframe is updated on
    every warm-up step 0..7, then every 2 steps while s < T - T_mid = 25 (8, 10, ..., 24;
    the jump from 24 lands on 26), then every 3 steps (26, 29, ..., 47, the last jump clamped
    to sigma = 0).  Its step sizes are the gaps to the next update, in sigma units."""
    T, T_w = 50, 8
    stride = [2] * 25 + [3] * 25
    p = oracle.schedule(F=2, S=T, is_key=[1, 0], stride=stride, T_w=T_w)
    active = [s for s in range(T) if p["mask"][s, 1]]
    assert active == list(range(8)) + list(range(8, 25, 2)) + list(range(26, 48, 3))
    nxt = active[1:] + [T]
    for s, n in zip(active, nxt):
        assert p["dt"][s, 1] == pytest.approx(-(n - s) / T, abs=1e-7)
    assert p["mask"][:, 0].all()                       # the keyframe on every step
    # a skipped step between 26 and 29 projects with alpha = (sigma_26 - sigma_s)/(3/50)
    assert p["alpha"][27, 1] == pytest.approx(1 / 3, abs=1e-7)
    assert p["alpha"][28, 1] == pytest.approx(2 / 3, abs=1e-7)


@pytest.mark.parametrize("name", list(wl.WORKLOADS))
def test_every_trajectory_reaches_zero(name):
    """Each frame's Euler steps sum to sigma_S - sigma_0 = -1, every frame is
    active at step 0, keyframes are active on every step, and alpha is in (0,1)
    for skipped frames."""
    w = wl.get(name)
    p = _plan(w)
    np.testing.assert_allclose(p["dt"].sum(axis=0), -1.0, rtol=0, atol=1e-12)
    assert p["mask"][0].all()
    for f in w.keyframes:
        assert p["mask"][:, f].all()
    sk = p["mask"] == 0
    assert ((p["alpha"][sk] > 0) & (p["alpha"][sk] < 1)).all()
    assert (p["dt"] <= 0).all()


def test_warmup_all_active():
    """Sec. 3.2.1: all frames are updated one step at a time for the first T_w steps."""
    w = wl.get("mid")
    p = _plan(w, T_w=8)
    assert p["mask"][:8].all()
    np.testing.assert_allclose(p["dt"][:8], -1.0 / w.S)


@pytest.mark.parametrize("n,T_w,T", [(2, 10, 50), (3, 8, 50), (2, 8, 20), (4, 0, 30)])
def test_matches_algorithm2_rule_constant_stride(n, T_w, T):
    """Under a constant stride the due-step rule equals Algorithm 2's printed
    active set (t = T - s; non-keyframe active iff (T - T_w - t) = 0 mod n)."""
    is_key = (1, 0, 0, 1, 0, 0, 0, 1)
    p = oracle.schedule(F=len(is_key), S=T, is_key=is_key, stride=[n] * T, T_w=T_w)
    for s in range(T):
        t = T - s
        want = oracle.active_set_alg2(t, T, T_w, is_key, n)
        got = [f for f in range(len(is_key)) if p["mask"][s, f]]
        assert got == want, (s, got, want)


def test_flop_example_step_counts():
    """Appendix B.1 numerical example: T = 50, T_warmup = 10, n = 2 gives 40
    asynchronous steps, 20 skip steps and 20 full denoising steps."""
    g = json.load(open(os.path.join(GOLDEN, "flop_example_wan21.json")))
    F, M = g["F"], g["M"]
    is_key = [1 if f < M else 0 for f in range(F)]
    p = oracle.schedule(F=F, S=g["T"], is_key=is_key, stride=[g["n"]] * g["T"],
                        T_w=g["T_warmup"])
    asyn = p["mask"][g["T_warmup"]:]
    full = int(asyn.all(axis=1).sum())
    skip = int((~asyn.all(axis=1)).sum())
    assert len(asyn) == g["T_RhymeFlow"]
    assert skip == g["N_skip"] and full == g["N_denoise"]
    # skip steps attend with exactly the M keyframes as queries
    assert (asyn[~asyn.all(axis=1)].sum(axis=1) == M).all()


def test_attention_flop_count_matches_printed_example():
    """Appendix B.1 prints the attention FLOPs of one dense Wan 2.1 layer (S = 75,600 tokens,
    D = 1,536 = 12 heads x 128) as 17.56 TFLOPs of 18.27, counting one FLOP per multiply-add.
    The oracle's count (two per multiply-add, the one the benchmark divides by) is exactly twice
    the printed attention term at full size."""
    g = json.load(open(os.path.join(GOLDEN, "attention_flops_wan21.json")))
    S, D = g["S"], g["D"]
    attn_mac = oracle.flops_attn(S, S, g["head_dim"], g["heads"]) // 2   # S^2 D, twice
    assert attn_mac == 2 * S * S * D
    assert round(attn_mac / 1e12, 2) == g["printed_attention_tflops_per_layer"]
    layer = 4 * S * D * D + attn_mac
    assert round(layer / 1e12, 2) == g["printed_layer_tflops"]
    assert round(100 * attn_mac / layer, 1) == g["printed_attention_share_pct"]
    # skip-step layer: the printed projection term is within 0.2% of the formula's 4 S D^2; the
    # printed attention term is exactly 4 S^2 D, twice the formula's 2 S^2 D (inconsistent
    # figures of the paper; the oracle follows the formula)
    Ss = g["S_skip"]
    proj, attn = g["printed_skip_layer_terms"]
    assert abs(proj / (4 * Ss * D * D) - 1) < 2e-3
    assert oracle.flops_attn(Ss, Ss, g["head_dim"], g["heads"]) // 2 == 2 * Ss * Ss * D
    assert attn == 2 * (2 * Ss * Ss * D)


@pytest.mark.parametrize("n", [2, 3, 4, 5])
def test_skip_count_identity(n):
    """Appendix B.1: N_skip = floor(T_R (n-1)/n) with T_R = 40."""
    T, T_w = 50, 10
    is_key = [1, 0, 0]
    p = oracle.schedule(F=3, S=T, is_key=is_key, stride=[n] * T, T_w=T_w)
    skip = int((p["mask"][T_w:, 1] == 0).sum())
    assert skip == math.floor((T - T_w) * (n - 1) / n)


def test_progressive_stride_segments():
    """Eq. 2 generalised: stride grows 1 -> 4 over 50 steps in equal segments."""
    st = wl.progressive_stride(50, 4)
    assert st[:13] == (1,) * 13 and st[13:25] == (2,) * 12
    assert st[25:38] == (3,) * 13 and st[38:] == (4,) * 12


def test_last_jump_clamped_to_sigma_zero():
    p = oracle.schedule(F=2, S=5, is_key=[1, 0], stride=[3] * 5, T_w=0)
    # frame 1: 0 -> 3, then 3 -> min(6, 5) = 5
    assert p["mask"][:, 1].tolist() == [1, 0, 0, 1, 0]
    np.testing.assert_allclose(p["dt"][:, 1], [-0.6, 0, 0, -0.4, 0])


# --------------------------------------------------------------------------
# Compaction
# --------------------------------------------------------------------------
@pytest.mark.parametrize("seed", range(6))
def test_compact_brute_force(seed):
    rng = np.random.default_rng(seed)
    F = int(rng.integers(1, 40))
    N = int(rng.integers(1, 50))
    mask = (rng.random(F) < rng.random()).astype(np.uint8)
    a, s, t, c = oracle.compact(mask, N)
    want_tokens = sorted({f * N + p for f in range(F) for p in range(N) if mask[f]})
    assert t.tolist() == want_tokens
    assert a.tolist() == np.flatnonzero(mask).tolist()
    assert s.tolist() == np.flatnonzero(mask == 0).tolist()
    assert c.tolist() == [int(mask.sum()), int(mask.sum()) * N]


def test_compact_edges():
    a, s, t, c = oracle.compact([0, 0, 0], 5)
    assert len(a) == 0 and s.tolist() == [0, 1, 2] and len(t) == 0 and c.tolist() == [0, 0]
    a, s, t, c = oracle.compact([1, 1], 3)
    assert t.tolist() == list(range(6)) and len(s) == 0


# --------------------------------------------------------------------------
# Projection (Eq. 3)
# --------------------------------------------------------------------------
def test_projection_endpoints_exact():
    rng = np.random.default_rng(1)
    a, b = rng.standard_normal((2, 3, 17))
    np.testing.assert_array_equal(oracle.project(a, b, [0.0] * 3), a)
    np.testing.assert_array_equal(oracle.project(a, b, [1.0] * 3), b)


def test_projection_straight_line_exact():
    """On a straight-line trajectory z(sigma) = a + sigma*b (the rectified-flow
    motivation of Eq. 3) the projection recovers z(sigma_s) exactly."""
    rng = np.random.default_rng(2)
    a, b = rng.standard_normal((2, 1, 64))
    s0, s1 = 0.8, 0.35
    for sig in np.linspace(s0, s1, 7):
        alpha = (s0 - sig) / (s0 - s1)
        got = oracle.project(a + s0 * b, a + s1 * b, [alpha])
        np.testing.assert_allclose(got, a + sig * b, rtol=0, atol=1e-14)


def test_projection_weight_limits():
    """Appendix B.2: alpha -> 0 as the step approaches the earlier cached state,
    alpha -> 1 as it approaches the later one (sigma decreasing)."""
    p = oracle.schedule(F=2, S=20, is_key=[1, 0], stride=[5] * 20, T_w=0)
    al = p["alpha"][1:5, 1]
    assert (np.diff(al) > 0).all() and al[0] == pytest.approx(0.2) and al[-1] == pytest.approx(0.8)


def test_sampler_constant_velocity():
    """Constant velocity v: every frame ends at z1 - v whatever the schedule,
    and every projected context equals the true straight-line state
    z1 + (sigma_s - 1) v."""
    w = wl.get("mid")
    p = _plan(w)
    rng = np.random.default_rng(3)
    z1 = rng.standard_normal((w.F, 8))
    v = rng.standard_normal((w.F, 8))
    zT, ctxs = oracle.sampler(z1, lambda s: v, p)
    np.testing.assert_allclose(zT, z1 - v, rtol=0, atol=1e-12)
    for s, ctx in enumerate(ctxs):
        np.testing.assert_allclose(ctx, z1 + (p["sigma"][s] - 1.0) * v, rtol=0, atol=1e-12)


def test_euler_identity_and_linear():
    rng = np.random.default_rng(4)
    z, v = rng.standard_normal((2, 3, 10))
    np.testing.assert_array_equal(oracle.euler(z, v, [0, 0, 0]), z)
    np.testing.assert_allclose(oracle.euler(z, v, [-0.5, 0.25, 1.0]),
                               z + np.array([-0.5, 0.25, 1.0])[:, None] * v)


# --------------------------------------------------------------------------
# Attention
# --------------------------------------------------------------------------
def _rand_qkv(S_tok, H, d, seed):
    g = torch.Generator().manual_seed(seed)
    return [torch.randn(S_tok, H, d, generator=g).to(torch.bfloat16) for _ in range(3)]


def test_attention_brute_force_tiny():
    """Pure-Python double loops with math.exp on a tiny case."""
    Q, K, V = _rand_qkv(12, 2, 4, 0)
    q, k, v = (oracle.to_f64(x) for x in (Q, K, V))
    scale = 0.37
    rows = [0, 3, 11]
    O, L = oracle.attention(Q, K, V, rows, scale)
    for hi in range(2):
        for ri, i in enumerate(rows):
            s = [scale * sum(q[i, hi, c] * k[j, hi, c] for c in range(4)) for j in range(12)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            tot = sum(e)
            for c in range(4):
                want = sum(e[j] * v[j, hi, c] for j in range(12)) / tot
                assert abs(O[ri, hi, c] - want) < 1e-13
            assert abs(L[hi, ri] - (m + math.log(tot))) < 1e-13


def test_attention_all_active_equals_sdpa():
    """With every frame active the path is dense attention: compare with
    torch's scaled_dot_product_attention in fp64."""
    w = wl.get("tiny")
    Q, K, V = wl.qkv(w)
    O, L = oracle.attention(Q, K, V, range(w.S_tok), w.softmax_scale)
    q, k, v = (x.double().permute(1, 0, 2) for x in (Q, K, V))
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, scale=w.softmax_scale)
    np.testing.assert_allclose(O, ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)
    lse = torch.logsumexp(w.softmax_scale * q @ k.transpose(1, 2), dim=-1)
    np.testing.assert_allclose(L, lse.numpy(), rtol=0, atol=1e-12)


def test_attention_rows_sum_to_one():
    """V = 1 gives O = 1; exp(s - LSE) sums to 1 over the keys."""
    Q, K, _ = _rand_qkv(40, 2, 16, 1)
    V = torch.ones(40, 2, 16)
    O, L = oracle.attention(Q, K, V, range(0, 40, 3), 0.25)
    np.testing.assert_allclose(O, 1.0, rtol=0, atol=1e-14)
    q, k = oracle.to_f64(Q), oracle.to_f64(K)
    s = 0.25 * np.einsum("ic,jc->ij", q[::3, 1], k[:, 1])
    np.testing.assert_allclose(np.exp(s - L[1][:, None]).sum(axis=1), 1.0, rtol=1e-13)


def test_attention_equal_keys_gives_mean():
    Q, _, V = _rand_qkv(30, 1, 8, 2)
    K = torch.randn(1, 1, 8).expand(30, 1, 8)
    O, _ = oracle.attention(Q, K, V, [0, 7, 29], 1.0)
    np.testing.assert_allclose(O, np.broadcast_to(oracle.to_f64(V).mean(axis=0), O.shape),
                               rtol=0, atol=1e-13)


def test_attention_planted_key():
    """q_i = 16 k_{j*}: the output row is v_{j*} to O(1) precision, whatever
    the index of the query and key (pins row/column indexing and K vs V)."""
    g = torch.Generator().manual_seed(5)
    S_tok, d = 256, 64
    K = torch.randn(S_tok, 1, d, generator=g)
    V = torch.randn(S_tok, 1, d, generator=g)
    perm = torch.randperm(S_tok, generator=g)
    Q = 16.0 * K[perm]
    O, _ = oracle.attention(Q, K, V, range(S_tok), 1.0 / math.sqrt(d))
    np.testing.assert_allclose(O[:, 0], V[perm, 0].double().numpy(), rtol=0, atol=1e-6)


# --------------------------------------------------------------------------
# Keyframe selection (Algorithm 1, Eq. 1) -- partly unpinned (no constants given)
# --------------------------------------------------------------------------
def _unit(theta):
    return np.array([math.cos(theta), math.sin(theta)])


def test_keyframes_identical_frames():
    P = np.ones((9, 5))
    assert oracle.keyframe_select(P, M=4, tau=0.9, dtau=0.1, delta_up=1, delta_down=1) == \
        ([0], list(range(1, 9)))


def test_keyframes_budget_and_orthogonal():
    P = np.eye(8)
    k, n = oracle.keyframe_select(P, M=3, tau=0.5, dtau=0.0, delta_up=1, delta_down=1)
    assert k == [0, 1, 2] and n == [3, 4, 5, 6, 7]


def test_keyframes_dynamic_threshold_hand_worked():
    """Unit vectors at the given angles (degrees), so cosine similarity is the
    cosine of the angle between frames.

    Case 1: angles 0,10,60,66,70,130; M = 3 (L_avg = 2); delta_up = delta_down = 1;
    tau0 = cos 45, dtau = 0.2.  Frame 2 (60 deg, gap 2) is a key with tau
    unchanged; frames 3, 4 are within 10 deg of it; frame 5 (70 deg from frame 2,
    gap 3 >= L_avg + 1) is a key and lowers tau.  With tau0 = cos 65 frame 2 is
    rejected and frame 3 (66 deg) is taken instead.
    """
    P = np.stack([_unit(math.radians(a)) for a in (0, 10, 60, 66, 70, 130)])
    k, n = oracle.keyframe_select(P, M=3, tau=math.cos(math.radians(45)), dtau=0.2,
                                  delta_up=1, delta_down=1)
    assert k == [0, 2, 5] and n == [1, 3, 4]
    k, _ = oracle.keyframe_select(P, M=3, tau=math.cos(math.radians(65)), dtau=0.2,
                                  delta_up=1, delta_down=1)
    assert k == [0, 3]


def test_keyframes_threshold_direction():
    """Angles 0,50,100,135; M = 4 (L_avg = 1); delta_down = 0, delta_up = 1;
    tau0 = cos 45.  Algorithm 1 raises tau after a short gap (gap 1 <= L_avg) and
    lowers it after a long one.  dtau = +0.3: frames 1, 2 (50 deg steps) each
    raise tau, so frame 3 (35 deg from frame 2) is also taken.  dtau = -0.3:
    tau drops to cos 45 - 0.3 after frame 1, frame 2 (50 deg) is rejected, and
    frame 3 (85 deg from frame 1, gap 2) is taken."""
    P = np.stack([_unit(math.radians(a)) for a in (0, 50, 100, 135)])
    tau0 = math.cos(math.radians(45))
    k, _ = oracle.keyframe_select(P, M=4, tau=tau0, dtau=0.3, delta_up=1, delta_down=0)
    assert k == [0, 1, 2, 3]
    k, _ = oracle.keyframe_select(P, M=4, tau=tau0, dtau=-0.3, delta_up=1, delta_down=0)
    assert k == [0, 1, 3]


# --------------------------------------------------------------------------
# Rolling key/value cache (Appendix B.2)
# --------------------------------------------------------------------------
def _kv_case(seed, F=5, N=3, D=8):
    rng = np.random.default_rng(seed)
    kv = rng.standard_normal((F, N, D))
    cache = rng.standard_normal((2, F, N, D))
    slot = rng.integers(0, 2, F)
    alpha = rng.random(F)
    mask = np.array([1, 0, 1, 0, 0][:F])
    return kv, cache, slot, alpha, mask


def test_kv_cache_endpoints_and_store():
    kv, cache, slot, alpha, mask = _kv_case(0)
    alpha[:] = 0.0
    out, c = oracle.project_kv_cache(kv, cache, slot, alpha, mask)
    for f in range(5):
        if mask[f]:
            np.testing.assert_array_equal(out[f], kv[f])                  # fresh rows kept
            np.testing.assert_array_equal(c[1 - slot[f], f], kv[f])       # shifted into cache
            np.testing.assert_array_equal(c[slot[f], f], cache[slot[f], f])
        else:
            np.testing.assert_array_equal(out[f], cache[1 - slot[f], f])  # alpha 0: "before"
            np.testing.assert_array_equal(c[:, f], cache[:, f])           # cache untouched
    alpha[:] = 1.0
    out, _ = oracle.project_kv_cache(kv, cache, slot, alpha, mask)
    for f in np.flatnonzero(mask == 0):
        np.testing.assert_array_equal(out[f], cache[slot[f], f])          # alpha 1: "after"


def test_kv_cache_commutes_with_affine_map():
    """Keys and values are an affine map of the hidden state (K = h W + b).  Projecting
    cached keys equals mapping the projected hidden state: the two computation orders
    agree for any weights (a transposed slot or a dropped (1 - alpha) breaks this)."""
    rng = np.random.default_rng(1)
    F, N, C, D = 4, 6, 5, 7
    z = rng.standard_normal((2, F, N, C))
    W = rng.standard_normal((C, D))
    b = rng.standard_normal(D)
    slot = np.array([0, 1, 1, 0])
    alpha = np.array([0.3, 0.0, 0.75, 0.5])
    mask = np.array([0, 0, 0, 1])
    kv_fresh = rng.standard_normal((F, N, D))
    out, _ = oracle.project_kv_cache(kv_fresh, z @ W + b, slot, alpha, mask)
    idx = np.arange(F)
    zp = oracle.project(z[1 - slot, idx].reshape(F, -1), z[slot, idx].reshape(F, -1), alpha)
    want = zp.reshape(F, N, C) @ W + b
    np.testing.assert_allclose(out[:3], want[:3], rtol=0, atol=1e-12)


# --------------------------------------------------------------------------
# Frame mask x token block mask (Appendix D, combined mask)
# --------------------------------------------------------------------------
def test_block_masked_attention_matches_sdpa_with_mask():
    """The element-wise product of the frame mask (rows = active frames' tokens) and a token
    block mask equals torch SDPA with the expanded boolean mask, row by row."""
    g = torch.Generator().manual_seed(9)
    F, N, H, d, blk = 4, 48, 2, 16, 32
    S_tok = F * N
    Q, K, V = (torch.randn(S_tok, H, d, generator=g).to(torch.bfloat16) for _ in range(3))
    nb = (S_tok + blk - 1) // blk
    rng = np.random.default_rng(9)
    bm = (rng.random((H, nb, nb)) < 0.5).astype(np.uint8)
    bm[:, np.arange(nb), np.arange(nb)] = 1           # every query block sees itself
    frame_mask = [1, 0, 1, 1]
    rows = [f * N + p for f in range(F) if frame_mask[f] for p in range(N)]
    O, L = oracle.attention_block_masked(Q, K, V, rows, 0.3, bm, block=blk)
    tok_blk = np.arange(S_tok) // blk
    full = torch.from_numpy(bm[:, tok_blk][:, :, tok_blk] != 0)            # [H, S, S]
    q, k, v = (x.double().permute(1, 0, 2) for x in (Q, K, V))
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=full, scale=0.3)
    np.testing.assert_allclose(O, ref.permute(1, 0, 2).numpy()[rows], rtol=0, atol=1e-12)
    s = 0.3 * q @ k.transpose(1, 2)
    lse = torch.logsumexp(s.masked_fill(~full, -np.inf), dim=-1)
    np.testing.assert_allclose(L, lse.numpy()[:, rows], rtol=0, atol=1e-12)


def test_block_masked_attention_all_allowed_is_dense_and_empty_rows_zero():
    g = torch.Generator().manual_seed(10)
    Q, K, V = (torch.randn(100, 1, 8, generator=g) for _ in range(3))
    ones = np.ones((1, 4, 4), np.uint8)
    O1, L1 = oracle.attention_block_masked(Q, K, V, range(100), 0.5, ones, block=32)
    O2, L2 = oracle.attention(Q, K, V, range(100), 0.5)
    np.testing.assert_allclose(O1, O2, rtol=0, atol=1e-13)
    none = np.zeros((1, 4, 4), np.uint8)
    none[0, 1] = 1                                      # only query block 1 sees anything
    O3, L3 = oracle.attention_block_masked(Q, K, V, [5, 40, 99], 0.5, none, block=32)
    assert (O3[[0, 2]] == 0).all() and np.isneginf(L3[0, [0, 2]]).all()
    np.testing.assert_allclose(O3[1], O2[40], rtol=0, atol=1e-13)
