"""GPU parity: every kernel through the C ABI against the fp64 oracle.

Integer outputs (index lists, counts) must match bit for bit; the fp32
projection and Euler update within 1e-5 relative error measured against the
magnitude of their terms; bf16 attention within the bounds of attn_check.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from attn_check import compare

pytestmark = pytest.mark.gpu

DEV = "cuda"
SENTINEL = 7.0  # rows the kernel must not write keep this value


def _plan(rf, w):
    return rf.rf_plan_build(w.F, w.S, w.is_key, w.stride, w.T_w)


# ---------------------------------------------------------------------------
# rf_schedule_compact
# ---------------------------------------------------------------------------
def _masks():
    out = []
    for name in ("tiny", "small", "mid", "large", "long"):
        w = wl.get(name)
        p = oracle.schedule(w.F, w.S, w.is_key, w.stride, w.T_w)
        for row in np.unique(p["mask"], axis=0):
            out.append((w.N, row))
    rng = np.random.default_rng(0)
    for F in (1, 2, 31, 32, 33, 64, 100, 1000, 4096):
        out.append((int(rng.integers(1, 200)), (rng.random(F) < 0.4).astype(np.uint8)))
    out.append((5, np.zeros(9, np.uint8)))
    out.append((3, np.ones(40, np.uint8)))
    out.append((1, np.array([1], np.uint8)))
    return out


@pytest.mark.parametrize("case", range(len(_masks())))
def test_compact_bit_exact(cuda_lib, case):
    rf = cuda_lib
    N, mask = _masks()[case]
    F = len(mask)
    d_mask = torch.from_numpy(mask).to(DEV)
    act = torch.full((F,), -1, dtype=torch.int32, device=DEV)
    skp = torch.full((F,), -1, dtype=torch.int32, device=DEV)
    tok = torch.full((F * N,), -1, dtype=torch.int32, device=DEV)
    cnt = torch.full((2,), -1, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(d_mask, F, N, act, skp, tok, cnt)
    torch.cuda.synchronize()
    a, s, t, c = oracle.compact(mask, N)
    A = len(a)
    assert cnt.cpu().tolist() == c.tolist()
    assert act.cpu().numpy()[:A].tolist() == a.tolist()
    assert (act.cpu().numpy()[A:] == -1).all()
    assert skp.cpu().numpy()[:F - A].tolist() == s.tolist()
    assert tok.cpu().numpy()[:A * N].tolist() == t.tolist()
    assert (tok.cpu().numpy()[A * N:] == -1).all()


# ---------------------------------------------------------------------------
# rf_project / rf_step
# ---------------------------------------------------------------------------
def _rel_err(g, want, scale):
    return float((np.abs(g - want) / np.maximum(np.maximum(np.abs(want), scale), 1e-30)).max())


@pytest.mark.parametrize("F,E", [(4, 64 * 16), (13, 1560 * 16), (21, 3600 * 16), (3, 4), (5, 1000)])
def test_project_parity(cuda_lib, F, E):
    rf = cuda_lib
    g = torch.Generator().manual_seed(F * 7 + E)
    z2 = torch.randn(2, F, E, generator=g)
    slot = (torch.rand(F, generator=g) < 0.5).to(torch.uint8)
    alpha = torch.rand(F, generator=g)
    active = torch.rand(F, generator=g) < 0.3
    alpha[active] = 1.0
    alpha64 = alpha.double()
    beta = (1.0 - alpha64).float()
    ctx = torch.full((F, E), SENTINEL, device=DEV)
    rf.rf_project(ctx, z2.to(DEV), slot.to(DEV), alpha.to(DEV), beta.to(DEV), F, E)
    torch.cuda.synchronize()
    idx = torch.arange(F)
    cur = z2[slot.long(), idx]
    prev = z2[1 - slot.long(), idx]
    want = oracle.project(prev, cur, alpha64.numpy())
    got = ctx.cpu().double().numpy()
    terms = np.abs(beta.double().numpy()[:, None] * prev.double().numpy()) + \
        np.abs(alpha64.numpy()[:, None] * cur.double().numpy())
    assert _rel_err(got, want, terms) <= 1e-5
    # active frames are copied exactly
    np.testing.assert_array_equal(got[active.numpy()], cur.double().numpy()[active.numpy()])


@pytest.mark.parametrize("F,E", [(4, 64 * 16), (13, 1560 * 16), (33, 3600 * 16), (2, 4)])
def test_step_parity(cuda_lib, F, E):
    rf = cuda_lib
    g = torch.Generator().manual_seed(F + E)
    z2 = torch.randn(2, F, E, generator=g)
    v = torch.randn(F, E, generator=g)
    slot = (torch.rand(F, generator=g) < 0.5).to(torch.uint8)
    dt = -torch.rand(F, generator=g)
    mask = (torch.rand(F, generator=g) < 0.6).to(torch.uint8)
    mask[0] = 1
    d_z2 = z2.to(DEV)
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(mask.to(DEV), F, 1, act, skp, None, cnt)
    rf.rf_step(d_z2, slot.to(DEV), v.to(DEV), dt.to(DEV), act, cnt, F, E)
    torch.cuda.synchronize()
    out = d_z2.cpu()
    idx = torch.arange(F)
    cur = z2[slot.long(), idx]
    want = oracle.euler(cur, v, dt.double().numpy())
    got_new = out[1 - slot.long(), idx].double().numpy()
    m = mask.numpy().astype(bool)
    terms = np.abs(cur.double().numpy()) + np.abs(dt.double().numpy()[:, None] * v.double().numpy())
    assert _rel_err(got_new[m], want[m], terms[m]) <= 1e-5
    # current slots untouched; inactive frames' other slot untouched
    np.testing.assert_array_equal(out[slot.long(), idx].numpy(), cur.numpy())
    np.testing.assert_array_equal(got_new[~m], z2[1 - slot.long(), idx].double().numpy()[~m])


def test_bandwidth_kernels_at_their_frame_limits(cuda_lib):
    """The largest frame counts the calls accept: rf_project over 65535 frames (the grid's
    y limit) of 4 elements; the compaction, rf_step and rf_project_kv over 4096 frames (the
    compaction's limit, which bounds the active lists the other two read); and E = 0, which
    launches nothing and leaves the buffers alone."""
    rf = cuda_lib
    g = torch.Generator().manual_seed(4096)
    # rf_project at F = 65535
    F, E = 65535, 4
    z2 = torch.randn(2, F, E, generator=g)
    slot = (torch.rand(F, generator=g) < 0.5).to(torch.uint8)
    alpha = torch.rand(F, generator=g)
    alpha[::7] = 1.0
    beta = (1.0 - alpha.double()).float()
    ctx = torch.full((F, E), SENTINEL, device=DEV)
    rf.rf_project(ctx, z2.to(DEV), slot.to(DEV), alpha.to(DEV), beta.to(DEV), F, E)
    torch.cuda.synchronize()
    idx = torch.arange(F)
    cur, prev = z2[slot.long(), idx], z2[1 - slot.long(), idx]
    want = oracle.project(prev, cur, alpha.double().numpy())
    terms = np.abs(beta.double().numpy()[:, None] * prev.double().numpy()) + \
        np.abs(alpha.double().numpy()[:, None] * cur.double().numpy())
    assert _rel_err(ctx.cpu().double().numpy(), want, terms) <= 1e-5
    # compaction, rf_step and rf_project_kv at F = 4096
    F, N, D, E = 4096, 1, 8, 8
    mask = (torch.rand(F, generator=g) < 0.3).to(torch.uint8)
    mask[-1] = 1
    act = torch.full((F,), -1, dtype=torch.int32, device=DEV)
    skp = torch.full((F,), -1, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(mask.to(DEV), F, N, act, skp, None, cnt)
    z2 = torch.randn(2, F, E, generator=g)
    v = torch.randn(F, E, generator=g)
    slot = (torch.rand(F, generator=g) < 0.5).to(torch.uint8)
    dt = -torch.rand(F, generator=g)
    d_z2 = z2.to(DEV)
    rf.rf_step(d_z2, slot.to(DEV), v.to(DEV), dt.to(DEV), act, cnt, F, E)
    torch.cuda.synchronize()
    idx = torch.arange(F)
    cur = z2[slot.long(), idx]
    m = mask.numpy().astype(bool)
    got = d_z2.cpu()[1 - slot.long(), idx].double().numpy()
    want = oracle.euler(cur, v, dt.double().numpy())
    terms = np.abs(cur.double().numpy()) + np.abs(dt.double().numpy()[:, None] * v.double().numpy())
    assert _rel_err(got[m], want[m], terms[m]) <= 1e-5
    np.testing.assert_array_equal(got[~m], z2[1 - slot.long(), idx].double().numpy()[~m])
    K = torch.randn(F * N, D, generator=g).to(torch.bfloat16)
    V = torch.randn(F * N, D, generator=g).to(torch.bfloat16)
    Kc = torch.randn(2, F, N, D, generator=g).to(torch.bfloat16)
    Vc = torch.randn(2, F, N, D, generator=g).to(torch.bfloat16)
    al = torch.rand(F, generator=g)
    al[m] = 1.0
    be = (1.0 - al.double()).float()
    dK, dV, dKc, dVc = (x.to(DEV) for x in (K, V, Kc, Vc))
    rf.rf_project_kv(dK, dV, D, dKc, dVc, slot.to(DEV), al.to(DEV), be.to(DEV), act, skp, cnt,
                     F, N, D)
    torch.cuda.synchronize()
    for X, c, dX, dc in ((K, Kc, dK, dKc), (V, Vc, dV, dVc)):
        want, want_c = oracle.project_kv_cache(X.view(F, N, D), c, slot.numpy(), al.numpy(),
                                               mask.numpy())
        got = dX.cpu().double().view(F, N, D).numpy()
        c0 = c.double().numpy()
        sl = slot.numpy().astype(np.int64)
        terms = (np.abs(be.double().numpy())[:, None, None] * np.abs(c0[1 - sl, idx])
                 + np.abs(al.double().numpy())[:, None, None] * np.abs(c0[sl, idx]))
        assert (np.abs(got[~m] - want[~m]) <= 2.0 ** -8 * terms[~m] + 1e-30).all()
        np.testing.assert_array_equal(got[m], X.view(F, N, D).double().numpy()[m])
        np.testing.assert_array_equal(dc.cpu().double().numpy(), want_c)
    # E = 0: nothing is launched, nothing is written
    before = d_z2.clone()
    rf.rf_step(d_z2, slot.to(DEV), v.to(DEV), dt.to(DEV), act, cnt, F, 0)
    rf.rf_project(ctx, d_z2, slot.to(DEV), al.to(DEV), be.to(DEV), F, 0)
    torch.cuda.synchronize()
    assert torch.equal(d_z2, before)


# ---------------------------------------------------------------------------
# rf_attn
# ---------------------------------------------------------------------------
_WS = {}


def _workspace(rf, d):
    """Split-KV workspace, zero-filled once per head dim and reused by every call."""
    if d not in _WS:
        n = rf.rf_attn_workspace_bytes(d)
        _WS[d] = torch.zeros((n + 3) // 4, dtype=torch.int32, device=DEV)
    return _WS[d]


def _run_attn(rf, Q, K, V, F, N, mask, scale, O=None, lse=True, split=True):
    H, d = Q.shape[1], Q.shape[2]
    S_tok = F * N
    if O is None:
        O = torch.full((S_tok, H, d), SENTINEL, dtype=torch.bfloat16, device=DEV)
    L = torch.full((H, S_tok), SENTINEL, dtype=torch.float32, device=DEV) if lse else None
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.as_tensor(np.asarray(mask, np.uint8)).to(DEV), F, N, act, skp,
                           None, cnt)
    ws = _workspace(rf, d) if split else None
    rf.rf_attn(O, L, Q, K, V, Q.stride(0), O.stride(0), F, N, H, d, act, cnt, scale, ws, status)
    torch.cuda.synchronize()
    assert status.item() == 0
    if ws is not None:
        assert int(ws[:1024].abs().sum()) == 0, "merge counters not reset"
    return O, L


def _active_rows(mask, N):
    return [f * N + p for f in range(len(mask)) if mask[f] for p in range(N)]


def _check_attn(Q, K, V, O, L, mask, N, scale, rows=None, heads=None, label=""):
    all_rows = _active_rows(mask, N)
    rows = all_rows if rows is None else rows
    Oref, Lref = oracle.attention(Q.cpu(), K.cpu(), V.cpu(), rows, scale, heads)
    hs = slice(None) if heads is None else list(heads)
    Og = O.cpu().float()[rows][:, hs].numpy()
    Lg = None if L is None else L.cpu()[hs][:, rows].numpy()
    stats = compare(Og, Oref, Lg, Lref if L is not None else None, label)
    # rows of skipped frames are untouched
    skipped = sorted(set(range(len(mask) * N)) - set(all_rows))
    if skipped:
        sk = torch.tensor(skipped[:4096])
        assert (O.cpu()[sk].float() == SENTINEL).all()
        if L is not None:
            assert (L.cpu()[:, sk] == SENTINEL).all()
    return stats


def _qkv(S_tok, H, d, seed, device=DEV):
    g = torch.Generator(device=device).manual_seed(seed)
    return [torch.randn(S_tok, H, d, generator=g, device=device).to(torch.bfloat16)
            for _ in range(3)]


def test_attn_tiny_every_step(cuda_lib):
    rf = cuda_lib
    w = wl.get("tiny")
    Q, K, V = (x.to(DEV) for x in wl.qkv(w))
    p = _plan(rf, w)
    for s in range(w.S):
        O, L = _run_attn(rf, Q, K, V, w.F, w.N, p["mask"][s], w.softmax_scale)
        _check_attn(Q, K, V, O, L, p["mask"][s], w.N, w.softmax_scale, label=f"tiny s={s}")


@pytest.mark.parametrize("F,N,H,d,mask", [
    (3, 1560, 2, 128, [1, 0, 1]),
    (3, 1560, 2, 128, [0, 1, 0]),
    (3, 1560, 1, 128, [1, 1, 1]),
    (5, 100, 2, 64, [1, 0, 1, 1, 0]),     # N % 8 != 0: padded rows
    (5, 100, 3, 128, [0, 0, 0, 0, 1]),
    (2, 8, 2, 64, [1, 1]),                # one tile, no second tile
    (7, 136, 2, 128, [1, 1, 1, 0, 1, 1, 1]),
    (1, 130, 1, 64, [1]),                 # KV tail of 2 keys
    (40, 8, 2, 64, [1, 0] * 20),          # a 128-row tile spans 16 frames (8-row gather)
    (64, 1, 2, 128, [1, 1, 0, 1] * 16),   # N = 1: seven padded rows per frame
    (3, 4096, 1, 128, [1, 0, 1]),         # frames of whole tiles (one 128-row box each)
    (2, 1, 1, 64, [1, 1]),                # two tokens in all
    (1, 8, 1024, 64, [1]),                # 1024 heads of one 8-row tile: many short items
    (2, 4, 300, 128, [0, 1]),             # 300 heads, one active frame of 4 tokens
])
def test_attn_ragged_shapes(cuda_lib, F, N, H, d, mask):
    rf = cuda_lib
    Q, K, V = _qkv(F * N, H, d, seed=F * 1000 + N + d)
    scale = 1.0 / math.sqrt(d)
    O, L = _run_attn(rf, Q, K, V, F, N, mask, scale)
    _check_attn(Q, K, V, O, L, mask, N, scale, label=f"{F}x{N} h{H} d{d} {mask}")


def test_attn_no_active_frames(cuda_lib):
    rf = cuda_lib
    Q, K, V = _qkv(4 * 64, 2, 64, seed=3)
    O, L = _run_attn(rf, Q, K, V, 4, 64, [0, 0, 0, 0], 0.125)
    assert (O.float() == SENTINEL).all() and (L == SENTINEL).all()


def test_attn_strided_rows(cuda_lib):
    """Q, K, V as slices of one fused [tokens, 3, H, d] buffer; O with padded rows."""
    rf = cuda_lib
    F, N, H, d = 4, 200, 3, 128
    g = torch.Generator(device=DEV).manual_seed(11)
    qkv = torch.randn(F * N, 3, H, d, generator=g, device=DEV).to(torch.bfloat16)
    Q, K, V = qkv[:, 0], qkv[:, 1], qkv[:, 2]
    O = torch.full((F * N, H * d + 64), SENTINEL, dtype=torch.bfloat16, device=DEV)
    Ov = O[:, : H * d].view(F * N, H, d)
    mask = [1, 0, 0, 1]
    _run_attn(rf, Q, K, V, F, N, mask, 1 / math.sqrt(d), O=Ov, lse=False)
    _check_attn(Q, K, V, Ov, None, mask, N, 1 / math.sqrt(d), label="strided")
    assert (O[:, H * d:].float() == SENTINEL).all()


def test_attn_planted_keys(cuda_lib):
    """q_i = 16 k_{pi(i)}: each output row must be v_{pi(i)} at O(1) scale."""
    rf = cuda_lib
    F, N, H, d = 3, 256, 2, 128
    g = torch.Generator(device=DEV).manual_seed(5)
    K = torch.randn(F * N, H, d, generator=g, device=DEV).to(torch.bfloat16)
    V = torch.randn(F * N, H, d, generator=g, device=DEV).to(torch.bfloat16)
    perm = torch.randperm(F * N, generator=g, device=DEV)
    Q = (16.0 * K[perm].float()).to(torch.bfloat16)
    O, _ = _run_attn(rf, Q, K, V, F, N, [1, 1, 1], 1 / math.sqrt(d))
    err = (O.float() - V[perm].float()).abs().max().item()
    assert err < 2e-2, err


@pytest.mark.parametrize("direction,mask,split", [
    ("up", [1, 1, 1], True), ("up", [1, 0, 1], False), ("down", [1, 1, 1], False),
    ("down", [0, 1, 1], True)])
def test_attn_running_max_moves_across_tiles(cuda_lib, direction, mask, split):
    """Keys scaled by a ramp along the sequence (x1 to x7), queries x2: with the ramp going up,
    every row's running max keeps growing from one KV tile to the next, so the lazy rescale of
    the accumulator fires many times per row and unnormalised p reaches 2^8 between rescales;
    going down, the max is set by the first tiles and later tiles contribute tiny p."""
    rf = cuda_lib
    F, N, H, d = 3, 700, 2, 128
    Q, K, V = _qkv(F * N, H, d, seed=71 if direction == "up" else 72)
    ramp = torch.linspace(1.0, 7.0, F * N, device=DEV)
    if direction == "down":
        ramp = ramp.flip(0)
    K = (K.float() * ramp[:, None, None]).to(torch.bfloat16)
    Q = (2.0 * Q.float()).to(torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    O, L = _run_attn(rf, Q, K, V, F, N, mask, scale, split=split)
    _check_attn(Q, K, V, O, L, mask, N, scale, label=f"ramp {direction} {mask} split={split}")


@pytest.mark.parametrize("split", [True, False])
def test_attn_extreme_scores_near_argmax(cuda_lib, split):
    """Queries and keys x20 (score std about 400 after the 1/sqrt(d) scale): each row is
    dominated by its largest score, the running max jumps by hundreds of log2 units, and
    nothing may overflow; against the fp64 oracle as usual."""
    rf = cuda_lib
    F, N, H, d = 3, 300, 2, 128
    Q, K, V = _qkv(F * N, H, d, seed=91)
    Q = (20.0 * Q.float()).to(torch.bfloat16)
    K = (20.0 * K.float()).to(torch.bfloat16)
    scale = 1.0 / math.sqrt(d)
    O, L = _run_attn(rf, Q, K, V, F, N, [1, 0, 1], scale, split=split)
    assert torch.isfinite(O.float()).all() and torch.isfinite(L[:, :N]).all()
    _check_attn(Q, K, V, O, L, [1, 0, 1], N, scale, label=f"x20 split={split}")


def test_attn_equal_scores_give_the_mean_of_v(cuda_lib):
    """Q = 0: every score is 0, so every output row is the mean of V over all keys (including
    the partial last key tile) and LSE = ln(S_tok)."""
    rf = cuda_lib
    F, N, H, d = 2, 700, 2, 64
    _, K, V = _qkv(F * N, H, d, seed=92)
    Q = torch.zeros_like(K)
    O, L = _run_attn(rf, Q, K, V, F, N, [1, 1], 0.125)
    mean = V.double().mean(dim=0)                         # [H, d]
    err = (O.double() - mean[None]).abs().max().item()
    assert err < 4e-3, err                                 # bf16 output rounding
    assert (L - math.log(F * N)).abs().max().item() < 1e-4


@pytest.mark.parametrize("name,steps", [("small", (0, 1)), ("mid", (0, 18)), ("large", (0, 1)),
                                        ("long", (0, 12))])
def test_attn_full_size_sampled_rows(cuda_lib, name, steps):
    """The benchmark's launch configuration at full size; sampled rows of every head against
    the oracle: the first and last row of every active frame, the rows around each 128-row
    tile boundary of the first frame, and seeded random rows, 512 rows in all."""
    rf = cuda_lib
    w = wl.get(name)
    Q, K, V = wl.qkv(w, device=DEV)
    p = _plan(rf, w)
    heads = list(range(w.H))
    n_rows = 512
    rng = np.random.default_rng(w.seed)
    for s in steps:
        mask = p["mask"][s]
        O, L = _run_attn(rf, Q, K, V, w.F, w.N, mask, w.softmax_scale)
        act = [f for f in range(w.F) if mask[f]]
        rows = set()
        for f in act:
            rows.update({f * w.N, f * w.N + w.N - 1})
        f0 = act[0]
        for t in range(1, w.N // 128 + 1):
            rows.update({f0 * w.N + min(t * 128 - 1, w.N - 1), f0 * w.N + min(t * 128, w.N - 1)})
        all_rows = np.array(_active_rows(mask, w.N))
        rest = np.setdiff1d(all_rows, np.array(sorted(rows)))
        if len(rows) < n_rows:
            rows.update(rng.choice(rest, size=n_rows - len(rows), replace=False).tolist())
        rows = sorted(rows)
        Oref, Lref = oracle.attention(Q.cpu(), K.cpu(), V.cpu(), rows, w.softmax_scale)
        Og = O.cpu().float()[rows].numpy()
        Lg = L.cpu()[:, rows].numpy()
        compare(Og, Oref, Lg, Lref, f"{name} s={s}")
        # every active row written, no skipped row written
        written = (O[:, heads[0]].float() != SENTINEL).any(dim=1).cpu().numpy()
        expect = np.zeros(w.S_tok, bool)
        expect[all_rows] = True
        assert (written == expect).all()


@pytest.mark.parametrize("s", [0, 1])
def test_attn_small_every_row_of_two_heads(cuda_lib, s):
    """Every active row of the first and last head of the 13 x 1560-token workload, against
    the fp64 oracle, in the benchmark's launch configuration (split-KV workspace)."""
    rf = cuda_lib
    w = wl.get("small")
    Q, K, V = wl.qkv(w, device=DEV)
    p = _plan(rf, w)
    mask = p["mask"][s]
    O, L = _run_attn(rf, Q, K, V, w.F, w.N, mask, w.softmax_scale)
    rows = _active_rows(mask, w.N)
    heads = [0, w.H - 1]
    Oref, Lref = oracle.attention(Q.cpu(), K.cpu(), V.cpu(), rows, w.softmax_scale, heads)
    compare(O.cpu().float()[rows][:, heads].numpy(), Oref, L.cpu()[heads][:, rows].numpy(),
            Lref, f"small s={s} every row, heads {heads}")


@pytest.mark.parametrize("name", ["large", "long"])
def test_attn_every_row_of_two_heads_keyframe_step(cuda_lib, name):
    """Every active row of the first and last head on the keyframe-only step of the 21 and
    33 x 3600-token workloads (6 keyframes: 21600 query rows against all keys), in the
    benchmark's launch configuration, against the fp64 oracle.  The large workload's tokens
    with std 2 give the rows that a few keys dominate."""
    rf = cuda_lib
    w = wl.get(name)
    Q, K, V = wl.qkv(w, device=DEV)
    p = _plan(rf, w)
    s = int(p["mask"].sum(axis=1).argmin())
    mask = p["mask"][s]
    O, L = _run_attn(rf, Q, K, V, w.F, w.N, mask, w.softmax_scale)
    rows = _active_rows(mask, w.N)
    heads = [0, w.H - 1]
    hq = torch.tensor(heads, device=DEV)
    Qs, Ks, Vs = (x.index_select(1, hq).cpu() for x in (Q, K, V))
    Oref, Lref = oracle.attention(Qs, Ks, Vs, rows, w.softmax_scale)
    compare(O.index_select(1, hq).cpu().float()[rows].numpy(), Oref,
            L.index_select(0, hq).cpu()[:, rows].numpy(), Lref,
            f"{name} step {s} every row, heads {heads}")


# ---------------------------------------------------------------------------
# Whole trajectory: compaction + projection + attention + Euler step, S steps
# ---------------------------------------------------------------------------
def _path_magnitude(z0, vels, plan):
    """Per step s and element, M_s = |z0| + sum of |dt * v| over the frame's updates before s:
    a bound on |z_start|, |z_end| and every partial sum that produced them, hence on the terms
    of every fp32 operation behind the state and the context at step s."""
    M = np.abs(oracle.to_f64(z0))
    out = []
    for s in range(plan["mask"].shape[0]):
        out.append(M.copy())
        act = plan["mask"][s].astype(bool)
        M[act] += np.abs(plan["dt"][s][act])[:, None] * np.abs(oracle.to_f64(vels[s])[act])
    out.append(M)
    return out


def _fresh_kv(K0, V0, s):
    """The keys and values the model would compute for step s: K0 and V0 rotated into each other
    by 0.1 s radians (cos K0 + sin V0, cos V0 - sin K0), distinct every step and with the
    workload's distribution (K0 and V0 are independent with the same per-token scales),
    rounded to bf16."""
    c, sn = math.cos(0.1 * s), math.sin(0.1 * s)
    K, V = K0.float(), V0.float()
    return (c * K + sn * V).to(torch.bfloat16), (c * V - sn * K).to(torch.bfloat16)


@pytest.mark.parametrize("name", ["tiny", "small", "mid", "large", "long"])
def test_trajectory_matches_oracle_sampler(cuda_lib, name):
    """Algorithm 2's whole S-step loop through the library, all five calls of every step
    (compaction, Eq. 3 on the latents, Eq. 3 on the rolling key/value cache, attention, Euler
    update on the two-slot store), against the oracle run step by step alongside:

    * the latent context at every step and the final latent, element by element, each
      element's error measured against the magnitude of the terms that produced it (the path
      magnitude M: |z0| plus every |dt * v| the frame took), as the single-call tests measure
      against |beta * prev| + |alpha * cur| and |z| + |dt * v|; after at most 50 fp32
      roundings per element it is below 4e-6 of M;
    * the keys and values attention reads at every step (two heads; elements are independent):
      skipped frames' rows within bf16 rounding of the oracle's cache projection, active
      frames' rows the fresh ones, and the cache itself bit for bit at the end;
    * the attention output of sampled active rows of those heads at several steps, against
      the oracle's attention over the keys and values the kernel read (the bf16 rows the
      previous check pinned to the oracle's projection: the kernel's inputs are bf16 by
      contract, and on rows a few keys dominate the rounding of K alone moves the output).

    The progressive strides (1 -> 4, 1 -> 6) change alpha, dt and the slot bits from one
    segment to the next, which only the whole loop exercises."""
    from paper_2606_06309_gb300.stepcore import StepCore, upload_plan
    w = wl.get(name)
    plan = upload_plan(w.F, w.S, w.is_key, w.stride, w.T_w, DEV)
    E = w.N * w.C
    core = StepCore(w.F, w.N, E, w.H, w.d, plan, DEV)
    z0 = wl.latents(w)
    core.set_state(z0.to(DEV))
    Q, K0, V0 = wl.qkv(w, device=DEV)
    core.set_kv_cache(K0, V0)
    K, V = K0.clone(), V0.clone()
    O = torch.zeros_like(Q)
    vels = [wl.velocity(w, s) for s in range(w.S)]
    oplan = oracle.schedule(w.F, w.S, w.is_key, w.stride, w.T_w)
    zT_ref, ctx_ref = oracle.sampler(z0, vels, oplan)
    mags = _path_magnitude(z0, vels, oplan)

    heads = [0, w.H - 1] if w.H > 1 else [0]
    hidx = torch.tensor(heads, device=DEV)

    def heads_of(X):  # [S_tok, H, d] -> fp64 [F, N, len(heads) * d]
        return oracle.to_f64(X.index_select(1, hidx)).reshape(w.F, w.N, -1)

    cK = np.stack([heads_of(K0)] * 2)
    cV = np.stack([heads_of(V0)] * 2)
    Qh = oracle.to_f64(Q.index_select(1, hidx))
    skip_steps = [s for s in range(w.S) if 0 < oplan["mask"][s].sum() < w.F]
    attn_steps = set(range(w.S)) if w.S_tok * w.H <= 300_000 else \
        {0, skip_steps[0], skip_steps[len(skip_steps) // 2], skip_steps[-1]}
    rng = np.random.default_rng(w.seed)
    worst = 0.0
    for s in range(w.S):
        Kf, Vf = _fresh_kv(K0, V0, s)
        K.copy_(Kf)
        V.copy_(Vf)
        core.run(s, vels[s].to(DEV), O, Q, K, V, w.softmax_scale)
        ctx = core.ctx.cpu().double().numpy()
        err = _rel_err(ctx, ctx_ref[s], mags[s])
        worst = max(worst, err)
        assert err <= 1e-5, (s, err)
        # keys and values the attention read at step s
        mask = oplan["mask"][s]
        sl, al = oplan["cur_slot"][s], oplan["alpha"][s]
        sk = mask == 0
        read = {}
        for X, Xf, c, lab in ((K, Kf, cK, "K"), (V, Vf, cV, "V")):
            fresh = heads_of(Xf)
            want, c_new = oracle.project_kv_cache(fresh, c, sl, al, mask)
            got = heads_of(X)
            read[lab] = got
            if sk.any():
                f_idx = np.flatnonzero(sk)
                terms = (np.abs(1.0 - al[sk])[:, None, None] * np.abs(c[1 - sl[sk], f_idx])
                         + np.abs(al[sk])[:, None, None] * np.abs(c[sl[sk], f_idx]))
                assert (np.abs(got[sk] - want[sk]) <= 2.0 ** -8 * terms + 1e-30).all(), (s, lab)
            np.testing.assert_array_equal(got[~sk], fresh[~sk])
            c[...] = c_new
        if s in attn_steps:
            act = np.flatnonzero(mask)
            rows = {int(f * w.N + p) for f in act for p in (0, w.N - 1)}
            all_rows = np.array(_active_rows(mask, w.N))
            rows.update(rng.choice(all_rows, size=min(64, len(all_rows)), replace=False).tolist())
            rows = sorted(rows)
            shape = (w.S_tok, len(heads), w.d)
            Oref, _ = oracle.attention(Qh, read["K"].reshape(shape), read["V"].reshape(shape),
                                       rows, w.softmax_scale)
            compare(O.index_select(1, hidx).cpu().float().numpy()[rows], Oref,
                    label=f"{name} step {s} attention over projected K/V")
    got = core.current(w.S).cpu().double().numpy()
    err = _rel_err(got, zT_ref, mags[w.S])
    assert err <= 1e-5, err
    for Xc, c in ((core.Kc, cK), (core.Vc, cV)):
        g = oracle.to_f64(Xc.view(2, w.F, w.N, w.H, w.d).index_select(3, hidx))
        np.testing.assert_array_equal(g.reshape(c.shape), c)
    assert core.status.item() == 0
    print(f"{name}: worst context error {worst:.2e}, final latent {err:.2e} (of the path "
          f"magnitude)")


@pytest.mark.parametrize("F,N,H,d,mask", [
    (3, 1560, 2, 128, [1, 0, 1]),
    (5, 100, 2, 64, [1, 0, 1, 1, 0]),
    (13, 1560, 12, 128, [1] * 13),        # 960 items: the last round is split 3 ways
])
def test_attn_split_and_unsplit_agree_with_oracle(cuda_lib, F, N, H, d, mask):
    """The same call with and without the split-KV workspace: both within tolerance of the
    oracle (sampled rows for the large case), and close to each other."""
    rf = cuda_lib
    Q, K, V = _qkv(F * N, H, d, seed=F + N + d)
    scale = 1.0 / math.sqrt(d)
    O1, L1 = _run_attn(rf, Q, K, V, F, N, mask, scale, split=True)
    O2, L2 = _run_attn(rf, Q, K, V, F, N, mask, scale, split=False)
    rows = _active_rows(mask, N)
    if len(rows) > 2048:
        rng = np.random.default_rng(0)
        rows = sorted(rng.choice(rows, 256, replace=False).tolist() + [rows[-1], rows[0]])
    heads = list(range(min(H, 2)))
    hq = torch.tensor(heads, device=DEV)
    Qs, Ks, Vs = (x.index_select(1, hq).cpu() for x in (Q, K, V))
    Oref, Lref = oracle.attention(Qs, Ks, Vs, rows, scale)
    for O, L, lab in ((O1, L1, "split"), (O2, L2, "unsplit")):
        compare(O.cpu().float()[rows][:, heads].numpy(), Oref, L.cpu()[heads][:, rows].numpy(),
                Lref, lab)
    assert (O1.float() - O2.float()).abs().max().item() < 1e-2


def _pipeline_against_device_path(F, N, H, d, E, plan_args, Q, K0, V0, vel, z0, scale, nsteps,
                                  depth):
    """The same steps on device-resident inputs (StepCore, fresh K/V rows written before each
    step) and through the native host-fed pipeline (fresh rows copied from pinned host
    memory, skipped frames' keys/values projected from its own device cache): O of the active
    rows, the latent store and the context must be identical.  Returns the pipeline's byte
    counts per step and the masks."""
    from paper_2606_06309_gb300.stepcore import HostPipeline, StepCore, upload_plan

    def fresh():
        c = StepCore(F, N, E, H, d, upload_plan(F, *plan_args, DEV), DEV)
        c.set_state(z0.to(DEV))
        c.set_kv_cache(K0, V0)
        return c

    kv = [_fresh_kv(K0, V0, s) for s in range(nsteps)]
    ref = fresh()
    O = torch.zeros_like(Q)
    K, V = K0.clone(), V0.clone()
    outs = []
    for s in range(nsteps):
        K.copy_(kv[s][0])
        V.copy_(kv[s][1])
        ref.run(s, vel[s].to(DEV), O, Q, K, V, scale)
        outs.append((O.cpu().clone(), ref.z2.cpu().clone(), ref.ctx.cpu().clone()))
    assert ref.status.item() == 0

    core = fresh()
    pipe = HostPipeline(core, F * N, K0.cpu(), V0.cpu(), DEV, depth=depth)
    hQ = Q.cpu().pin_memory()
    hK = [k.cpu().pin_memory() for k, _ in kv]
    hV = [v.cpu().pin_memory() for _, v in kv]
    hv = [v.cpu().pin_memory() for v in vel[:nsteps]]
    hO = [torch.zeros(Q.shape, dtype=Q.dtype).pin_memory() for _ in range(nsteps)]
    hz = [torch.zeros(core.z2.shape).pin_memory() for _ in range(nsteps)]
    hc = [torch.zeros(core.ctx.shape).pin_memory() for _ in range(nsteps)]
    for s in range(nsteps):
        pipe.step(s, hQ, hK[s], hV[s], hv[s], hO[s], hz[s], scale, hctx=hc[s])
    assert pipe.sync() == 0
    masks = ref.plan.host["mask"]
    for s in range(nsteps):
        act = np.array(_active_rows(masks[s], N))
        assert torch.equal(hO[s][act], outs[s][0][act]), s
        assert torch.equal(hz[s], outs[s][1]), s
        assert torch.equal(hc[s], outs[s][2]), s
        skipped = np.setdiff1d(np.arange(F * N), act)
        assert (hO[s][skipped] == 0).all(), s      # rows no step writes are not copied back
    nbytes = pipe.bytes_per_step()
    pipe.close()
    pipe.close()                                    # closing twice is harmless
    return nbytes, masks


@pytest.mark.parametrize("name,depth", [("tiny", 2), ("tiny", 5), ("small", 3)])
def test_host_pipeline_matches_device_path(cuda_lib, name, depth):
    """The native host-fed pipeline (inputs from pinned host memory, copies overlapped with
    compute, `depth` device buffer sets, its own rolling key/value cache) gives exactly the
    outputs of the same steps run on device-resident inputs, and counts the bytes it copies."""
    w = wl.get(name)
    E = w.N * w.C
    Q, K0, V0 = wl.qkv(w, device=DEV)
    vel = [wl.velocity(w, s) for s in range(w.S)]
    nsteps = min(w.S, 6)
    (h2d, d2h), masks = _pipeline_against_device_path(
        w.F, w.N, w.H, w.d, E, (w.S, w.is_key, w.stride, w.T_w), Q, K0, V0, vel,
        wl.latents(w), w.softmax_scale, nsteps, depth)
    # bytes: the active frames' Q, K and V rows and the velocity in; the active O rows, both
    # latent slots and the context out
    row = w.H * w.d * 2
    n_act = sum(len(_active_rows(masks[s], w.N)) for s in range(nsteps))
    assert h2d == round((3 * n_act * row + nsteps * w.F * E * 4) / nsteps)
    assert d2h == round((n_act * row + nsteps * 3 * w.F * E * 4) / nsteps)


@pytest.mark.parametrize("F,N,H,d,keys,depth", [
    (5, 100, 3, 64, [0, 3], 2),      # N % 8 != 0: padded query tiles, partial frames
    (1, 37, 1, 128, [0], 4),         # one frame, a 37-token sequence (KV tail only)
    (9, 24, 2, 128, [0, 4, 8], 8),   # the deepest buffer ring, more steps in flight than sets
])
def test_host_pipeline_ragged_shapes(cuda_lib, F, N, H, d, keys, depth):
    """The native pipeline on ragged shapes gives the device path's outputs bit for bit."""
    S, E = 10, N * 16
    is_key = [1 if f in keys else 0 for f in range(F)]
    g = torch.Generator(device=DEV).manual_seed(F * 100 + N)
    Q, K0, V0 = (torch.randn(F * N, H, d, generator=g, device=DEV).to(torch.bfloat16)
                 for _ in range(3))
    vel = [torch.randn(F, E, generator=g, device=DEV) for _ in range(S)]
    z0 = torch.randn(F, E, generator=g, device=DEV)
    _pipeline_against_device_path(F, N, H, d, E, (S, is_key, [2] * S, 0), Q, K0, V0, vel, z0,
                                  1 / math.sqrt(d), S, depth)


# ---------------------------------------------------------------------------
# rf_project_kv: rolling key/value cache (Appendix B.2)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("F,N,H,d,fused", [
    (5, 64, 2, 64, False),
    (7, 1560, 12, 128, False),
    (4, 200, 3, 128, True),   # K, V slices of a fused [tokens, 3, H, d] buffer
    (1, 8, 1, 64, False),
])
def test_project_kv_parity(cuda_lib, F, N, H, d, fused):
    rf = cuda_lib
    D = H * d
    g = torch.Generator(device=DEV).manual_seed(F * 17 + N + D)
    if fused:
        qkv = torch.randn(F * N, 3, D, generator=g, device=DEV).to(torch.bfloat16)
        K, V = qkv[:, 1], qkv[:, 2]
    else:
        K = torch.randn(F * N, D, generator=g, device=DEV).to(torch.bfloat16)
        V = torch.randn(F * N, D, generator=g, device=DEV).to(torch.bfloat16)
    Kc = torch.randn(2, F, N, D, generator=g, device=DEV).to(torch.bfloat16)
    Vc = torch.randn(2, F, N, D, generator=g, device=DEV).to(torch.bfloat16)
    rng = np.random.default_rng(F + N)
    mask = (rng.random(F) < 0.4).astype(np.uint8)
    slot = rng.integers(0, 2, F).astype(np.uint8)
    alpha = rng.random(F).astype(np.float32)
    alpha[mask == 1] = 1.0
    beta = (1.0 - alpha.astype(np.float64)).astype(np.float32)
    K0, V0, Kc0, Vc0 = (x.cpu().clone() for x in (K, V, Kc, Vc))
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.from_numpy(mask).to(DEV), F, N, act, skp, None, cnt)
    rf.rf_project_kv(K, V, K.stride(0), Kc, Vc, torch.from_numpy(slot).to(DEV),
                     torch.from_numpy(alpha).to(DEV), torch.from_numpy(beta).to(DEV), act, skp,
                     cnt, F, N, D)
    torch.cuda.synchronize()
    for X, X0, Xc, Xc0 in ((K, K0, Kc, Kc0), (V, V0, Vc, Vc0)):
        want, want_c = oracle.project_kv_cache(X0.view(F, N, D), Xc0, slot, alpha, mask)
        got = X.cpu().double().view(F, N, D).numpy()
        idx = np.arange(F)
        c0 = Xc0.double().numpy()
        sl = slot.astype(np.int64)
        terms = (np.abs(beta.astype(np.float64))[:, None, None] * np.abs(c0[1 - sl, idx])
                 + np.abs(alpha.astype(np.float64))[:, None, None] * np.abs(c0[sl, idx]))
        sk = mask == 0
        err = np.abs(got[sk] - want[sk])
        assert (err <= 2.0 ** -8 * np.abs(terms[sk]) + 1e-30).all(), err.max()
        np.testing.assert_array_equal(got[~sk], X0.view(F, N, D).double().numpy()[~sk])
        # caches: active frames' other slot holds the fresh rows, everything else untouched
        np.testing.assert_array_equal(Xc.cpu().double().numpy(), want_c)
    if fused:
        assert torch.equal(qkv[:, 0].cpu(), qkv[:, 0].cpu())  # Q untouched by construction


def test_project_kv_then_attention_matches_oracle(cuda_lib):
    """The step's keys/values of skipped frames come from the cache projection; attention
    of the active frames over them matches the oracle computed on the projected K/V."""
    rf = cuda_lib
    F, N, H, d = 4, 256, 2, 128
    D = H * d
    g = torch.Generator(device=DEV).manual_seed(7)
    Q, K, V = (torch.randn(F * N, H, d, generator=g, device=DEV).to(torch.bfloat16)
               for _ in range(3))
    Kc, Vc = (torch.randn(2, F, N, D, generator=g, device=DEV).to(torch.bfloat16)
              for _ in range(2))
    mask = np.array([1, 0, 0, 1], np.uint8)
    slot = np.array([0, 1, 0, 1], np.uint8)
    alpha = np.array([1.0, 0.25, 0.5, 1.0], np.float32)
    beta = (1.0 - alpha.astype(np.float64)).astype(np.float32)
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.from_numpy(mask).to(DEV), F, N, act, skp, None, cnt)
    rf.rf_project_kv(K, V, K.stride(0), Kc, Vc, torch.from_numpy(slot).to(DEV),
                     torch.from_numpy(alpha).to(DEV), torch.from_numpy(beta).to(DEV), act, skp,
                     cnt, F, N, D)
    O = torch.full_like(Q, SENTINEL)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    rf.rf_attn(O, None, Q, K, V, Q.stride(0), O.stride(0), F, N, H, d, act, cnt,
               1 / math.sqrt(d), None, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    rows = _active_rows(mask, N)
    Oref, _ = oracle.attention(Q.cpu(), K.cpu(), V.cpu(), rows, 1 / math.sqrt(d))
    compare(O.cpu().float()[rows].numpy(), Oref, label="attention over projected K/V")


# ---------------------------------------------------------------------------
# Keyframe selection: inner products on the device, Algorithm 1 on the host
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("F,E,ld", [(21, 3600 * 16, 3600 * 16), (33, 1000, 1003), (1, 37, 37),
                                    (64, 4096, 4096), (13, 1560 * 16 * 12, 1560 * 16 * 12),
                                    (40, 777, 780), (17, 129, 132)])
def test_frame_gram_matches_fp64_matmul(cuda_lib, F, E, ld):
    rf = cuda_lib
    g = torch.Generator(device=DEV).manual_seed(F + E)
    Pfull = torch.randn(F, ld, generator=g, device=DEV)
    P = Pfull[:, :E]
    G = torch.full((F, F), 7.0, dtype=torch.float64, device=DEV)
    rf.rf_frame_gram(P, G)
    torch.cuda.synchronize()
    ref = P.double().cpu().numpy() @ P.double().cpu().numpy().T
    scale = np.sqrt(np.outer(np.diag(ref), np.diag(ref)))
    err = np.abs(G.cpu().numpy() - ref) / scale
    assert err.max() < 1e-5, err.max()


def test_keyframes_from_device_gram_match_oracle(cuda_lib):
    """Scene-structured proxies (5 scenes over 21 frames of 3600 tokens x 16 channels):
    the keyframes are the scene starts, as the oracle's Algorithm 1 finds them."""
    rf = cuda_lib
    F, E, starts = 21, 3600 * 16, (0, 4, 9, 13, 17)
    rng = np.random.default_rng(3)
    base = rng.standard_normal((len(starts), E))
    scene = np.searchsorted(np.array(starts), np.arange(F), side="right") - 1
    P = base[scene] + 0.3 * rng.standard_normal((F, E))
    Pd = torch.from_numpy(P.astype(np.float32)).to(DEV)
    G = torch.empty(F, F, dtype=torch.float64, device=DEV)
    rf.rf_frame_gram(Pd, G)
    torch.cuda.synchronize()
    for M, tau, dtau in ((8, 0.5, 0.0), (4, 0.5, 0.1), (6, 0.95, -0.2)):
        got = np.flatnonzero(rf.rf_keyframe_select(G.cpu().numpy(), M, tau, dtau, 1.0, 1.0))
        want, _ = oracle.keyframe_select(P.astype(np.float32), M, tau, dtau, 1.0, 1.0)
        assert got.tolist() == want, (M, tau, dtau)
    assert np.flatnonzero(rf.rf_keyframe_select(G.cpu().numpy(), 8, 0.5, 0.0, 1, 1)).tolist() == \
        list(starts)


@pytest.mark.parametrize("name", ["tiny", "small"])
def test_graph_replay_matches_eager(cuda_lib, name):
    """A whole trajectory captured in one CUDA graph and replayed gives the eager results:
    the latent store, the attention output, the keys/values with their projected rows and the
    rolling cache."""
    from paper_2606_06309_gb300.stepcore import StepCore, upload_plan
    w = wl.get(name)
    E = w.N * w.C
    Q, K0, V0 = wl.qkv(w, device=DEV)
    vels = [wl.velocity(w, s, device=DEV) for s in range(w.S)]
    z0 = wl.latents(w, device=DEV)

    def fresh():
        plan = upload_plan(w.F, w.S, w.is_key, w.stride, w.T_w, DEV)
        c = StepCore(w.F, w.N, E, w.H, w.d, plan, DEV)
        c.set_state(z0)
        c.set_kv_cache(K0, V0)
        return c

    eager = fresh()
    O1 = torch.zeros_like(Q)
    K1, V1 = K0.clone(), V0.clone()
    for s in range(w.S):
        eager.run(s, vels[s], O1, Q, K1, V1, w.softmax_scale)
    torch.cuda.synchronize()

    cg = fresh()
    O2 = torch.zeros_like(Q)
    K2, V2 = K0.clone(), V0.clone()
    g = cg.capture_trajectory(vels, O2, Q, K2, V2, w.softmax_scale)  # runs step 0 eagerly
    cg.set_state(z0)
    cg.set_kv_cache(K0, V0)
    K2.copy_(K0)
    V2.copy_(V0)
    O2.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(cg.z2, eager.z2)
    assert torch.equal(O1, O2)
    assert torch.equal(K1, K2) and torch.equal(V1, V2)
    assert torch.equal(cg.Kc, eager.Kc) and torch.equal(cg.Vc, eager.Vc)
    assert cg.status.item() == 0


# ---------------------------------------------------------------------------
# rf_attn_block_masked: frame mask x token block mask (Appendix D)
# ---------------------------------------------------------------------------
def _run_masked(rf, Q, K, V, F, N, mask, scale, bmask, split=True):
    """split=True passes a workspace.  Block-masked launches never split; with a workspace
    they take work items from a queue in its counter words and leave them at zero."""
    H, d = Q.shape[1], Q.shape[2]
    S_tok = F * N
    O = torch.full((S_tok, H, d), SENTINEL, dtype=torch.bfloat16, device=DEV)
    L = torch.full((H, S_tok), SENTINEL, dtype=torch.float32, device=DEV)
    act = torch.zeros(F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.as_tensor(np.asarray(mask, np.uint8)).to(DEV), F, N, act, skp,
                           None, cnt)
    ws = _workspace(rf, d) if split else None
    rf.rf_attn_block_masked(O, L, Q, K, V, Q.stride(0), O.stride(0), F, N, H, d, act, cnt, scale,
                            torch.from_numpy(bmask).to(DEV), ws, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    if ws is not None:
        assert int(ws[:1024].abs().sum()) == 0
    return O, L


def _check_masked(Q, K, V, O, L, mask, N, scale, bmask, label):
    rows = _active_rows(mask, N)
    Oref, Lref = oracle.attention_block_masked(Q.cpu(), K.cpu(), V.cpu(), rows, scale, bmask)
    Og = O.cpu().float()[rows].numpy()
    Lg = L.cpu()[:, rows].numpy()
    empty = np.isneginf(Lref)                      # [H, rows]: no allowed key
    assert (Og.transpose(1, 0, 2)[empty] == 0).all(), label
    assert np.isneginf(Lg[empty]).all(), label
    keep = ~empty.any(axis=0)
    if keep.any():
        compare(Og[keep], Oref[keep], Lg[:, keep], Lref[:, keep], label)
    skipped = sorted(set(range(len(mask) * N)) - set(rows))
    if skipped:
        assert (O.cpu()[torch.tensor(skipped[:4096])].float() == SENTINEL).all()


@pytest.mark.parametrize("name,kind", [("mid", "band"), ("large", "band"), ("large", "causal")])
def test_attn_block_masked_full_size_sampled(cuda_lib, name, kind):
    """Block-masked attention at full size, through the longest-first work queue (workspace):
    the benchmark's banded mask (|qb - kb| <= nb / 8) and a causal block mask (items from one
    key tile to all of them), schedule steps 0 and 1.  Sampled rows: 512 of every head on
    13/21 x 1560 tokens; on 21 x 3600 tokens x 40 heads, 128 rows of four heads spread over
    the head range (the masked oracle gathers each row's allowed keys, 5-12 ms per row and
    head there)."""
    rf = cuda_lib
    w = wl.get(name)
    Q, K, V = wl.qkv(w, device=DEV)
    p = _plan(rf, w)
    nb = (w.S_tok + 127) // 128
    qb, kb = np.meshgrid(np.arange(nb), np.arange(nb), indexing="ij")
    allow = (np.abs(qb - kb) <= max(1, nb // 8)) if kind == "band" else (kb <= qb)
    bmask = np.broadcast_to(allow.astype(np.uint8), (w.H, nb, nb)).copy()
    big = w.S_tok * w.H > 2_000_000
    n_rows = 128 if big else 512
    heads = [0, w.H // 3, 2 * w.H // 3, w.H - 1] if big else list(range(w.H))
    rng = np.random.default_rng(w.seed + 7)
    for s in (0, 1):
        mask = p["mask"][s]
        O, L = _run_masked(rf, Q, K, V, w.F, w.N, mask, w.softmax_scale, bmask)
        all_rows = np.array(_active_rows(mask, w.N))
        rows = {int(r) for f in range(w.F) if mask[f] for r in (f * w.N, f * w.N + w.N - 1)}
        rest = np.setdiff1d(all_rows, np.array(sorted(rows)))
        rows.update(rng.choice(rest, size=n_rows - len(rows), replace=False).tolist())
        rows = sorted(rows)
        Oref, Lref = oracle.attention_block_masked(Q.cpu(), K.cpu(), V.cpu(), rows,
                                                   w.softmax_scale, bmask, heads=heads)
        compare(O.cpu().float()[rows][:, heads].numpy(), Oref, L.cpu()[heads][:, rows].numpy(),
                Lref, f"{name} {kind} s={s}")


@pytest.mark.parametrize("F,N,H,d,mask,density,split", [
    (4, 256, 2, 128, [1, 1, 1, 1], 0.5, True),
    (4, 256, 2, 128, [1, 0, 0, 1], 0.3, False),
    (5, 100, 2, 64, [1, 0, 1, 1, 0], 0.6, True),     # N % 8 != 0
    (3, 1560, 2, 128, [1, 0, 1], 0.4, True),         # ragged KV tail, several tiles per frame
    (3, 1560, 2, 128, [1, 1, 1], 0.15, False),
    # 8-token frames, every 32nd active: a tile pair holds 32 frames in 32 separate query
    # blocks, more ranges than a unit keeps, so the last range is widened (a superset)
    (1024, 8, 2, 64, ([1] + [0] * 31) * 32, 0.3, True),
])
def test_attn_block_masked_parity(cuda_lib, F, N, H, d, mask, density, split):
    rf = cuda_lib
    Q, K, V = _qkv(F * N, H, d, seed=F * 31 + N + d)
    nb = (F * N + 127) // 128
    rng = np.random.default_rng(F + N + int(100 * density))
    bm = (rng.random((H, nb, nb)) < density).astype(np.uint8)
    bm[:, 0, :] = 0                                  # query block 0 may attend to nothing
    scale = 1.0 / math.sqrt(d)
    O, L = _run_masked(rf, Q, K, V, F, N, mask, scale, bm, split)
    _check_masked(Q, K, V, O, L, mask, N, scale, bm, f"{F}x{N} d{d} {mask} p={density}")


def test_attn_block_masked_all_allowed_equals_unmasked(cuda_lib):
    rf = cuda_lib
    F, N, H, d = 3, 1560, 2, 128
    Q, K, V = _qkv(F * N, H, d, seed=77)
    nb = (F * N + 127) // 128
    ones = np.ones((H, nb, nb), np.uint8)
    O1, L1 = _run_masked(rf, Q, K, V, F, N, [1, 0, 1], 0.088, ones)
    O2, L2 = _run_attn(rf, Q, K, V, F, N, [1, 0, 1], 0.088)
    assert (O1.float() - O2.float()).abs().max().item() < 1e-2
    rows = _active_rows([1, 0, 1], N)
    assert (L1[:, rows] - L2[:, rows]).abs().max().item() < 1e-3


def test_attn_block_masked_local_window_and_empty_items(cuda_lib):
    """A local-window mask (each query block sees key blocks within +-2) and a head whose
    mask is empty everywhere (every work item of that head has no key tile at all)."""
    rf = cuda_lib
    F, N, H, d = 5, 512, 2, 128
    Q, K, V = _qkv(F * N, H, d, seed=5)
    nb = (F * N + 127) // 128
    qb, kb = np.meshgrid(np.arange(nb), np.arange(nb), indexing="ij")
    bm = np.zeros((H, nb, nb), np.uint8)
    bm[0] = (np.abs(qb - kb) <= 2)
    mask = [1, 0, 1, 0, 1]
    for split in (True, False):
        O, L = _run_masked(rf, Q, K, V, F, N, mask, 1 / math.sqrt(d), bm, split)
        _check_masked(Q, K, V, O, L, mask, N, 1 / math.sqrt(d), bm, f"window split={split}")
        rows = _active_rows(mask, N)
        assert (O[rows, 1].float() == 0).all() and torch.isneginf(L[1, rows]).all()


def test_attn_block_masked_more_than_1024_key_blocks(cuda_lib):
    """1025 key blocks: a work item's tile bitmap runs past the first 1024 tiles, and one query
    block may attend only to key blocks near the end (the last one ragged, 64 keys)."""
    rf = cuda_lib
    F, N, H, d = 2, 65600, 1, 64
    Q, K, V = _qkv(F * N, H, d, seed=11)
    nb = (F * N + 127) // 128
    assert nb == 1025
    rng = np.random.default_rng(3)
    bm = (rng.random((H, nb, nb)) < 0.02).astype(np.uint8)
    bm[0, :, nb - 1] = 1
    bm[0, 7, :] = 0
    bm[0, 7, 1000:] = 1
    scale = 1.0 / math.sqrt(d)
    O, L = _run_masked(rf, Q, K, V, F, N, [1, 0], scale, bm, split=False)
    rows = np.array([0, 1, 127, 7 * 128, 7 * 128 + 77, 8 * 128 - 1, 30000, 65599])
    Oref, Lref = oracle.attention_block_masked(Q.cpu(), K.cpu(), V.cpu(), rows, scale, bm)
    compare(O.cpu().float()[rows].numpy(), Oref, L.cpu()[:, rows].numpy(), Lref,
            "1025 key blocks")


@pytest.mark.parametrize("split", [True, False])
def test_attn_block_masked_causal_blocks(cuda_lib, split):
    """A causal block mask (key block <= query block): work items differ in cost from one
    key tile to all of them, which the longest-first work queue (with a workspace) and the
    round-robin deal (without) must both compute exactly."""
    rf = cuda_lib
    F, N, H, d = 4, 512, 3, 128
    Q, K, V = _qkv(F * N, H, d, seed=23)
    nb = (F * N + 127) // 128
    qb, kb = np.meshgrid(np.arange(nb), np.arange(nb), indexing="ij")
    bm = np.broadcast_to((kb <= qb).astype(np.uint8), (H, nb, nb)).copy()
    mask = [1, 1, 0, 1]
    O, L = _run_masked(rf, Q, K, V, F, N, mask, 1 / math.sqrt(d), bm, split)
    _check_masked(Q, K, V, O, L, mask, N, 1 / math.sqrt(d), bm, f"causal split={split}")


@pytest.mark.parametrize("split", [True, False])
def test_attn_block_masked_empty_active_set(cuda_lib, split):
    """No active frame: nothing is written, the status stays clear and (with a workspace) the
    work-queue words are back at zero, so the next call on the same workspace is correct."""
    rf = cuda_lib
    F, N, H, d = 3, 512, 2, 128
    Q, K, V = _qkv(F * N, H, d, seed=31)
    nb = (F * N + 127) // 128
    bm = np.ones((H, nb, nb), np.uint8)
    O, L = _run_masked(rf, Q, K, V, F, N, [0, 0, 0], 1 / math.sqrt(d), bm, split)
    assert (O.float() == SENTINEL).all() and (L == SENTINEL).all()
    O, L = _run_masked(rf, Q, K, V, F, N, [0, 1, 0], 1 / math.sqrt(d), bm, split)
    _check_masked(Q, K, V, O, L, [0, 1, 0], N, 1 / math.sqrt(d), bm, f"after empty split={split}")


# ---------------------------------------------------------------------------
# Bandwidth kernels at the hidden-width stress shape the bench times (C = H*d), sampled
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,s", [("small", 1), ("large", 14)])
def test_bandwidth_kernels_at_stress_shape_sampled(cuda_lib, name, s):
    """rf_project, rf_step and rf_project_kv on the full hidden-width buffers of the workload
    (up to 1.5 GB per fp32 buffer), at a step with skipped frames; 65536 sampled elements per
    frame against the oracle, which computes them one by one."""
    rf = cuda_lib
    w = wl.get(name)
    D = w.H * w.d
    E = w.N * D
    p = oracle.schedule(w.F, w.S, w.is_key, w.stride, w.T_w)
    mask = p["mask"][s].astype(np.uint8)
    assert 0 < mask.sum() < w.F
    slot = p["cur_slot"][s].astype(np.uint8)
    alpha = p["alpha"][s].astype(np.float32)
    beta = (1.0 - p["alpha"][s]).astype(np.float32)
    dt = p["dt"][s].astype(np.float32)
    g = torch.Generator(device=DEV).manual_seed(7 + s)
    z2 = torch.randn(2, w.F, E, generator=g, device=DEV)
    v = torch.randn(w.F, E, generator=g, device=DEV)
    act = torch.zeros(w.F, dtype=torch.int32, device=DEV)
    skp = torch.zeros(w.F, dtype=torch.int32, device=DEV)
    cnt = torch.zeros(2, dtype=torch.int32, device=DEV)
    rf.rf_schedule_compact(torch.from_numpy(mask).to(DEV), w.F, w.N, act, skp, None, cnt)
    rng = np.random.default_rng(s)
    idx = torch.from_numpy(np.sort(rng.choice(E, size=65536, replace=False))).to(DEV)
    frames = torch.arange(w.F, device=DEV)
    sl = torch.from_numpy(slot.astype(np.int64)).to(DEV)
    cur = z2[sl, frames][:, idx].cpu().double().numpy()
    prev = z2[1 - sl, frames][:, idx].cpu().double().numpy()
    # Eq. 3 projection
    ctx = torch.full((w.F, E), SENTINEL, device=DEV)
    rf.rf_project(ctx, z2, torch.from_numpy(slot).to(DEV), torch.from_numpy(alpha).to(DEV),
                  torch.from_numpy(beta).to(DEV), w.F, E)
    got = ctx[:, idx].cpu().double().numpy()
    want = oracle.project(prev, cur, p["alpha"][s])
    terms = np.abs(beta.astype(np.float64))[:, None] * np.abs(prev) + \
        np.abs(alpha.astype(np.float64))[:, None] * np.abs(cur)
    assert _rel_err(got, want, terms) <= 1e-5
    del ctx
    # Euler update of the active frames into the other slot
    vs = v[:, idx].cpu().double().numpy()
    rf.rf_step(z2, torch.from_numpy(slot).to(DEV), v, torch.from_numpy(dt).to(DEV), act, cnt,
               w.F, E)
    got_new = z2[1 - sl, frames][:, idx].cpu().double().numpy()
    m = mask.astype(bool)
    want = oracle.euler(cur, vs, dt.astype(np.float64))
    terms = np.abs(cur) + np.abs(dt.astype(np.float64))[:, None] * np.abs(vs)
    assert _rel_err(got_new[m], want[m], terms[m]) <= 1e-5
    np.testing.assert_array_equal(got_new[~m], prev[~m])       # skipped frames untouched
    del z2, v
    # rolling K/V cache: projected rows of skipped frames, fresh rows stored for active ones
    K = torch.randn(w.F * w.N, D, generator=g, device=DEV).to(torch.bfloat16)
    Kc = torch.randn(2, w.F, w.N, D, generator=g, device=DEV).to(torch.bfloat16)
    Vv = torch.randn(w.F * w.N, D, generator=g, device=DEV).to(torch.bfloat16)
    Vc = torch.randn(2, w.F, w.N, D, generator=g, device=DEV).to(torch.bfloat16)
    kcur = Kc[sl, frames].reshape(w.F, E)[:, idx].cpu().double().numpy()
    kprev = Kc[1 - sl, frames].reshape(w.F, E)[:, idx].cpu().double().numpy()
    kfresh = K.view(w.F, E)[:, idx].cpu().double().numpy()
    rf.rf_project_kv(K, Vv, K.stride(0), Kc, Vc, torch.from_numpy(slot).to(DEV),
                     torch.from_numpy(alpha).to(DEV), torch.from_numpy(beta).to(DEV), act, skp,
                     cnt, w.F, w.N, D)
    got_k = K.view(w.F, E)[:, idx].cpu().double().numpy()
    want_k = oracle.project(kprev, kcur, p["alpha"][s])
    terms = np.abs(beta.astype(np.float64))[:, None] * np.abs(kprev) + \
        np.abs(alpha.astype(np.float64))[:, None] * np.abs(kcur)
    sk = ~m
    assert (np.abs(got_k[sk] - want_k[sk]) <= 2.0 ** -8 * terms[sk] + 1e-30).all()
    np.testing.assert_array_equal(got_k[m], kfresh[m])          # active rows untouched
    stored = Kc[1 - sl, frames].reshape(w.F, E)[:, idx].cpu().double().numpy()
    np.testing.assert_array_equal(stored[m], kfresh[m])         # fresh rows shifted in
    np.testing.assert_array_equal(stored[sk], kprev[sk])        # skipped frames' cache kept


def test_attn_block_masked_queue_with_several_head_groups(cuda_lib):
    """A sequence long enough that only some heads' K/V fit in half of L2, so the longest-first
    pre-pass orders the items in more than one group of heads (the last one smaller); a causal
    block mask makes the costs differ.  Sampled rows of every head against the oracle, and a
    second call on the same workspace (the group counters must be back at zero)."""
    rf = cuda_lib
    F, N, H, d = 2, 65536, 3, 64
    Q, K, V = _qkv(F * N, H, d, seed=41)
    nb = (F * N + 127) // 128
    qb, kb = np.meshgrid(np.arange(nb), np.arange(nb), indexing="ij")
    bm = np.broadcast_to((kb <= qb).astype(np.uint8), (H, nb, nb)).copy()
    scale = 1.0 / math.sqrt(d)
    rows = np.array([0, 127, 128, 5000, 65535, 65536, 70000, 100000, 131071])
    for call in range(2):
        O, L = _run_masked(rf, Q, K, V, F, N, [1, 1], scale, bm, split=True)
        Oref, Lref = oracle.attention_block_masked(Q.cpu(), K.cpu(), V.cpu(), rows, scale, bm)
        compare(O.cpu().float()[rows].numpy(), Oref, L.cpu()[:, rows].numpy(), Lref,
                f"several head groups, call {call}")
