"""Plain fp64 CPU oracle of one RhymeFlow asynchronous denoising step.

TEST INFRASTRUCTURE ONLY (see the package docstring): the product path never
imports this module.

Citations name the paper's sections, equations and algorithms:

* schedule()        -- Algorithm 2 (asynchronous denoising flow scheduling),
                       Sec. 3.2.1-3.2.3, Eq. 2 (progressive stride), with the
                       "due step" reading of the active-set rule.
* active_set_alg2() -- the active set exactly as Algorithm 2 writes it
                       (non-keyframe j active when (T - T_w - t) = 0 mod n_skip).
* compact()         -- the active set I_active of Algorithm 2 as ordered index
                       lists.
* project()         -- Eq. 3, latent trajectory projection.
* attention()       -- Sec. 3.2.4 / Appendix B.2: active queries attend to the
                       keys and values of all F*N tokens; textbook softmax
                       attention in fp64, brute force over every key.
* euler()           -- the heterogeneous update of Algorithm 2 / Sec. 3.2.3 as a
                       rectified-flow Euler step z <- z + (sigma_to - sigma_from) v.
* attention_block_masked() -- Appendix D, Eq. (combined mask): the frame-level mask of the
                       method times a token-level block mask; active queries attend only
                       to the key blocks their query block allows.
* project_kv_cache() -- Appendix B.2, per-layer rolling cache: skipped frames'
                       keys/values projected with Eq. 3 from the two cached states,
                       active frames' fresh keys/values shifted into the cache.
* keyframe_select() -- Algorithm 1 (dynamic sequential keyframe selection),
                       Eq. 1.  The paper gives no values for tau, delta tau,
                       delta_up or delta_down; they are parameters, and the
                       function is pinned by hand-worked cases (identical frames,
                       orthogonal frames, two angle cases that fix the order of
                       the threshold test and the direction of its adjustment).
* sampler()         -- a whole trajectory of Algorithm 2 with given velocities
                       (schedule, Eq. 3 context and Euler updates in order).
* flops_attn()      -- the attention FLOP count, two per multiply-add; Appendix
                       B.1 prints the same terms at one per multiply-add.

Readings where the paper is silent or inconsistent are stated at each function.
"""
from __future__ import annotations

import math
from typing import Dict, Optional, Sequence

import numpy as np

__all__ = ["sigmas", "schedule", "active_set_alg2", "compact", "project", "attention",
           "euler", "sampler", "flops_attn", "keyframe_select", "project_kv_cache",
           "attention_block_masked", "to_f64"]


def to_f64(x) -> np.ndarray:
    """Widen a torch tensor (bf16/fp32) or array to fp64 exactly."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return x.detach().to("cpu").to(torch.float64).numpy()
    except ImportError:  # pragma: no cover
        pass
    return np.asarray(x, dtype=np.float64)


def sigmas(S: int) -> np.ndarray:
    """Uniform flow-matching noise levels sigma_s = 1 - s/S, s = 0..S (sigma_S = 0)."""
    return np.array([1.0 - s / S for s in range(S + 1)], dtype=np.float64)


def schedule(F: int, S: int, is_key: Sequence[int], stride: Sequence[int], T_w: int,
             sigma: Optional[Sequence[float]] = None) -> Dict[str, np.ndarray]:
    """Per-step active set, projection weights and Euler step sizes (Algorithm 2).

    Step index s = 0..S-1 runs from sigma_0 = 1 (pure noise, the paper's t = T)
    to sigma_S = 0.  For every frame we keep the step at which it last jumped
    (start) and the step its state has reached (due).

    * Warm-up (Sec. 3.2.1): for s < T_w every frame is active, stride 1.
    * Keyframes (Sec. 3.2.3) are active on every step and advance one step.
    * A non-keyframe is active when its state has reached the current step
      (due == s, the "due step" reading of Algorithm 2's modulo rule, which it
      equals whenever the stride is constant); it then jumps n_skip = stride[s]
      steps, clamped so the last jump lands on sigma = 0 (Eq. 2 and Sec. 3.2.3).
    * Euler step size for an active frame: dt = sigma_due - sigma_s.
    * A skipped frame is projected to sigma_s by Eq. 3 from its state before
      its last jump (sigma_start) and after it (sigma_due):
      alpha = (sigma_start - sigma_s) / (sigma_start - sigma_due).  Eq. 3 is
      written in timestep units; with uniform sigma the two agree.  When
      sigma_start == sigma_due (no skipped step) alpha = 0, the identity, as at
      the cache initialisation of Appendix B.2.  Active frames use alpha = 1.

    Returns (all [S, F]): mask (uint8), alpha, beta = 1 - alpha, dt (fp64),
    start, due (int, after the step's update), cur_slot (uint8: which of two
    storage slots holds the frame's current state when step s begins; an active
    frame writes its new state to the other slot).
    """
    sig = sigmas(S) if sigma is None else np.asarray(sigma, dtype=np.float64)
    assert sig.shape == (S + 1,)
    start = [0] * F
    due = [0] * F
    slot = [0] * F
    out = {k: np.zeros((S, F), dtype=np.float64) for k in ("alpha", "beta", "dt")}
    mask = np.zeros((S, F), dtype=np.uint8)
    st = np.zeros((S, F), dtype=np.int64)
    du = np.zeros((S, F), dtype=np.int64)
    cs = np.zeros((S, F), dtype=np.uint8)
    for s in range(S):
        for f in range(F):
            cs[s, f] = slot[f]
            warm = s < T_w
            active = bool(is_key[f]) or warm or due[f] == s
            if active:
                n = 1 if (is_key[f] or warm) else int(stride[s])
                assert n >= 1
                start[f] = s
                due[f] = min(s + n, S)
                mask[s, f] = 1
                out["alpha"][s, f] = 1.0
                out["beta"][s, f] = 0.0
                out["dt"][s, f] = sig[due[f]] - sig[s]
                slot[f] = 1 - slot[f]
            else:
                a0, a1 = sig[start[f]], sig[due[f]]
                alpha = 0.0 if a0 == a1 else (a0 - sig[s]) / (a0 - a1)
                out["alpha"][s, f] = alpha
                out["beta"][s, f] = 1.0 - alpha
                out["dt"][s, f] = 0.0
            st[s, f] = start[f]
            du[s, f] = due[f]
    return {"mask": mask, "alpha": out["alpha"], "beta": out["beta"], "dt": out["dt"],
            "start": st, "due": du, "cur_slot": cs, "sigma": sig}


def active_set_alg2(t: int, T: int, T_w: int, is_key: Sequence[int], n_skip: int):
    """I_active of Algorithm 2 at timestep t (T down to 1), written as printed:
    all frames during warm-up (t > T - T_w); afterwards the keyframes plus every
    non-keyframe j with (T - T_w - t) = 0 mod n_skip."""
    F = len(is_key)
    if t > T - T_w:
        return [f for f in range(F)]
    due = (T - T_w - t) % n_skip == 0
    return [f for f in range(F) if is_key[f] or due]


def compact(mask: Sequence[int], N: int):
    """Ordered index lists of one step's active set (Algorithm 2's I_active).

    active  = frames with mask 1, ascending;  skipped = the rest, ascending;
    token_idx = for each active frame f in order, the tokens f*N + p, p < N;
    counts = [len(active), len(token_idx)].
    """
    active = [f for f in range(len(mask)) if mask[f]]
    skipped = [f for f in range(len(mask)) if not mask[f]]
    token_idx = [f * N + p for f in active for p in range(N)]
    return (np.array(active, dtype=np.int32), np.array(skipped, dtype=np.int32),
            np.array(token_idx, dtype=np.int32),
            np.array([len(active), len(token_idx)], dtype=np.int32))


def project(z_start, z_end, alpha) -> np.ndarray:
    """Eq. 3: z_hat = (1 - alpha) * z_start + alpha * z_end, per frame.

    z_start, z_end: [F, E]; alpha: [F].  fp64."""
    zs = to_f64(z_start)
    ze = to_f64(z_end)
    a = np.asarray(alpha, dtype=np.float64)[:, None]
    return (1.0 - a) * zs + a * ze


def attention(Q, K, V, rows: Sequence[int], scale: float, heads: Optional[Sequence[int]] = None,
              chunk: int = 256):
    """Softmax attention of the query tokens `rows` against every key token.

    Q, K, V: [S_tok, H, d] (any float dtype; widened to fp64 exactly).
    For each head h and query row i:
        s_j = scale * <q_i, k_j>   over all S_tok keys j
        m = max_j s_j,  l = sum_j exp(s_j - m)
        o_i = sum_j exp(s_j - m) v_j / l,   lse_i = m + ln l
    Rows are independent; they are evaluated `chunk` at a time only to bound
    memory.  Returns O [len(rows), len(heads), d] and LSE [len(heads), len(rows)].
    """
    Kf = to_f64(K)
    Vf = to_f64(V)
    Qf = to_f64(Q)
    rows = np.asarray(rows, dtype=np.int64)
    H = Kf.shape[1]
    heads = list(range(H)) if heads is None else list(heads)
    d = Kf.shape[2]
    O = np.zeros((len(rows), len(heads), d), dtype=np.float64)
    L = np.zeros((len(heads), len(rows)), dtype=np.float64)
    for hi, h in enumerate(heads):
        Kh = Kf[:, h, :]
        Vh = Vf[:, h, :]
        for c0 in range(0, len(rows), chunk):
            r = rows[c0:c0 + chunk]
            s = scale * (Qf[r, h, :] @ Kh.T)           # [rows, S_tok]
            m = s.max(axis=1, keepdims=True)
            e = np.exp(s - m)
            l = e.sum(axis=1, keepdims=True)
            O[c0:c0 + chunk, hi, :] = (e @ Vh) / l
            L[hi, c0:c0 + chunk] = (m + np.log(l))[:, 0]
    return O, L


def project_kv_cache(KV, cache, cur_slot, alpha, mask):
    """Per-layer rolling cache of Appendix B.2 for one key or value tensor.

    KV: [F, N, D] the step's keys (or values): rows of active frames are fresh.
    cache: [2, F, N, D] two cached states per frame; slot cur_slot[f] holds the frame's
    latest state ("after"), the other slot the one before it ("before").
    alpha: [F] projection weights of the step; mask: [F] 1 = active.
    Skipped frame: its rows become (1 - alpha) * before + alpha * after (Eq. 3 with the
    cache's two states and the step's weight).  Active frame: its fresh rows are stored as
    the new "after" (into the other slot; the slot flip of the plan makes the old "after"
    the new "before": shift-and-store).
    Returns (KV_out [F, N, D], cache_out [2, F, N, D]) in fp64.
    """
    kv = to_f64(KV).copy()
    c = to_f64(cache).copy()
    for f in range(kv.shape[0]):
        cur = int(cur_slot[f])
        if mask[f]:
            c[1 - cur, f] = kv[f]
        else:
            a = float(alpha[f])
            kv[f] = (1.0 - a) * c[1 - cur, f] + a * c[cur, f]
    return kv, c


def attention_block_masked(Q, K, V, rows, scale, block_mask, block: int = 128,
                           heads: Optional[Sequence[int]] = None):
    """Attention under M_combined = M_Rhyme (element-wise) M_SAP.

    M_Rhyme is the step's frame mask: only the query tokens `rows` (of active frames) are
    computed.  M_SAP is a token-level block mask, block_mask[h][qb][kb] (nonzero = allowed)
    over blocks of `block` consecutive tokens: query token i may attend to key token j only
    when block_mask[h][i // block][j // block] is nonzero.  Scores of excluded keys are
    removed from the softmax.  A row with no allowed key has O = 0 and LSE = -inf.
    """
    Kf, Vf, Qf = to_f64(K), to_f64(V), to_f64(Q)
    M = np.asarray(block_mask)
    rows = np.asarray(rows, dtype=np.int64)
    H, S_tok, d = Kf.shape[1], Kf.shape[0], Kf.shape[2]
    heads = list(range(H)) if heads is None else list(heads)
    kb = np.arange(S_tok) // block
    O = np.zeros((len(rows), len(heads), d), dtype=np.float64)
    L = np.full((len(heads), len(rows)), -np.inf, dtype=np.float64)
    for hi, h in enumerate(heads):
        for ri, i in enumerate(rows):
            allowed = M[h, i // block, kb] != 0
            if not allowed.any():
                continue
            s = scale * (Kf[allowed, h, :] @ Qf[i, h, :])
            m = s.max()
            e = np.exp(s - m)
            l = e.sum()
            O[ri, hi] = (e @ Vf[allowed, h, :]) / l
            L[hi, ri] = m + np.log(l)
    return O, L


def euler(z, v, dt) -> np.ndarray:
    """Rectified-flow Euler update z <- z + dt * v per frame (dt = sigma_to - sigma_from).

    z, v: [F, E]; dt: [F].  fp64."""
    return to_f64(z) + np.asarray(dt, dtype=np.float64)[:, None] * to_f64(v)


def sampler(z0, velocities, plan: Dict[str, np.ndarray]):
    """Run the whole asynchronous trajectory with given per-step velocities.

    z0: [F, E] initial noise; velocities: callable s -> [F, E] (or list).
    At each step the context is: active frames at their true state, skipped
    frames projected by Eq. 3 (Algorithm 2's context C, read as all F frames at
    sigma_s); then active frames take their Euler step.  Returns the final
    states [F, E] and the list of per-step contexts.
    """
    z_cur = to_f64(z0).copy()
    z_prev = z_cur.copy()
    S, F = plan["mask"].shape
    ctxs = []
    for s in range(S):
        ctx = project(z_prev, z_cur, plan["alpha"][s])
        act = plan["mask"][s].astype(bool)
        ctx[act] = z_cur[act]
        ctxs.append(ctx)
        v = to_f64(velocities(s) if callable(velocities) else velocities[s])
        new = euler(z_cur, v, plan["dt"][s])
        z_prev[act] = z_cur[act]
        z_cur[act] = new[act]
    return z_cur, ctxs


def flops_attn(n_query_tokens: int, S_tok: int, d: int, H: int) -> int:
    """Algorithmic attention FLOPs of one call: QK^T and PV, 2 flops per MAC each."""
    return 4 * n_query_tokens * S_tok * d * H


def keyframe_select(proxies, M: int, tau: float, dtau: float, delta_up: float,
                    delta_down: float):
    """Algorithm 1 with Eq. 1 (dynamic sequential keyframe selection).

    proxies: [F, E] clean-latent proxies z_hat_0 (the single-step prediction of
    Algorithm 1's first step is a model call and is an input here).  Frame 0 is
    the first keyframe.  Frames are visited in order; while fewer than M
    keyframes exist, a frame whose cosine similarity to the last keyframe is
    below tau becomes a keyframe, and tau is first moved by -dtau if the gap to
    the last keyframe is at least L_avg + delta_up, or by +dtau if it is at most
    L_avg - delta_down, with L_avg = F / M.  Returns (keyframes, non-keyframes).
    """
    P = to_f64(proxies)
    F = P.shape[0]
    keys = [0]
    last = 0
    L_avg = F / M
    for i in range(1, F):
        if len(keys) < M:
            a, b = P[i], P[last]
            sim = float(a @ b) / (math.sqrt(float(a @ a)) * math.sqrt(float(b @ b)))
            if sim < tau:
                gap = i - last
                if gap >= L_avg + delta_up:
                    tau -= dtau
                elif gap <= L_avg - delta_down:
                    tau += dtau
                keys.append(i)
                last = i
    non = [f for f in range(F) if f not in keys]
    return keys, non
