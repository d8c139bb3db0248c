"""Python binding of librf.so, the RhymeFlow asynchronous step core for GB300.

Argument marshalling only: each function takes torch tensors (or host numpy
arrays for the planner), passes their raw pointers and sizes to the C ABI
declared in ``include/rf.h`` and raises ``RFError`` on a non-OK status.  Every
step of the computation runs in the library's CUDA kernels; there is no CPU or
PyTorch fallback, and a missing library is an error.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

__all__ = ["load", "lib_path", "RFError", "rf_plan_build", "rf_schedule_compact",
           "rf_project", "rf_project_kv", "rf_attn", "rf_attn_block_masked",
           "rf_attn_workspace_bytes", "rf_attn_noalloc", "rf_step", "rf_frame_gram",
           "rf_keyframe_select", "rf_selftest_bounded_wait", "rf_pipeline_create",
           "rf_pipeline_step", "rf_pipeline_sync", "rf_pipeline_bytes", "rf_pipeline_destroy",
           "rf_status_str", "rf_version", "EXPORTS"]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB: Optional[ctypes.CDLL] = None

# Every symbol include/rf.h declares.
EXPORTS = ("rf_status_str", "rf_version", "rf_last_error", "rf_plan_build",
           "rf_schedule_compact", "rf_project", "rf_project_kv", "rf_attn",
           "rf_attn_block_masked", "rf_attn_workspace_bytes",
           "rf_attn_noalloc", "rf_step", "rf_frame_gram", "rf_keyframe_select",
           "rf_pipeline_create", "rf_pipeline_step", "rf_pipeline_sync", "rf_pipeline_bytes",
           "rf_pipeline_destroy", "rf_selftest_bounded_wait")

_vp, _i32, _i64, _f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float
_SIG = {
    "rf_status_str": ([_i32], ctypes.c_char_p),
    "rf_version": ([], _i32),
    "rf_last_error": ([], ctypes.c_char_p),
    "rf_plan_build": ([_i32, _i32, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp], _i32),
    "rf_schedule_compact": ([_vp, _i32, _i32, _vp, _vp, _vp, _vp, _vp], _i32),
    "rf_project": ([_vp, _vp, _vp, _vp, _vp, _i32, _i64, _vp], _i32),
    "rf_project_kv": ([_vp, _vp, _i64, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _i32, _i32,
                       _vp], _i32),
    "rf_attn": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i32, _i32, _i32, _i32, _vp, _vp, _f32,
                 _vp, _i64, _vp, _vp], _i32),
    "rf_attn_workspace_bytes": ([_i32], _i64),
    "rf_attn_block_masked": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i32, _i32, _i32, _i32, _vp,
                              _vp, _f32, _vp, _vp, _i64, _vp, _vp], _i32),
    "rf_selftest_bounded_wait": ([_vp, _i32, _vp], _i32),
    "rf_frame_gram": ([_vp, _i32, _i64, _i64, _vp, _vp], _i32),
    "rf_keyframe_select": ([_vp, _i32, _i32, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                            ctypes.c_double, _vp, _vp], _i32),
    "rf_attn_noalloc": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i32, _i32, _i32, _i32, _vp, _vp,
                         _f32, _vp, _vp], _i32),
    "rf_step": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, _i64, _vp], _i32),
    "rf_pipeline_create": ([_i32, _i32, _i32, _i32, _i64, _i32, _vp, _vp, _vp, _vp, _vp, _vp,
                            _vp, _vp, _i32, _vp, _vp, _vp, ctypes.POINTER(_vp)], _i32),
    "rf_pipeline_step": ([_vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _f32], _i32),
    "rf_pipeline_sync": ([_vp, _vp], _i32),
    "rf_pipeline_bytes": ([_vp, _vp, _vp, _vp], _i32),
    "rf_pipeline_destroy": ([_vp], None),
}


class RFError(RuntimeError):
    def __init__(self, fn: str, status: int):
        detail = load().rf_last_error().decode()
        super().__init__(f"{fn} failed: {rf_status_str(status)} ({status}): {detail}")
        self.status = status


def lib_path() -> str:
    return os.path.join(_HERE, "librf.so")


def load() -> ctypes.CDLL:
    """Load librf.so (built by ``build.build()``); raises if it is missing."""
    global _LIB
    if _LIB is None:
        p = lib_path()
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: build it with __graft_entry__.build() "
                               "(there is no fallback implementation)")
        lib = ctypes.CDLL(p)
        for name, (args, res) in _SIG.items():
            f = getattr(lib, name)
            f.argtypes = args
            f.restype = res
        _LIB = lib
    return _LIB


def _check(fn: str, st: int):
    if st != 0:
        raise RFError(fn, st)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def rf_status_str(status: int) -> str:
    return load().rf_status_str(int(status)).decode()


def rf_version() -> int:
    return load().rf_version()


def rf_plan_build(F: int, S: int, is_key, stride, T_w: int, sigma=None):
    """Host planner.  Returns numpy arrays mask, alpha, beta, dt, cur_slot ([S, F])."""
    is_key = np.ascontiguousarray(np.asarray(is_key, dtype=np.uint8))
    stride = np.ascontiguousarray(np.asarray(stride, dtype=np.int32))
    sig = None if sigma is None else np.ascontiguousarray(np.asarray(sigma, dtype=np.float64))
    mask = np.zeros((S, F), np.uint8)
    alpha = np.zeros((S, F), np.float32)
    beta = np.zeros((S, F), np.float32)
    dt = np.zeros((S, F), np.float32)
    slot = np.zeros((S, F), np.uint8)
    _check("rf_plan_build", load().rf_plan_build(
        F, S, _ptr(is_key), _ptr(stride), T_w, _ptr(sig), _ptr(mask), _ptr(alpha), _ptr(beta),
        _ptr(dt), _ptr(slot)))
    return {"mask": mask, "alpha": alpha, "beta": beta, "dt": dt, "cur_slot": slot}


def rf_schedule_compact(mask, F: int, N: int, active, skipped, token_idx, counts, stream=None):
    _check("rf_schedule_compact", load().rf_schedule_compact(
        _ptr(mask), F, N, _ptr(active), _ptr(skipped), _ptr(token_idx), _ptr(counts),
        _stream(stream)))


def rf_project(ctx, z2, cur_slot, alpha, beta, F: int, E: int, stream=None):
    _check("rf_project", load().rf_project(
        _ptr(ctx), _ptr(z2), _ptr(cur_slot), _ptr(alpha), _ptr(beta), F, E, _stream(stream)))


def rf_project_kv(K, V, kv_row_stride: int, Kc, Vc, cur_slot, alpha, beta, active, skipped,
                  counts, F: int, N: int, D: int, stream=None):
    _check("rf_project_kv", load().rf_project_kv(
        _ptr(K), _ptr(V), kv_row_stride, _ptr(Kc), _ptr(Vc), _ptr(cur_slot), _ptr(alpha),
        _ptr(beta), _ptr(active), _ptr(skipped), _ptr(counts), F, N, D, _stream(stream)))


def rf_attn(O, lse, Q, K, V, qkv_row_stride: int, o_row_stride: int, F: int, N: int, H: int,
            d: int, active, counts, softmax_scale: float, workspace=None, status=None,
            stream=None):
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("rf_attn", load().rf_attn(
        _ptr(O), _ptr(lse), _ptr(Q), _ptr(K), _ptr(V), qkv_row_stride, o_row_stride, F, N, H, d,
        _ptr(active), _ptr(counts), float(softmax_scale), _ptr(workspace), ws_bytes,
        _ptr(status), _stream(stream)))


def rf_attn_block_masked(O, lse, Q, K, V, qkv_row_stride: int, o_row_stride: int, F: int,
                         N: int, H: int, d: int, active, counts, softmax_scale: float, block_mask,
                         workspace=None, status=None, stream=None):
    """rf_attn under the frame mask x token block mask (block_mask uint8 [H, nb, nb])."""
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("rf_attn_block_masked", load().rf_attn_block_masked(
        _ptr(O), _ptr(lse), _ptr(Q), _ptr(K), _ptr(V), qkv_row_stride, o_row_stride, F, N, H, d,
        _ptr(active), _ptr(counts), float(softmax_scale), _ptr(block_mask), _ptr(workspace),
        ws_bytes, _ptr(status), _stream(stream)))


def rf_attn_noalloc(O, lse, Q, K, V, qkv_row_stride: int, o_row_stride: int, F: int, N: int,
                    H: int, d: int, active, counts, softmax_scale: float, status=None,
                    stream=None):
    """rf_attn for callers that cannot allocate: the library's own static scratch."""
    _check("rf_attn_noalloc", load().rf_attn_noalloc(
        _ptr(O), _ptr(lse), _ptr(Q), _ptr(K), _ptr(V), qkv_row_stride, o_row_stride, F, N, H, d,
        _ptr(active), _ptr(counts), float(softmax_scale), _ptr(status), _stream(stream)))


def rf_selftest_bounded_wait(status, limit_us: int, stream=None):
    """Run the device bounded-wait self-test; *status receives RF_ERR_DEVICE_TIMEOUT."""
    _check("rf_selftest_bounded_wait", load().rf_selftest_bounded_wait(
        _ptr(status), int(limit_us), _stream(stream)))


def rf_frame_gram(P, G, stream=None):
    """G[i][j] = <P_i, P_j> for fp32 proxies P [F, E] (row stride P.stride(0)) into fp64 G."""
    F, E = P.shape
    _check("rf_frame_gram", load().rf_frame_gram(_ptr(P), F, E, P.stride(0), _ptr(G),
                                                 _stream(stream)))


def rf_keyframe_select(G, M: int, tau: float, dtau: float, delta_up: float, delta_down: float):
    """Algorithm 1 over a host fp64 Gram matrix; returns the keyframe mask (uint8 [F])."""
    G = np.ascontiguousarray(np.asarray(G, dtype=np.float64))
    F = G.shape[0]
    is_key = np.zeros(F, np.uint8)
    n = np.zeros(1, np.int32)
    _check("rf_keyframe_select", load().rf_keyframe_select(
        _ptr(G), F, M, tau, dtau, delta_up, delta_down, _ptr(is_key), _ptr(n)))
    return is_key


def rf_attn_workspace_bytes(d: int) -> int:
    n = load().rf_attn_workspace_bytes(d)
    if n < 0:
        raise RFError("rf_attn_workspace_bytes", 1)
    return n


def rf_step(z2, cur_slot, v, dt, active, counts, F: int, E: int, stream=None):
    _check("rf_step", load().rf_step(
        _ptr(z2), _ptr(cur_slot), _ptr(v), _ptr(dt), _ptr(active), _ptr(counts), F, E,
        _stream(stream)))


def rf_pipeline_create(F: int, N: int, H: int, d: int, E: int, plan: dict, z2, K0, V0,
                       depth: int, compute, h2d, d2h) -> int:
    """Host-fed step pipeline over the host plan (rf_plan_build's arrays), an initial fp32
    [2, F, E] latent store (host array or tensor) and the initial keys and values K0, V0 (bf16
    [F*N, H, d] contiguous host tensors) that both slots of the rolling cache start with;
    returns an opaque handle."""
    # every array is bound to a name, so that none is freed before the call reads it
    mask = np.ascontiguousarray(plan["mask"], dtype=np.uint8)
    alpha = np.ascontiguousarray(plan["alpha"], dtype=np.float32)
    beta = np.ascontiguousarray(plan["beta"], dtype=np.float32)
    dt = np.ascontiguousarray(plan["dt"], dtype=np.float32)
    slot = np.ascontiguousarray(plan["cur_slot"], dtype=np.uint8)
    z = np.ascontiguousarray(np.asarray(z2.cpu() if hasattr(z2, "cpu") else z2), dtype=np.float32)
    k0, v0 = (x.cpu().contiguous() if hasattr(x, "cpu") else np.ascontiguousarray(x)
              for x in (K0, V0))
    S = mask.shape[0]
    out = _vp()
    _check("rf_pipeline_create", load().rf_pipeline_create(
        F, N, H, d, E, S, _ptr(mask), _ptr(alpha), _ptr(beta), _ptr(dt), _ptr(slot), _ptr(z),
        _ptr(k0), _ptr(v0), depth, _stream(compute), _stream(h2d), _stream(d2h),
        ctypes.byref(out)))
    return out.value


def rf_pipeline_step(handle: int, s: int, hQ, hK, hV, hv, hO, hz2, hctx,
                     softmax_scale: float):
    _check("rf_pipeline_step", load().rf_pipeline_step(
        handle, s, _ptr(hQ), _ptr(hK), _ptr(hV), _ptr(hv), _ptr(hO), _ptr(hz2), _ptr(hctx),
        float(softmax_scale)))


def rf_pipeline_sync(handle: int) -> int:
    """Wait for every enqueued step; returns the device status word."""
    st = np.zeros(1, np.int32)
    _check("rf_pipeline_sync", load().rf_pipeline_sync(handle, _ptr(st)))
    return int(st[0])


def rf_pipeline_bytes(handle: int):
    """(steps, host->device bytes, device->host bytes) enqueued so far."""
    v = np.zeros(3, np.int64)
    _check("rf_pipeline_bytes", load().rf_pipeline_bytes(
        handle, v.ctypes.data, v.ctypes.data + 8, v.ctypes.data + 16))
    return int(v[0]), int(v[1]), int(v[2])


def rf_pipeline_destroy(handle: int):
    if handle:
        load().rf_pipeline_destroy(handle)
