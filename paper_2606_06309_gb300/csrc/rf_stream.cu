// rf_stream.cu -- the bandwidth kernels of the step core:
//   rf_schedule_compact  active-frame mask -> index lists (warp ballot / popc scan)
//   rf_project           Eq. 3 latent trajectory projection (128-bit streaming)
//   rf_project_kv        rolling key/value cache of Appendix B.2 (bf16, 128-bit streaming)
//   rf_step              Euler update of the active frames (128-bit streaming)
#include <cuda_runtime.h>

#include "rf_host.h"

namespace rf {
namespace {

constexpr int kMaxFrames = 4096;
constexpr int kCompactThreads = 256;

// ---------------------------------------------------------------------------------------
// Compaction.  Every block rebuilds the (tiny) active list in shared memory with a
// ballot/popc scan, block 0 publishes the lists and counts, and all blocks write the
// token index list with a grid-stride loop (int4 stores).
// ---------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kCompactThreads)
    compact_kernel(const uint8_t* __restrict__ mask, int F, int N, int32_t* __restrict__ active,
                   int32_t* __restrict__ skipped, int32_t* __restrict__ token_idx,
                   int32_t* __restrict__ counts) {
  __shared__ int s_active[kMaxFrames];
  __shared__ int s_chunk_base[kMaxFrames / 32 + 1];
  __shared__ int s_A;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nchunks = (F + 31) >> 5;
  // per-32-frame chunk population counts
  for (int c = warp; c < nchunks; c += kCompactThreads / 32) {
    const int f = c * 32 + lane;
    const bool on = f < F && mask[f] != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, on);
    if (lane == 0) s_chunk_base[c] = __popc(bal);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int run = 0;
    for (int c = 0; c < nchunks; ++c) {
      const int n = s_chunk_base[c];
      s_chunk_base[c] = run;
      run += n;
    }
    s_A = run;
  }
  __syncthreads();
  const int A = s_A;
  for (int c = warp; c < nchunks; c += kCompactThreads / 32) {
    const int f = c * 32 + lane;
    const bool on = f < F && mask[f] != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, on);
    const int below = __popc(bal & ((1u << lane) - 1u));
    const int pos_on = s_chunk_base[c] + below;
    if (on) s_active[pos_on] = f;
    if (blockIdx.x == 0 && f < F) {
      if (on)
        active[pos_on] = f;
      else
        skipped[(c * 32 + lane) - pos_on] = f;  // frames before f that are skipped
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    counts[0] = A;
    counts[1] = A * N;
  }
  if (token_idx == nullptr) return;
  __syncthreads();
  const int total = A * N;
  const int nvec = total >> 2;
  int4* out4 = reinterpret_cast<int4*>(token_idx);
  for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < nvec; v += gridDim.x * blockDim.x) {
    int t[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int i = 4 * v + k;
      const int a = i / N;
      t[k] = s_active[a] * N + (i - a * N);
    }
    out4[v] = make_int4(t[0], t[1], t[2], t[3]);
  }
  for (int i = 4 * nvec + blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += gridDim.x * blockDim.x) {
    const int a = i / N;
    token_idx[i] = s_active[a] * N + (i - a * N);
  }
}

// ---------------------------------------------------------------------------------------
// Streaming kernels.  grid = (blocks per frame, F); a block walks its frame's float4s with
// a stride of (blocks per frame * threads), four independent 16-byte loads in flight.
// ---------------------------------------------------------------------------------------
constexpr int kStreamThreads = 256;
constexpr int kUnroll = 4;

__device__ __forceinline__ float4 ld_stream(const float4* p) { return __ldcs(p); }
__device__ __forceinline__ void st_stream(float4* p, float4 v) { __stcs(p, v); }

__global__ void __launch_bounds__(kStreamThreads)
    project_kernel(float4* __restrict__ ctx, const float4* __restrict__ z2,
                   const uint8_t* __restrict__ cur_slot, const float* __restrict__ alpha,
                   const float* __restrict__ beta, int F, int64_t E4) {
  const int f = blockIdx.y;
  const int c = cur_slot[f] & 1;
  const float a = alpha[f], b = beta[f];
  const float4* cur = z2 + (static_cast<int64_t>(c) * F + f) * E4;
  const float4* prev = z2 + (static_cast<int64_t>(c ^ 1) * F + f) * E4;
  float4* out = ctx + static_cast<int64_t>(f) * E4;
  const int64_t step = static_cast<int64_t>(gridDim.x) * kStreamThreads;
  int64_t i = static_cast<int64_t>(blockIdx.x) * kStreamThreads + threadIdx.x;
  if (b == 0.0f) {  // active frame (or alpha == 1): ctx = cur, prev never read
    for (; i + (kUnroll - 1) * step < E4; i += kUnroll * step) {
      float4 v[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) v[u] = ld_stream(cur + i + u * step);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) st_stream(out + i + u * step, v[u]);
    }
    for (; i < E4; i += step) st_stream(out + i, ld_stream(cur + i));
    return;
  }
  for (; i + (kUnroll - 1) * step < E4; i += kUnroll * step) {
    float4 x[kUnroll], y[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      x[u] = ld_stream(cur + i + u * step);
      y[u] = ld_stream(prev + i + u * step);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      float4 r;
      r.x = fmaf(a, x[u].x, b * y[u].x);
      r.y = fmaf(a, x[u].y, b * y[u].y);
      r.z = fmaf(a, x[u].z, b * y[u].z);
      r.w = fmaf(a, x[u].w, b * y[u].w);
      st_stream(out + i + u * step, r);
    }
  }
  for (; i < E4; i += step) {
    const float4 x = ld_stream(cur + i), y = ld_stream(prev + i);
    float4 r;
    r.x = fmaf(a, x.x, b * y.x);
    r.y = fmaf(a, x.y, b * y.y);
    r.z = fmaf(a, x.z, b * y.z);
    r.w = fmaf(a, x.w, b * y.w);
    st_stream(out + i, r);
  }
}

// Euler step over the active frames only.  The active count lives on the device, so the grid
// is fixed (a few waves) and walks (active frame, chunk of kStreamThreads*kUnroll float4s)
// pairs with a stride of gridDim.x chunks: the work spreads over every SM whatever A is.
__global__ void __launch_bounds__(kStreamThreads)
    step_kernel(float4* __restrict__ z2, const uint8_t* __restrict__ cur_slot,
                const float4* __restrict__ vel, const float* __restrict__ dt,
                const int32_t* __restrict__ active, const int32_t* __restrict__ counts, int F,
                int64_t E4) {
  constexpr int64_t kChunk = static_cast<int64_t>(kStreamThreads) * kUnroll;
  int A = counts[0];
  A = A < 0 ? 0 : (A > F ? F : A);
  const int64_t per_frame = (E4 + kChunk - 1) / kChunk;
  const int64_t total = per_frame * A;
  for (int64_t c = blockIdx.x; c < total; c += gridDim.x) {
    const int a = static_cast<int>(c / per_frame);
    const int64_t base = (c - a * per_frame) * kChunk + threadIdx.x;
    const int f = active[a];
    if (f < 0 || f >= F) continue;
    const int sl = cur_slot[f] & 1;
    const float h = dt[f];
    const float4* z = z2 + (static_cast<int64_t>(sl) * F + f) * E4;
    float4* out = z2 + (static_cast<int64_t>(sl ^ 1) * F + f) * E4;
    const float4* v = vel + static_cast<int64_t>(f) * E4;
    float4 x[kUnroll], y[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + u * kStreamThreads;
      if (i < E4) {
        x[u] = ld_stream(z + i);
        y[u] = ld_stream(v + i);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t i = base + u * kStreamThreads;
      if (i < E4) {
        float4 r;
        r.x = fmaf(h, y[u].x, x[u].x);
        r.y = fmaf(h, y[u].y, x[u].y);
        r.z = fmaf(h, y[u].z, x[u].z);
        r.w = fmaf(h, y[u].w, x[u].w);
        st_stream(out + i, r);
      }
    }
  }
}

// ---------------------------------------------------------------------------------------
// Rolling key/value cache (Appendix B.2).  blockIdx.y selects keys or values.  The grid walks
// (frame-list index, chunk) pairs over all F frames: list index a < A is the active frame
// active[a], whose fresh rows are stored into its cache's other slot (shift-and-store); the
// rest are skipped[a - A], whose rows are rewritten with Eq. 3 from the two cached states.
// Eight bf16 per 16-byte access; fp32 arithmetic, rounded to nearest even.
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t proj_pair(uint32_t cur, uint32_t prev, float a, float b) {
  const float lo = fmaf(a, bf16_lo(cur), b * bf16_lo(prev));
  const float hi = fmaf(a, bf16_hi(cur), b * bf16_hi(prev));
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__global__ void __launch_bounds__(kStreamThreads)
    project_kv_kernel(uint16_t* __restrict__ K, uint16_t* __restrict__ V, int64_t row_stride,
                      uint16_t* __restrict__ Kc, uint16_t* __restrict__ Vc,
                      const uint8_t* __restrict__ cur_slot, const float* __restrict__ alpha,
                      const float* __restrict__ beta, const int32_t* __restrict__ active,
                      const int32_t* __restrict__ skipped, const int32_t* __restrict__ counts,
                      int F, int N, int D) {
  uint16_t* X = blockIdx.y ? V : K;
  uint16_t* Xc = blockIdx.y ? Vc : Kc;
  int A = counts[0];
  A = A < 0 ? 0 : (A > F ? F : A);
  const int D8 = D >> 3;                      // 16-byte vectors per row
  const int64_t frame_vecs = static_cast<int64_t>(N) * D8;
  constexpr int64_t kChunk = static_cast<int64_t>(kStreamThreads) * kUnroll;
  const int64_t per_frame = (frame_vecs + kChunk - 1) / kChunk;
  const int64_t total = per_frame * F;
  const int64_t slot_stride = static_cast<int64_t>(F) * N * D;  // elements between slots
  const bool contiguous = row_stride == D;  // K/V rows back to back: no row arithmetic
  for (int64_t c = blockIdx.x; c < total; c += gridDim.x) {
    const int a = static_cast<int>(c / per_frame);
    const int64_t base = (c - a * per_frame) * kChunk + threadIdx.x;
    const bool is_active = a < A;
    const int f = is_active ? active[a] : skipped[a - A];
    if (f < 0 || f >= F) continue;
    const int sl = cur_slot[f] & 1;
    const uint4* cur = reinterpret_cast<const uint4*>(Xc + sl * slot_stride +
                                                      static_cast<int64_t>(f) * N * D);
    uint4* prev = reinterpret_cast<uint4*>(Xc + (sl ^ 1) * slot_stride +
                                           static_cast<int64_t>(f) * N * D);
    uint16_t* rows = X + static_cast<int64_t>(f) * N * row_stride;
    // vector index of the k-th vector of this thread inside the frame's K/V rows: (row, col)
    // advanced incrementally (one division per chunk, none per vector)
    int64_t off[kUnroll];
    {
      int64_t p = 0, q = base;
      if (!contiguous) {
        p = static_cast<uint32_t>(base) / static_cast<uint32_t>(D8);  // < 2^31 (host check)
        q = base - p * D8;
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        off[u] = contiguous ? base + u * kStreamThreads : p * (row_stride >> 3) + q;
        if (!contiguous) {
          q += kStreamThreads;
          while (q >= D8) {
            q -= D8;
            ++p;
          }
        }
      }
    }
    uint4* rv = reinterpret_cast<uint4*>(rows);
    if (is_active) {
      uint4 x[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (base + u * kStreamThreads < frame_vecs) x[u] = __ldcs(rv + off[u]);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t v = base + u * kStreamThreads;
        if (v < frame_vecs) __stcs(prev + v, x[u]);  // the other slot
      }
    } else {
      const float al = alpha[f], be = beta[f];
      uint4 x[kUnroll], y[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t v = base + u * kStreamThreads;
        if (v < frame_vecs) {
          x[u] = __ldcs(cur + v);
          y[u] = __ldcs(prev + v);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        if (base + u * kStreamThreads < frame_vecs) {
          uint4 r;
          r.x = proj_pair(x[u].x, y[u].x, al, be);
          r.y = proj_pair(x[u].y, y[u].y, al, be);
          r.z = proj_pair(x[u].z, y[u].z, al, be);
          r.w = proj_pair(x[u].w, y[u].w, al, be);
          __stcs(rv + off[u], r);
        }
      }
    }
  }
}

// Blocks per frame so that the whole grid covers a few waves of the device even when only
// one frame is active, without launching blocks that would have nothing to do.
int blocks_per_frame(int64_t E4, int sm_count) {
  const int64_t per_block = static_cast<int64_t>(kStreamThreads) * kUnroll;
  int64_t bx = (E4 + per_block - 1) / per_block;
  const int64_t cap = 4LL * sm_count;
  if (bx > cap) bx = cap;
  if (bx < 1) bx = 1;
  return static_cast<int>(bx);
}

}  // namespace
}  // namespace rf

using namespace rf;

extern "C" rf_status rf_schedule_compact(const uint8_t* d_mask, int F, int N, int32_t* d_active,
                                         int32_t* d_skipped, int32_t* d_token_idx,
                                         int32_t* d_counts, rf_stream_t stream) {
  if (!d_mask || !d_active || !d_skipped || !d_counts) return RF_ERR_INVALID_ARG;
  if (F < 1 || F > kMaxFrames || N < 1) return RF_ERR_INVALID_ARG;
  if (static_cast<int64_t>(F) * N > 0x7FFFFFFF) return RF_ERR_INVALID_ARG;
  if (d_token_idx && !aligned16(d_token_idx)) return RF_ERR_MISALIGNED;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  int blocks = 1;
  if (d_token_idx) {
    const int64_t nvec = (static_cast<int64_t>(F) * N + 3) / 4;
    int64_t b = (nvec + kCompactThreads - 1) / kCompactThreads;
    if (b > di.sm_count) b = di.sm_count;
    blocks = static_cast<int>(b < 1 ? 1 : b);
  }
  compact_kernel<<<blocks, kCompactThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      d_mask, F, N, d_active, d_skipped, d_token_idx, d_counts);
  return launch_status("compact_kernel launch");
}

extern "C" rf_status rf_project(float* d_ctx, const float* d_z2, const uint8_t* d_cur_slot,
                                const float* d_alpha, const float* d_beta, int F, int64_t E,
                                rf_stream_t stream) {
  if (!d_ctx || !d_z2 || !d_cur_slot || !d_alpha || !d_beta) return RF_ERR_INVALID_ARG;
  if (F < 1 || F > 65535 || E < 0) return RF_ERR_INVALID_ARG;
  if (E % 4 != 0) return RF_ERR_MISALIGNED;
  if (!aligned16(d_ctx) || !aligned16(d_z2)) return RF_ERR_MISALIGNED;
  if (E == 0) return RF_OK;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  const int64_t E4 = E / 4;
  dim3 grid(blocks_per_frame(E4, di.sm_count), F);
  project_kernel<<<grid, kStreamThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<float4*>(d_ctx), reinterpret_cast<const float4*>(d_z2), d_cur_slot,
      d_alpha, d_beta, F, E4);
  return launch_status("project_kernel launch");
}

extern "C" rf_status rf_step(float* d_z2, const uint8_t* d_cur_slot, const float* d_v,
                             const float* d_dt, const int32_t* d_active, const int32_t* d_counts,
                             int F, int64_t E, rf_stream_t stream) {
  if (!d_z2 || !d_cur_slot || !d_v || !d_dt || !d_active || !d_counts) return RF_ERR_INVALID_ARG;
  if (F < 1 || F > 65535 || E < 0) return RF_ERR_INVALID_ARG;
  if (E % 4 != 0) return RF_ERR_MISALIGNED;
  if (!aligned16(d_z2) || !aligned16(d_v)) return RF_ERR_MISALIGNED;
  if (E == 0) return RF_OK;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  const int64_t E4 = E / 4;
  // enough chunks in flight to cover every SM a few times, never more than the largest A needs
  const int64_t chunk = static_cast<int64_t>(kStreamThreads) * kUnroll;
  int64_t blocks = ((E4 + chunk - 1) / chunk) * F;
  if (blocks > 8LL * di.sm_count) blocks = 8LL * di.sm_count;
  step_kernel<<<static_cast<int>(blocks), kStreamThreads, 0,
                reinterpret_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<float4*>(d_z2), d_cur_slot, reinterpret_cast<const float4*>(d_v), d_dt,
      d_active, d_counts, F, E4);
  return launch_status("step_kernel launch");
}

extern "C" rf_status rf_project_kv(void* d_K, void* d_V, int64_t kv_row_stride, void* d_Kc,
                                   void* d_Vc, const uint8_t* d_cur_slot, const float* d_alpha,
                                   const float* d_beta, const int32_t* d_active,
                                   const int32_t* d_skipped, const int32_t* d_counts, int F,
                                   int N, int D, rf_stream_t stream) {
  if (!d_K || !d_V || !d_Kc || !d_Vc || !d_cur_slot || !d_alpha || !d_beta || !d_active ||
      !d_skipped || !d_counts)
    return RF_ERR_INVALID_ARG;
  if (F < 1 || F > kMaxFrames || N < 1 || D < 8) return RF_ERR_INVALID_ARG;
  if (kv_row_stride < D) return RF_ERR_INVALID_ARG;
  if (static_cast<int64_t>(N) * (D / 8) > 0x7FFFFFFF) return RF_ERR_INVALID_ARG;
  if (D % 8 != 0 || kv_row_stride % 8 != 0) return RF_ERR_MISALIGNED;
  if (!aligned16(d_K) || !aligned16(d_V) || !aligned16(d_Kc) || !aligned16(d_Vc))
    return RF_ERR_MISALIGNED;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  const int64_t frame_vecs = static_cast<int64_t>(N) * (D / 8);
  const int64_t chunk = static_cast<int64_t>(kStreamThreads) * kUnroll;
  int64_t blocks = ((frame_vecs + chunk - 1) / chunk) * F;
  if (blocks > 4LL * di.sm_count) blocks = 4LL * di.sm_count;
  dim3 grid(static_cast<unsigned>(blocks), 2);
  project_kv_kernel<<<grid, kStreamThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      static_cast<uint16_t*>(d_K), static_cast<uint16_t*>(d_V), kv_row_stride,
      static_cast<uint16_t*>(d_Kc), static_cast<uint16_t*>(d_Vc), d_cur_slot, d_alpha, d_beta,
      d_active, d_skipped, d_counts, F, N, D);
  return launch_status("project_kv_kernel launch");
}
