// rf_keyframe.cu -- inner products of the clean-latent proxies for keyframe selection.
//
// Sequential keyframe selection (Sec. 3.1, Eq. 1, Algorithm 1) compares each candidate frame
// with the latest keyframe by cosine similarity.  Which pairs are compared depends on earlier
// decisions, so the device computes every inner product <P_i, P_j> of the F frame proxies at
// once (the Gram matrix; its diagonal gives the norms) and the host runs the sequential rule
// over it (rf_keyframe_select in rf_plan.cpp).
//
// Kernel: split-K over the proxy length E.  Each CTA of 256 threads owns a grid-stride set of
// 128-element slices of every frame, stages them in shared memory k-major, and accumulates
// partial products in registers (4 x 4 per thread, fp32) for the upper triangle of a tile of
// 16, 24, 40, 48 or 64 frames (the smallest that holds F); at the end it adds its tile to the fp64 result with atomics.
#include <cuda_runtime.h>

#include "rf_host.h"

namespace rf {
namespace {

constexpr int kGramMaxF = 64;  // frames per call
constexpr int kGramK = 128;    // elements per stage
constexpr int kGramThreads = 256;

// TILE frames (>= F, padded with zeros).  Thread tiles are 4 x 4; (TILE/4)^2 threads form a
// k-group, and the 256/((TILE/4)^2) k-groups of a CTA take interleaved elements of each stage,
// so small F does not pay for a 64 x 64 product.  The Gram matrix is symmetric: thread tiles
// below the diagonal are skipped and the upper ones written to both halves.  The next stage's
// global loads are issued before the current stage is multiplied (register double buffer).
template <int TILE>
__global__ void __launch_bounds__(kGramThreads)
    gram_kernel(const float* __restrict__ P, int F, int64_t E, int64_t ld, double* __restrict__ G) {
  constexpr int TG = (TILE / 4) * (TILE / 4);  // threads per k-group
  static_assert(TILE % 8 == 0 && TG <= kGramThreads && kGramK % 16 == 0, "tile");
  constexpr int KG = kGramThreads / TG;          // k-groups per CTA (leftover threads only load)
  constexpr int kStageV = TILE * kGramK / 4;     // float4 per stage
  constexpr int NV = (kStageV + kGramThreads - 1) / kGramThreads;  // per thread
  __shared__ __align__(16) float tile[kGramK][TILE + 4];
  __shared__ float red[KG > 1 ? KG : 1][TG][16];
  const int g = threadIdx.x / TG, r = threadIdx.x % TG;
  const int ty = r / (TILE / 4), tx = r % (TILE / 4);
  const bool upper = g < KG && ty <= tx;
  float acc[4][4] = {};
  const bool vec_ok = (ld % 4 == 0) && ((reinterpret_cast<uintptr_t>(P) & 15) == 0);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * kGramK;
  float4 pre[NV];
  // float4 v of a stage -> (frame lf, element lk): a warp's 32 consecutive v cover 8 frames x 16
  // elements (64 contiguous bytes per frame), so the transposed stores below spread over 16
  // banks (2-way) where 32 rows of one frame column would fall into 2 banks (16-way)
  auto frame_of = [](int v) { return ((v >> 5) % (TILE / 8)) * 8 + ((v & 31) >> 2); };
  auto elem_of = [](int v) { return ((v >> 5) / (TILE / 8)) * 16 + (v & 3) * 4; };
  auto load = [&](int64_t k0) {
#pragma unroll
    for (int q = 0; q < NV; ++q) {
      const int v = threadIdx.x + q * kGramThreads;
      const int idx = v * 4;
      const int lf = frame_of(v), lk = elem_of(v);
      const float* prow = P + static_cast<int64_t>(lf) * ld + k0 + lk;
      if (idx >= kStageV * 4) {
        pre[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      } else if (lf < F && vec_ok && k0 + lk + 4 <= E) {
        pre[q] = __ldcs(reinterpret_cast<const float4*>(prow));
      } else {
        float t[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) t[e] = (lf < F && k0 + lk + e < E) ? prow[e] : 0.f;
        pre[q] = make_float4(t[0], t[1], t[2], t[3]);
      }
    }
  };
  int64_t k0 = static_cast<int64_t>(blockIdx.x) * kGramK;
  if (k0 < E) load(k0);
  for (; k0 < E; k0 += stride) {
    __syncthreads();  // the previous stage has been consumed
#pragma unroll
    for (int q = 0; q < NV; ++q) {
      const int v = threadIdx.x + q * kGramThreads;
      if (v * 4 >= kStageV * 4) break;
      const int lf = frame_of(v), lk = elem_of(v);
      tile[lk][lf] = pre[q].x;
      tile[lk + 1][lf] = pre[q].y;
      tile[lk + 2][lf] = pre[q].z;
      tile[lk + 3][lf] = pre[q].w;
    }
    __syncthreads();
    if (k0 + stride < E) load(k0 + stride);  // in flight while this stage is multiplied
    if (upper) {
#pragma unroll 4
      for (int k = g; k < kGramK; k += KG) {
        const float4 a = *reinterpret_cast<const float4*>(&tile[k][ty * 4]);
        const float4 b = *reinterpret_cast<const float4*>(&tile[k][tx * 4]);
        const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) acc[i][jj] = fmaf(av[i], bv[jj], acc[i][jj]);
      }
    }
  }
  if (KG > 1) {  // sum the k-groups' partial tiles
    if (g < KG) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) red[g][r][i * 4 + jj] = acc[i][jj];
    }
    __syncthreads();
    if (g != 0) return;
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int jj = 0; jj < 4; ++jj) {
        float t = 0.f;
        for (int q = 0; q < KG; ++q) t += red[q][r][i * 4 + jj];
        acc[i][jj] = t;
      }
  }
  if (!upper) return;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int fi = ty * 4 + i, fj = tx * 4 + jj;
      if (fi < F && fj < F && acc[i][jj] != 0.f && (ty < tx || fi <= fj)) {
        atomicAdd(G + static_cast<int64_t>(fi) * F + fj, static_cast<double>(acc[i][jj]));
        if (fi != fj)
          atomicAdd(G + static_cast<int64_t>(fj) * F + fi, static_cast<double>(acc[i][jj]));
      }
    }
}

}  // namespace
}  // namespace rf

using namespace rf;

extern "C" rf_status rf_frame_gram(const float* d_P, int F, int64_t E, int64_t ld, double* d_G,
                                   rf_stream_t stream) {
  if (!d_P || !d_G) return RF_ERR_INVALID_ARG;
  if (F < 1 || F > kGramMaxF || E < 1 || ld < E) return RF_ERR_INVALID_ARG;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaError_t e = cudaMemsetAsync(d_G, 0, sizeof(double) * F * F, s))
    return fail(RF_ERR_CUDA, "cudaMemsetAsync(gram)", e);
  int64_t blocks = (E + kGramK - 1) / kGramK;
  if (blocks > 4LL * di.sm_count) blocks = 4LL * di.sm_count;
  const int b = static_cast<int>(blocks);
  if (F <= 16)
    gram_kernel<16><<<b, kGramThreads, 0, s>>>(d_P, F, E, ld, d_G);
  else if (F <= 24)
    gram_kernel<24><<<b, kGramThreads, 0, s>>>(d_P, F, E, ld, d_G);
  else if (F <= 40)
    gram_kernel<40><<<b, kGramThreads, 0, s>>>(d_P, F, E, ld, d_G);
  else if (F <= 48)
    gram_kernel<48><<<b, kGramThreads, 0, s>>>(d_P, F, E, ld, d_G);
  else
    gram_kernel<64><<<b, kGramThreads, 0, s>>>(d_P, F, E, ld, d_G);
  return launch_status("gram_kernel launch");
}
