// rf_attn.cu -- active-query x full-sequence attention on sm_103a (tcgen05 / TMEM / TMA).
//
// RhymeFlow (Sec. 3.2.4, Appendix B.2): at each timestep only the active frames issue
// queries, and those queries attend to the keys and values of all F*N tokens.  This kernel
// computes, for every active frame f, token p < N and head h,
//     O[f*N+p, h, :] = softmax_j(scale * q . k_j) V_j     over all F*N tokens j.
//
// Design (one persistent CTA per SM, 384 threads, warp-specialised):
//   warp 0      TMA producer: gathers the two query tiles of a work item by frame index
//               (8-row boxes, so a tile can span several active frames) and streams K/V
//               tiles of 128 tokens through a ring of shared-memory slots.
//   warp 1      owns TMEM (512 columns) and one lane issues every tcgen05.mma:
//               S = Q K^T (both operands in shared memory) and O += P V (P in TMEM).
//   warps 4-7   softmax for query tile A, warps 8-11 for query tile B: thread = query row;
//               online softmax in fp32 with base-2 exponentials, lazy rescaling of the O
//               accumulator (only when the running max grows by more than 2^8), P rounded
//               to bf16 and written back over S in TMEM; final normalisation and bf16 store.
// TMEM columns: S_A [0,128), S_B [128,256), O_A [256,256+d), O_B [384,384+d); P_X aliases
// the first 64 columns of S_X.
//
// MMA issue order per KV tile j (after the prologue S_A(0), S_B(0), PV_A(0)):
//   S_A(j+1), PV_B(j), S_B(j+1), PV_A(j+1)
// so each softmax group has one QK^T and one PV of the other group to hide behind.  Each
// S_X(j+1) is committed after PV_X(j) was issued, so the softmax warps that wait for S_X(j+1)
// also know that O_X is no longer being written and may rescale it in place.  Reuse of the
// S/P columns by the next QK^T relies on tcgen05.mma operations issued by one thread
// executing in issue order.
//
// Work item = (head, pair of 128-row query tiles) over the flattened list of active rows
// (each frame padded to a multiple of 8 rows); items are dealt round-robin to the CTAs, so
// consecutive CTAs share the same head's K/V through L2.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdio>
#include <mutex>

#include "rf_host.h"
#include "rf_ptx.cuh"

namespace rf {
namespace {

constexpr int BM = 128;  // query rows per tile
constexpr int BN = 128;  // keys per KV tile
constexpr int kThreads = 384;  // three warpgroups
// Register split after launch (setmaxnreg): the launch gives 384 x 168 = 64512 registers; the
// producer/MMA warpgroup drops to 104 and each softmax warpgroup grows to 200:
// 128*104 + 2*128*200 = 64512 (the smallest split at which neither side spills).
constexpr int kRegsLaunch = 168, kRegsControl = 104, kRegsSoftmax = 200;
static_assert(128 * kRegsControl + 256 * kRegsSoftmax <= kThreads * kRegsLaunch, "register split");
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s: no legitimate wait comes close
constexpr uint64_t kDrainLimitNs = 200000000ull;  // 0.2 s for in-flight copies at teardown
constexpr float kRescaleLog2 = 8.0f;

template <int D>
struct Cfg {
  static_assert(D == 64 || D == 128, "head dim");
  static constexpr int kHalves = D / 64;          // 128-byte swizzle atoms across the head dim
  static constexpr int kTileBytes = BM * D * 2;   // one Q tile == one K or V tile
  static constexpr int kHalfBytes = BM * 128;     // one 64-column half of a tile
  static constexpr int kSlots = (D == 128) ? 4 : 8;
  static constexpr int kOffKV = 2 * kTileBytes;
  static constexpr int kOffBar = kOffKV + kSlots * kTileBytes;
  // barriers: q_full[2] q_empty[2] kv_full[S] kv_empty[S] s_full[2] p_full[2] o_done[2] drain
  static constexpr int kBarQFull = 0, kBarQEmpty = 2, kBarKVFull = 4, kBarKVEmpty = 4 + kSlots,
                       kBarSFull = 4 + 2 * kSlots, kBarPFull = kBarSFull + 2,
                       kBarODone = kBarPFull + 2, kBarDrain = kBarODone + 2,
                       kNumBars = kBarDrain + 1;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 16 + 1024;  // + slack to align the base
};

struct AttnParams {
  uint16_t* O;
  float* lse;
  const int32_t* active;
  const int32_t* counts;
  int32_t* status;
  int64_t o_row_stride;
  int F, N, Np, H, S_tok, nkv;
  float scale_log2;
};

struct Work {
  int tiles, pairs, items, R;
};

__device__ __forceinline__ Work work_shape(const AttnParams& p) {
  int A = p.counts[0];
  A = A < 0 ? 0 : (A > p.F ? p.F : A);
  Work w;
  w.R = A * p.Np;
  w.tiles = (w.R + BM - 1) / BM;
  w.pairs = (w.tiles + 1) / 2;
  w.items = w.pairs * p.H;
  return w;
}

__device__ __forceinline__ void flag_error(const AttnParams& p, int where) {
  if (p.status) atomicOr(p.status, RF_ERR_DEVICE_TIMEOUT | (1 << (8 + where)));
}

// Wait with no regard to the abort flag (teardown only).
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return;
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > kDrainLimitNs) return;
}

// ---------------------------------------------------------------------------------------
// TMA producer (one thread).
// ---------------------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void producer(const CUtensorMap* tmQ, const CUtensorMap* tmK,
                                         const CUtensorMap* tmV, const AttnParams& p,
                                         const Work& wk, uint32_t sQ0, uint32_t sKV0,
                                         uint32_t bar0, volatile int* abort) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  int q_cnt[2] = {0, 0};
  int it = 0;
  for (int w = blockIdx.x; w < wk.items; w += gridDim.x) {
    const int h = w / wk.pairs, pr = w - h * wk.pairs;
    for (int X = 0; X < 2; ++X) {
      const int t = 2 * pr + X;
      if (t >= wk.tiles) break;
      if (!mbar_wait(bar(C::kBarQEmpty + X), (q_cnt[X] & 1) ^ 1, abort, kWaitLimitNs)) {
        flag_error(p, 0);
        goto drain;
      }
      mbar_arrive_expect_tx(bar(C::kBarQFull + X), C::kTileBytes);
      const uint32_t dst = sQ0 + X * C::kTileBytes;
#pragma unroll 1
      for (int b = 0; b < BM / 8; ++b) {
        const int r = t * BM + b * 8;
        int tok = p.S_tok;  // rows past the active list: out of bounds, zero filled
        if (r < wk.R) {
          const int a = r / p.Np;
          tok = p.active[a] * p.N + (r - a * p.Np);
        }
#pragma unroll
        for (int hb = 0; hb < C::kHalves; ++hb)
          tma_load_3d(dst + hb * C::kHalfBytes + b * 1024, tmQ, bar(C::kBarQFull + X), hb * 64,
                      h, tok);
      }
      ++q_cnt[X];
    }
#pragma unroll 1
    for (int j = 0; j < p.nkv; ++j) {
#pragma unroll
      for (int kv = 0; kv < 2; ++kv) {
        const int s = it % C::kSlots, u = it / C::kSlots;
        if (!mbar_wait(bar(C::kBarKVEmpty + s), (u & 1) ^ 1, abort, kWaitLimitNs)) {
          flag_error(p, 1);
          goto drain;
        }
        mbar_arrive_expect_tx(bar(C::kBarKVFull + s), C::kTileBytes);
        const uint32_t dst = sKV0 + s * C::kTileBytes;
#pragma unroll
        for (int hb = 0; hb < C::kHalves; ++hb)
          tma_load_3d(dst + hb * C::kHalfBytes, kv ? tmV : tmK, bar(C::kBarKVFull + s), hb * 64,
                      h, j * BN);
        ++it;
      }
    }
  }
drain:
  // every armed fill has all its copies issued; wait for the last fill of each buffer
  for (int s = 0; s < C::kSlots; ++s)
    if (it > s) drain_wait(bar(C::kBarKVFull + s), ((it - 1 - s) / C::kSlots) & 1);
  for (int X = 0; X < 2; ++X)
    if (q_cnt[X] > 0) drain_wait(bar(C::kBarQFull + X), (q_cnt[X] - 1) & 1);
}

// ---------------------------------------------------------------------------------------
// MMA issuer (one thread).
// ---------------------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void mma_qk(uint32_t tS, uint32_t sQ, uint32_t sK) {
  constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, 0, 0);
#pragma unroll
  for (int k = 0; k < D / 16; ++k) {
    const uint32_t off = (k >> 2) * (BM * 128) + (k & 3) * 32;
    tc_mma_ss(tS, smem_desc_sw128(sQ + off, 16, 1024), smem_desc_sw128(sK + off, 16, 1024), idesc,
              k > 0);
  }
}

template <int D>
__device__ __forceinline__ void mma_pv(uint32_t tO, uint32_t tP, uint32_t sV, uint32_t acc) {
  constexpr uint32_t idesc = idesc_bf16_f32(BM, D, 0, 1);
#pragma unroll
  for (int k = 0; k < BN / 16; ++k)
    tc_mma_ts(tO, tP + k * 8, smem_desc_sw128(sV + k * 2048, BN * 128, 1024), idesc,
              (acc | k) != 0);
}

template <int D>
__device__ __forceinline__ void mma_issuer(const AttnParams& p, const Work& wk, uint32_t tmem,
                                           uint32_t sQ0, uint32_t sKV0, uint32_t bar0,
                                           volatile int* abort) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const uint32_t tS[2] = {tmem, tmem + 128};
  const uint32_t tO[2] = {tmem + 256, tmem + 384};
  const uint32_t sQ[2] = {sQ0, sQ0 + C::kTileBytes};
  int q_cnt[2] = {0, 0};
  int p_cnt[2] = {0, 0};
  int it = 0;
  auto next_slot = [&](int& s) -> bool {
    s = it % C::kSlots;
    const bool ok = mbar_wait(bar(C::kBarKVFull + s), (it / C::kSlots) & 1, abort, kWaitLimitNs);
    ++it;
    tc_fence_after();
    return ok;
  };
  auto wait_p = [&](int X) -> bool {
    const bool ok = mbar_wait(bar(C::kBarPFull + X), p_cnt[X] & 1, abort, kWaitLimitNs);
    ++p_cnt[X];
    tc_fence_after();
    return ok;
  };
  for (int w = blockIdx.x; w < wk.items; w += gridDim.x) {
    const int h = w / wk.pairs, pr = w - h * wk.pairs;
    (void)h;
    const bool hasB = 2 * pr + 1 < wk.tiles;
    if (!mbar_wait(bar(C::kBarQFull + 0), q_cnt[0] & 1, abort, kWaitLimitNs)) goto fail;
    ++q_cnt[0];
    if (hasB) {
      if (!mbar_wait(bar(C::kBarQFull + 1), q_cnt[1] & 1, abort, kWaitLimitNs)) goto fail;
      ++q_cnt[1];
    }
    tc_fence_after();
    int sK, sV;
    if (!next_slot(sK)) goto fail;
    mma_qk<D>(tS[0], sQ[0], sKV0 + sK * C::kTileBytes);
    tc_commit(bar(C::kBarSFull + 0));
    if (hasB) {
      mma_qk<D>(tS[1], sQ[1], sKV0 + sK * C::kTileBytes);
      tc_commit(bar(C::kBarSFull + 1));
    }
    tc_commit(bar(C::kBarKVEmpty + sK));
    if (!next_slot(sV)) goto fail;
    if (!wait_p(0)) goto fail;
    mma_pv<D>(tO[0], tS[0], sKV0 + sV * C::kTileBytes, 0);
#pragma unroll 1
    for (int j = 0; j + 1 < p.nkv; ++j) {
      if (!next_slot(sK)) goto fail;
      mma_qk<D>(tS[0], sQ[0], sKV0 + sK * C::kTileBytes);
      tc_commit(bar(C::kBarSFull + 0));
      if (hasB) {
        if (!wait_p(1)) goto fail;
        mma_pv<D>(tO[1], tS[1], sKV0 + sV * C::kTileBytes, j > 0);
      }
      tc_commit(bar(C::kBarKVEmpty + sV));
      if (hasB) {
        mma_qk<D>(tS[1], sQ[1], sKV0 + sK * C::kTileBytes);
        tc_commit(bar(C::kBarSFull + 1));
      }
      tc_commit(bar(C::kBarKVEmpty + sK));
      if (!next_slot(sV)) goto fail;
      if (!wait_p(0)) goto fail;
      mma_pv<D>(tO[0], tS[0], sKV0 + sV * C::kTileBytes, 1);
    }
    tc_commit(bar(C::kBarODone + 0));
    tc_commit(bar(C::kBarQEmpty + 0));
    if (hasB) {
      if (!wait_p(1)) goto fail;
      mma_pv<D>(tO[1], tS[1], sKV0 + sV * C::kTileBytes, p.nkv > 1);
      tc_commit(bar(C::kBarODone + 1));
      tc_commit(bar(C::kBarQEmpty + 1));
    }
    tc_commit(bar(C::kBarKVEmpty + sV));
  }
  goto drain;
fail:
  flag_error(p, 2);
drain:
  // all MMAs issued so far complete before TMEM is released
  tc_commit(bar(C::kBarDrain));
  drain_wait(bar(C::kBarDrain), 0);
}

// ---------------------------------------------------------------------------------------
// Softmax / epilogue warpgroup (128 threads, thread = query row of tile X).
// ---------------------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void softmax_group(const AttnParams& p, const Work& wk, int X,
                                              uint32_t tmem, uint32_t bar0,
                                              volatile int* abort) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3;  // TMEM lanes this warp may access
  const int row = quarter * 32 + lane;
  const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
  const uint32_t tS = tmem + lane_base + X * 128;
  const uint32_t tO = tmem + lane_base + 256 + X * 128;
  const float sl2 = p.scale_log2;
  int s_cnt = 0, o_cnt = 0;
  for (int w = blockIdx.x; w < wk.items; w += gridDim.x) {
    const int h = w / wk.pairs, pr = w - h * wk.pairs;
    const int t = 2 * pr + X;
    if (t >= wk.tiles) continue;
    float m = -INFINITY, l = 0.f;
#pragma unroll 1
    for (int j = 0; j < p.nkv; ++j) {
      // the result is made warp-uniform: tcgen05.ld/st below are warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait(bar(C::kBarSFull + X), s_cnt & 1, abort,
                                            kWaitLimitNs))) {
        flag_error(p, 3);
        return;
      }
      ++s_cnt;
      tc_fence_after();
      uint32_t s[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_ld32(tS + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&s[c * 32]));
      tmem_wait_ld();
      float* sf = reinterpret_cast<float*>(s);
      if (j == p.nkv - 1) {
        const int valid = p.S_tok - j * BN;
#pragma unroll
        for (int c = 0; c < BN; ++c)
          if (c >= valid) sf[c] = -INFINITY;
      }
      // row max: 8 independent chains of three-input maxima (a single 128-long chain of
      // two-input maxima is pure latency on the path from QK^T to PV)
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = fmaxf(sf[i], sf[i + 8]);
#pragma unroll
      for (int c = 16; c < BN; c += 16)
#pragma unroll
        for (int i = 0; i < 8; ++i) mx8[i] = fmax3(mx8[i], sf[c + i], sf[c + 8 + i]);
      const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                             fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      const float m_new = fmaxf(m, mx * sl2);
      const bool need = m_new > m + kRescaleLog2;
      const bool rescale = __any_sync(0xffffffffu, need);
      float fac = 1.f;
      if (rescale) {
        fac = ex2_approx(m - m_new);
        l *= fac;
        m = m_new;
      }
      // p = 2^(s*scale*log2(e) - m) with packed fp32 pairs for the scale/subtract and the
      // row sum (8 independent sum chains in 4 packed accumulators)
      const uint64_t sl2x2 = f2_pack(sl2, sl2), nmx2 = f2_pack(-m, -m);
      uint64_t l4[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t pk[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          float x0, x1;
          f2_unpack(ffma2(f2_pack(sf[half * 64 + 2 * e], sf[half * 64 + 2 * e + 1]), sl2x2, nmx2),
                    x0, x1);
          const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          l4[e & 3] = fadd2(l4[e & 3], f2_pack(p0, p1));
          pk[e] = pack_bf16x2(p0, p1);
        }
        tmem_st32(tS + half * 32, pk);
      }
      {
        const uint64_t t = fadd2(fadd2(l4[0], l4[1]), fadd2(l4[2], l4[3]));
        float a, b;
        f2_unpack(t, a, b);
        l += a + b;
      }
      // O was last written by PV(j-1), which completed before S(j) was signalled
      if (rescale && j > 0) {
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + c * 32, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * fac);
          tmem_st32(tO + c * 32, o);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(bar(C::kBarPFull + X));
    }
    // epilogue: O / l -> bf16
    if (!__all_sync(0xffffffffu,
                    mbar_wait(bar(C::kBarODone + X), o_cnt & 1, abort, kWaitLimitNs))) {
      flag_error(p, 4);
      return;
    }
    ++o_cnt;
    tc_fence_after();
    const int r = t * BM + row;
    bool valid = r < wk.R;
    int64_t token = 0;
    if (valid) {
      const int a = r / p.Np, pp = r - a * p.Np;
      valid = pp < p.N;
      token = static_cast<int64_t>(p.active[a]) * p.N + pp;
    }
    const float inv_l = 1.0f / l;
    uint16_t* orow = p.O + token * p.o_row_stride + static_cast<int64_t>(h) * D;
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      uint32_t o[32];
      tmem_ld32(tO + c * 32, o);
      tmem_wait_ld();
      if (valid) {
        uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint4 v;
          v.x = pack_bf16x2(__uint_as_float(o[8 * q + 0]) * inv_l, __uint_as_float(o[8 * q + 1]) * inv_l);
          v.y = pack_bf16x2(__uint_as_float(o[8 * q + 2]) * inv_l, __uint_as_float(o[8 * q + 3]) * inv_l);
          v.z = pack_bf16x2(__uint_as_float(o[8 * q + 4]) * inv_l, __uint_as_float(o[8 * q + 5]) * inv_l);
          v.w = pack_bf16x2(__uint_as_float(o[8 * q + 6]) * inv_l, __uint_as_float(o[8 * q + 7]) * inv_l);
          dst[q] = v;
        }
      }
    }
    if (valid && p.lse)
      p.lse[static_cast<int64_t>(h) * p.S_tok + token] = (m + __log2f(l)) * 0.69314718055994531f;
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const AttnParams p) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t pad = (1024u - (raw & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  const uint32_t sbase = raw + pad;
  const uint32_t sQ0 = sbase, sKV0 = sbase + C::kOffKV, bar0 = sbase + C::kOffBar;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int X = 0; X < 2; ++X) {
      mbar_init(bar0 + 8 * (C::kBarQFull + X), 1);
      mbar_init(bar0 + 8 * (C::kBarQEmpty + X), 1);
      mbar_init(bar0 + 8 * (C::kBarSFull + X), 1);
      mbar_init(bar0 + 8 * (C::kBarPFull + X), 128);
      mbar_init(bar0 + 8 * (C::kBarODone + X), 1);
    }
    for (int s = 0; s < C::kSlots; ++s) {
      mbar_init(bar0 + 8 * (C::kBarKVFull + s), 1);
      mbar_init(bar0 + 8 * (C::kBarKVEmpty + s), 1);
    }
    mbar_init(bar0 + 8 * C::kBarDrain, 1);
    *abort = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const Work wk = work_shape(p);

  // Every warp of warpgroup 0 gives registers back before any softmax warp asks for more,
  // so the increase below always finds them.
  if (warp < 4) {
    reg_dealloc<kRegsControl>();
    if (warp == 0) {
      if (lane == 0) producer<D>(&tmQ, &tmK, &tmV, p, wk, sQ0, sKV0, bar0, abort);
      __syncwarp();
    } else if (warp == 1) {
      if (lane == 0) mma_issuer<D>(p, wk, tmem, sQ0, sKV0, bar0, abort);
      __syncwarp();
    }
  } else {
    reg_alloc<kRegsSoftmax>();
    softmax_group<D>(p, wk, (warp - 4) >> 2, tmem, bar0, abort);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// [S_tok][H][d] bf16 rows of `row_stride` elements, boxes of 64 x 1 x box_rows, 128-byte swizzle.
rf_status make_map(CUtensorMap* m, const void* base, int d, int H, int S_tok, int64_t row_stride,
                   int box_rows) {
  auto enc = encode_fn();
  if (!enc) return fail(RF_ERR_CUDA, "cuTensorMapEncodeTiled entry point not found");
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(H),
                        static_cast<cuuint64_t>(S_tok)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(row_stride) * 2};
  cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r =
      enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
          estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char buf[96];
    std::snprintf(buf, sizeof(buf), "cuTensorMapEncodeTiled failed (CUresult %d)", static_cast<int>(r));
    return fail(RF_ERR_CUDA, buf);
  }
  return RF_OK;
}

template <int D>
rf_status launch(const CUtensorMap& q, const CUtensorMap& k, const CUtensorMap& v,
                 const AttnParams& p, const DeviceInfo& di, cudaStream_t stream) {
  using C = Cfg<D>;
  static bool attr_set[64] = {};
  if (C::kSmemBytes > di.max_smem_optin) return fail(RF_ERR_UNSUPPORTED, "shared memory");
  if (!attr_set[di.device]) {
    if (cudaError_t e = cudaFuncSetAttribute(
            attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes))
      return fail(RF_ERR_CUDA, "cudaFuncSetAttribute(attn_kernel)", e);
    attr_set[di.device] = true;
  }
  const int64_t rows = static_cast<int64_t>(p.F) * p.Np;
  const int64_t tiles = (rows + BM - 1) / BM;
  const int64_t max_items = ((tiles + 1) / 2) * p.H;
  int grid = di.sm_count;
  if (max_items < grid) grid = static_cast<int>(max_items);
  if (grid < 1) grid = 1;
  attn_kernel<D><<<grid, kThreads, C::kSmemBytes, stream>>>(q, k, v, p);
  return launch_status("attn_kernel launch");
}

}  // namespace
}  // namespace rf

using namespace rf;

extern "C" rf_status rf_attn(void* d_O, float* d_lse, const void* d_Q, const void* d_K,
                             const void* d_V, int64_t qkv_row_stride, int64_t o_row_stride, int F,
                             int N, int H, int d, const int32_t* d_active,
                             const int32_t* d_counts, float softmax_scale, int32_t* d_status,
                             rf_stream_t stream) {
  if (!d_O || !d_Q || !d_K || !d_V || !d_active || !d_counts) return RF_ERR_INVALID_ARG;
  if (F < 1 || N < 1 || H < 1 || H > 65535) return RF_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return RF_ERR_UNSUPPORTED;
  if (!(softmax_scale > 0.f) || !std::isfinite(softmax_scale)) return RF_ERR_INVALID_ARG;
  const int64_t S_tok = static_cast<int64_t>(F) * N;
  const int64_t Np = (static_cast<int64_t>(N) + 7) / 8 * 8;
  if (S_tok > 0x7FFFFFFF - BN || static_cast<int64_t>(F) * Np > 0x7FFFFFFF - 2 * BM)
    return RF_ERR_INVALID_ARG;
  if (qkv_row_stride < static_cast<int64_t>(H) * d || o_row_stride < static_cast<int64_t>(H) * d)
    return RF_ERR_INVALID_ARG;
  if (qkv_row_stride % 8 != 0 || o_row_stride % 8 != 0) return RF_ERR_MISALIGNED;
  if (!aligned16(d_Q) || !aligned16(d_K) || !aligned16(d_V) || !aligned16(d_O))
    return RF_ERR_MISALIGNED;
  DeviceInfo di;
  if (rf_status st = current_device_info(&di)) return st;
  if (di.cc_major != 10 || di.cc_minor != 3) return fail(RF_ERR_UNSUPPORTED, "needs sm_103");

  CUtensorMap mq, mk, mv;
  if (rf_status st = make_map(&mq, d_Q, d, H, static_cast<int>(S_tok), qkv_row_stride, 8)) return st;
  if (rf_status st = make_map(&mk, d_K, d, H, static_cast<int>(S_tok), qkv_row_stride, BN)) return st;
  if (rf_status st = make_map(&mv, d_V, d, H, static_cast<int>(S_tok), qkv_row_stride, BN)) return st;

  AttnParams p;
  p.O = static_cast<uint16_t*>(d_O);
  p.lse = d_lse;
  p.active = d_active;
  p.counts = d_counts;
  p.status = d_status;
  p.o_row_stride = o_row_stride;
  p.F = F;
  p.N = N;
  p.Np = static_cast<int>(Np);
  p.H = H;
  p.S_tok = static_cast<int>(S_tok);
  p.nkv = static_cast<int>((S_tok + BN - 1) / BN);
  p.scale_log2 = static_cast<float>(static_cast<double>(softmax_scale) * 1.4426950408889634);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return d == 128 ? launch<128>(mq, mk, mv, p, di, s) : launch<64>(mq, mk, mv, p, di, s);
}
