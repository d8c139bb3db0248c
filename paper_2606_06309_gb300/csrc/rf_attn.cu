// rf_attn.cu -- active-query x full-sequence attention on sm_103a (tcgen05 / TMEM / TMA).
//
// RhymeFlow (Sec. 3.2.4, Appendix B.2): at each timestep only the active frames issue
// queries, and those queries attend to the keys and values of all F*N tokens.  This kernel
// computes, for every active frame f, token p < N and head h,
//     O[f*N+p, h, :] = softmax_j(scale * q . k_j) V_j     over all F*N tokens j.
//
// Design (one persistent CTA per SM, 384 threads, warp-specialised):
//   warp 0      TMA producer: loads the two query tiles of a work item (one 128-row box
//               when the tile lies in one active frame, else gathered by frame index in
//               8-row boxes) and streams K/V tiles of 128 tokens through a ring of
//               shared-memory slots.
//   warp 1      owns TMEM (512 columns) and one lane issues every tcgen05.mma:
//               S = Q K^T (both operands in shared memory) and O += P V (P in TMEM).
//   warp 2      (block-masked launches) builds each work item's list of KV tiles.
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
// consecutive CTAs share the same head's K/V through L2 (block-masked launches with a
// workspace take items from a longest-first work queue instead).  When the last round of items
// would leave more than half of the CTAs idle and the caller supplied a workspace, each item of
// that round is split into C ranges of KV tiles (split-KV, unmasked launches only): every range
// writes its unnormalised O row, running max and sum to the workspace, and the CTA that
// finishes the last range of an item merges them (counter per item and query tile, reset to
// zero by the merging CTA).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <mutex>

#include "rf_host.h"
#include "rf_ptx.cuh"

namespace rf {
namespace {

constexpr int BM = 128;       // query rows per tile
constexpr int BN = 128;       // keys per KV tile
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
constexpr int kMaxSplit = 16;          // KV ranges per split item
constexpr int kMaxGrid = 1024;         // workspace is sized for at most this many CTAs
// Block-masked launches: a ring of per-unit KV-tile bitmaps in shared memory, one bit per KV
// tile (so at most kTLWords * 32 tiles of 128 keys), followed by the number of set bits.
constexpr int kTLSlots = 4;
constexpr int kTLWords = 128;
constexpr int kTLSlotBytes = kTLWords * 4 + 16;
constexpr int kTLMaxTiles = kTLWords * 32;

template <int D>
struct Cfg {
  static_assert(D == 64 || D == 128, "head dim");
  static constexpr int kHalves = D / 64;          // 128-byte swizzle atoms across the head dim
  static constexpr int kTileBytes = BM * D * 2;   // one Q tile == one K or V tile
  static constexpr int kHalfBytes = BM * 128;     // one 64-column half of a tile
  static constexpr int kSlots = (D == 128) ? 4 : 8;
  static constexpr int kOffKV = 2 * kTileBytes;
  static constexpr int kOffBar = kOffKV + kSlots * kTileBytes;
  // barriers: q_full[2] q_empty[2] kv_full[S] kv_empty[S] s_full[2] p_full[2] o_done[2]
  // group[2] (the 128 threads of one softmax warpgroup) drain
  static constexpr int kBarQFull = 0, kBarQEmpty = 2, kBarKVFull = 4, kBarKVEmpty = 4 + kSlots,
                       kBarSFull = 4 + 2 * kSlots, kBarPFull = kBarSFull + 2,
                       kBarODone = kBarPFull + 2, kBarGroup = kBarODone + 2,
                       kBarDrain = kBarGroup + 2, kNumBars = kBarDrain + 1;
  // misc: tmem address, abort flag, merge flags [2 groups][2 alternating slots]
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmemBytes = kOffMisc + 32 + 1024;  // + slack to align the base
  // (MASKED) tile-list ring: barriers tl_full[kTLSlots] tl_empty[kTLSlots] tl_claim (+ 8 bytes
  // of padding), then the slots
  static constexpr int kOffTL = (kOffMisc + 32 + 15) / 16 * 16;
  static constexpr int kOffTLSlot = kOffTL + (2 * kTLSlots + 2) * 8;
  static constexpr int kSmemBytesMasked = kOffTLSlot + kTLSlots * kTLSlotBytes + 1024;
  // split-KV partial row: D unnormalised outputs, running max (log2 units), running sum
  static constexpr int kPartFloats = D + 4;
};

struct AttnParams {
  uint16_t* O;
  float* lse;
  const int32_t* active;
  const int32_t* counts;
  int32_t* status;
  int* ws_count;   // [kMaxGrid] merge counters (zero between launches), or null: no split
  float* ws_part;  // [kMaxGrid][2][BM][D+4] partial rows
  const uint8_t* block_mask;  // [H][nkv][nkv] token block mask (128-token blocks), or null
  const int* lpt_order;       // (block mask, with a workspace) unit order for the queue, or null
  int lpt_heads_l2;           // heads whose K/V fit in half of L2 (at least 1)
  int lpt_grid;               // CTAs of the attention launch
  int64_t o_row_stride;
  int F, N, Np, H, S_tok, nkv;
  float scale_log2;
};

// The schedule every role derives identically from the active count on the device.
struct Sched {
  int R, tiles, pairs;  // active rows (padded per frame), query tiles and tile pairs per head
  int T_full;           // items processed whole
  int C;                // KV ranges per item of the split tail (1: no split)
  int units;            // T_full + tail items * C
};

// One unit of work: a tile pair of one head over KV tiles [j0, j1).
struct Unit {
  int h, pr, j0, j1;
  int part;  // split: partial slot (tail item index * C + range), else -1
  int item;  // split: tail item index
};

__device__ __forceinline__ Sched make_sched(const AttnParams& p) {
  int A = p.counts[0];
  A = A < 0 ? 0 : (A > p.F ? p.F : A);
  Sched s;
  s.R = A * p.Np;
  s.tiles = (s.R + BM - 1) / BM;
  s.pairs = (s.tiles + 1) / 2;
  const int T = s.pairs * p.H;
  const int G = gridDim.x;
  s.T_full = T;
  s.C = 1;
  // Block-masked launches never split: their items differ in cost, so the makespan of the
  // static assignment is set by the costliest CTA rather than by the last round's tail, and a
  // split only adds the merge (measured slower on the 13 x 1560-token workload).
  if (T > 0 && p.ws_count != nullptr && p.block_mask == nullptr) {
    const int rounds = (T + G - 1) / G;
    const int tail = T - (rounds - 1) * G;
    int c = G / tail;
    if (c > kMaxSplit) c = kMaxSplit;
    if (c > p.nkv) c = p.nkv;
    if (c >= 2) {
      s.T_full = (rounds - 1) * G;
      s.C = c;
    }
  }
  s.units = s.T_full + (T - s.T_full) * s.C;
  return s;
}

__device__ __forceinline__ Unit get_unit(const Sched& s, const AttnParams& p, int w) {
  Unit u;
  int item;
  if (w < s.T_full) {
    item = w;
    u.j0 = 0;
    u.j1 = p.nkv;
    u.part = -1;
    u.item = -1;
  } else {
    const int k = w - s.T_full;
    const int ti = k / s.C, c = k - ti * s.C;
    item = s.T_full + ti;
    // 32-bit arithmetic on purpose (c <= 16, nkv < 2^24): a 64-bit divide here slowed the
    // single MMA-issuing thread by ~10% even on launches that never split
    u.j0 = (c * p.nkv) / s.C;
    u.j1 = ((c + 1) * p.nkv) / s.C;
    u.part = k;
    u.item = ti;
  }
  u.h = item / s.pairs;
  u.pr = item - u.h * s.pairs;
  return u;
}

// Token block mask (combined frame x token mask).  The valid query rows of a unit's tile pair
// form runs of consecutive tokens (one per active frame they touch), so the query blocks they
// cover are a few ranges, non-decreasing along the rows; overlapping or adjacent ranges are
// merged and, past kMaxQRanges, the last range is extended (a superset only costs skipped
// work, never correctness: every row still applies its own mask).
constexpr int kMaxQRanges = 6;
struct QRanges {
  int n;
  int lo[kMaxQRanges], hi[kMaxQRanges];
  const uint8_t* mh;  // this head's [nkv][nkv] mask
};

__device__ __forceinline__ QRanges unit_qranges(const AttnParams& p, const Sched& sc,
                                                const Unit& u) {
  QRanges q;
  q.n = 0;
  q.mh = p.block_mask + static_cast<int64_t>(u.h) * p.nkv * p.nkv;
  const int r0 = u.pr * 2 * BM;
  const int r1 = min(r0 + 2 * BM, sc.R);
  for (int r = r0; r < r1;) {
    const int a = r / p.Np;
    const int seg_end = min(r1, (a + 1) * p.Np);
    const int p_lo = r - a * p.Np, p_hi = min(seg_end - a * p.Np, p.N) - 1;
    if (p_lo <= p_hi) {
      const int t0 = p.active[a] * p.N;
      const int lo = (t0 + p_lo) / BN, hi = (t0 + p_hi) / BN;
      if (q.n > 0 && lo <= q.hi[q.n - 1] + 1) {
        q.hi[q.n - 1] = max(q.hi[q.n - 1], hi);
      } else if (q.n < kMaxQRanges) {
        q.lo[q.n] = lo;
        q.hi[q.n] = hi;
        ++q.n;
      } else {
        q.hi[q.n - 1] = max(q.hi[q.n - 1], hi);
      }
    }
    r = seg_end;
  }
  return q;
}

// First set bit at or after j in a unit's tile bitmap of nw words; nw * 32 (>= nkv) if none.
__device__ __forceinline__ int next_kept(const uint32_t* words, int j, int nw) {
  int wi = j >> 5;
  if (wi >= nw) return nw << 5;
  uint32_t x = words[wi] & (0xFFFFFFFFu << (j & 31));
  while (x == 0) {
    if (++wi >= nw) return nw << 5;
    x = words[wi];
  }
  return (wi << 5) + __ffs(x) - 1;
}

// The KV tiles a role visits for a unit: [j0, j1) unmasked, the builder's bitmap when MASKED.
template <bool MASKED>
__device__ __forceinline__ int tile_first(const Unit& u, const uint32_t* tw, int nw) {
  if constexpr (MASKED) return next_kept(tw, 0, nw);
  else return u.j0;
}
template <bool MASKED>
__device__ __forceinline__ int tile_next(const uint32_t* tw, int nw, int j) {
  if constexpr (MASKED) return next_kept(tw, j + 1, nw);
  else return j + 1;
}
template <bool MASKED>
__device__ __forceinline__ int tile_end(const Unit& u, const AttnParams& p) {
  if constexpr (MASKED) return p.nkv;
  else return u.j1;
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

// All 128 threads of one softmax warpgroup meet on an mbarrier (count 128); the wait is
// bounded like every other wait and its result is warp-uniform.
__device__ __forceinline__ bool group_sync(uint32_t bar, int& cnt, volatile int* abort) {
  mbar_arrive(bar);
  const bool ok = __all_sync(0xffffffffu, mbar_wait(bar, cnt & 1, abort, kWaitLimitNs));
  ++cnt;
  return ok;
}

// (MASKED) The tile-list ring in shared memory: slot k % kTLSlots holds the KV-tile bitmap of
// the CTA's k-th unit and, after kTLWords words, its number of set bits.
struct TLRing {
  uint32_t bar;     // shared address of tl_full[0]; tl_empty[s] follows the kTLSlots full barriers
  uint32_t* slots;  // slot 0
  __device__ __forceinline__ uint32_t full(int k) const { return bar + 8u * (k % kTLSlots); }
  __device__ __forceinline__ uint32_t empty(int k) const {
    return bar + 8u * (kTLSlots + k % kTLSlots);
  }
  // (work queue) the producer arrives once per unit, when at most kClaimAhead of the unit's KV
  // tiles are left to load: the builder may then take the next unit from the queue
  __device__ __forceinline__ uint32_t claim() const { return bar + 8u * (2 * kTLSlots); }
  __device__ __forceinline__ uint32_t* words(int k) const {
    return slots + (k % kTLSlots) * (kTLSlotBytes / 4);
  }
  __device__ __forceinline__ int parity(int k) const { return (k / kTLSlots) & 1; }
  // the unit the slot describes, or -1: the CTA has no more units
  __device__ __forceinline__ int unit(int k) const {
    return static_cast<int>(words(k)[kTLWords + 1]);
  }
};
// Arrivals that release a slot: the producer, the MMA issuer and the 256 softmax threads.
constexpr int kTLConsumers = 2 + 256;
// (work queue, at most kJitUnitsPerCta units per CTA) KV tiles of the current unit still to load
// when the next unit is claimed.  A unit is then taken from the queue only when its CTA is about
// to need it, so the queue's longest-first order decides which CTA gets which item as CTAs
// actually free up.  Claimed as soon as the previous unit started, the first two units of every
// CTA are all handed out at launch when a step has about two items per CTA: a static pairing
// (the keyframe-only step of 13 x 1560 tokens under a banded mask, items of 21 to 78 KV tiles:
// 0.200 ms; claimed this way 0.186 ms).  With many units per CTA the earlier claim is as good
// and hides the claim's latency better (21 x 3600 tokens: 1-2% faster), so it stays there.
// Three tiles are about 5 us of work, more than the claim and the tile list take to prepare.
constexpr int kClaimAhead = 3;
constexpr int kJitUnitsPerCta = 4;
__device__ __forceinline__ bool claim_jit(const AttnParams& p, const Sched& sc) {
  return p.ws_count != nullptr && sc.units <= kJitUnitsPerCta * static_cast<int>(gridDim.x);
}
// (MASKED, with a workspace) work-queue words in the workspace's counter area, which split-KV
// would use but block-masked launches never split: the next unit to hand out, and the number
// of CTAs done.  The last CTA to finish sets both back to zero.
constexpr int kQueueNext = 0, kQueueDone = 1;

// ---------------------------------------------------------------------------------------
// Tile-list builder (MASKED only; warp 2, all 32 lanes).
// ---------------------------------------------------------------------------------------
// For every unit of this CTA, in order, one ring slot receives the bitmap of the KV tiles the
// unit visits: the tiles some query block of its rows may attend to (block-masked launches
// never split, so a unit is a whole item).  The producer and the softmax warps walk this
// bitmap and the MMA issuer uses its count, so the block mask in global memory is scanned once
// per unit, with 32 lanes loading independent bytes, instead of tile by tile on the critical
// paths of the producer and the MMA issuer.
__device__ __forceinline__ void tile_list_builder(const AttnParams& p, const Sched& sc,
                                                  const TLRing& tl, volatile int* abort) {
  const int lane = threadIdx.x & 31;
  const int nw = (p.nkv + 31) >> 5;
  for (int k = 0;; ++k) {
    // At most two units in flight per CTA: the one being processed and the next.  A unit
    // taken from the queue long before it is processed would unbalance the end of the launch.
    // Unit k - 2 released also means slot k's previous unit, k - 4, was released.
    if (k >= 2 && !__all_sync(0xffffffffu, mbar_wait(tl.empty(k - 2), tl.parity(k - 2), abort,
                                                     kWaitLimitNs))) {
      if (lane == 0) flag_error(p, 7);
      return;
    }
    // With the work queue and few units per CTA, the next unit is claimed only once the
    // producer is within kClaimAhead tiles of the end of the current one.
    if (k >= 1 && claim_jit(p, sc) &&
        !__all_sync(0xffffffffu, mbar_wait(tl.claim(), (k - 1) & 1, abort, kWaitLimitNs))) {
      if (lane == 0) flag_error(p, 9);
      return;
    }
    // with a workspace: the next unit of the queue shared by all CTAs (greedy list
    // scheduling: items differ in cost under a mask); without: the static round-robin deal
    int w;
    if (p.ws_count != nullptr) {
      int t = 0;
      if (lane == 0) {
        t = atomicAdd(p.ws_count + kQueueNext, 1);
        if (p.lpt_order != nullptr && t < sc.units) t = p.lpt_order[t];
      }
      w = __shfl_sync(0xffffffffu, t, 0);
    } else {
      w = blockIdx.x + k * static_cast<int>(gridDim.x);
    }
    uint32_t* words = tl.words(k);
    if (w >= sc.units) {
      if (lane == 0) {
        words[kTLWords] = 0u;
        words[kTLWords + 1] = 0xFFFFFFFFu;
      }
      mbar_arrive(tl.full(k));
      return;
    }
    const Unit u = get_unit(sc, p, w);
    const QRanges q = unit_qranges(p, sc, u);
    int total = 0;
    for (int k0 = 0; k0 < nw; k0 += 32) {
      // bit l of acc: may some query block of the unit attend to tile (k0 + l) * 32 + lane?
      uint32_t acc = 0;
      for (int i = 0; i < q.n; ++i)
        for (int qb = q.lo[i]; qb <= q.hi[i]; ++qb) {
          const uint8_t* mrow = q.mh + static_cast<int64_t>(qb) * p.nkv;
#pragma unroll
          for (int l = 0; l < 32; ++l) {
            const int j = (k0 + l) * 32 + lane;
            if (j < p.nkv && mrow[j] != 0) acc |= 1u << l;
          }
        }
      // transpose: lane l collects word k0 + l (tiles (k0 + l) * 32 .. + 31)
      uint32_t mine = 0;
#pragma unroll
      for (int l = 0; l < 32; ++l) {
        const uint32_t bits = __ballot_sync(0xffffffffu, (acc >> l) & 1u);
        if (lane == l) mine = bits;
      }
      if (k0 + lane < nw) words[k0 + lane] = mine;
      total += __popc(mine);  // zero for words past nw: their tiles are >= nkv
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) total += __shfl_xor_sync(0xffffffffu, total, off);
    if (lane == 0) {
      words[kTLWords] = static_cast<uint32_t>(total);
      words[kTLWords + 1] = static_cast<uint32_t>(w);
    }
    mbar_arrive(tl.full(k));  // every lane (count 32) releases its own stores
  }
}

// ---------------------------------------------------------------------------------------
// TMA producer (one thread).
// ---------------------------------------------------------------------------------------
template <int D, bool MASKED>
__device__ __forceinline__ void producer(const CUtensorMap* tmQ, const CUtensorMap* tmQ128,
                                         const CUtensorMap* tmK,
                                         const CUtensorMap* tmV, const AttnParams& p,
                                         const Sched& sc, uint32_t sQ0, uint32_t sKV0,
                                         uint32_t bar0, const TLRing& tl, volatile int* abort) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const int nw = (p.nkv + 31) >> 5;
  int q_cnt[2] = {0, 0};
  int it = 0;
  // L2 priorities: a query tile is read once, a head's K/V by every unit of that head.  Marking
  // the query loads evict-first and the K/V loads evict-last cut the DRAM reads of an
  // all-active 33 x 3600-token launch from 8.6-10.8 GB to 7.1-9.4 GB (same box, in alternation;
  // K/V of one head is 61 MB and is swept once per round of work items), at the same speed.
  const uint64_t pol_q = l2_policy_evict_first();
  const uint64_t pol_kv = l2_policy_evict_last();
  for (int k = 0;; ++k) {  // k: units so far (MASKED: tile-list ring position)
    int w;
    const uint32_t* tw = nullptr;
    if constexpr (MASKED) {
      if (!mbar_wait(tl.full(k), tl.parity(k), abort, kWaitLimitNs)) {
        flag_error(p, 0);
        goto drain;
      }
      w = tl.unit(k);
      if (w < 0) break;
      tw = tl.words(k);
    } else {
      w = blockIdx.x + k * static_cast<int>(gridDim.x);
      if (w >= sc.units) break;
    }
    const Unit u = get_unit(sc, p, w);
    for (int X = 0; X < 2; ++X) {
      const int t = 2 * u.pr + X;
      if (t >= sc.tiles) break;
      if (!mbar_wait(bar(C::kBarQEmpty + X), (q_cnt[X] & 1) ^ 1, abort, kWaitLimitNs)) {
        flag_error(p, 0);
        goto drain;
      }
      mbar_arrive_expect_tx(bar(C::kBarQFull + X), C::kTileBytes);
      const uint32_t dst = sQ0 + X * C::kTileBytes;
      const int r0 = t * BM;
      const int a0 = r0 / p.Np;
      if (a0 == (min(r0 + BM, sc.R) - 1) / p.Np) {
        // every row of the tile in one frame: one 128-row box per half (rows past the frame or
        // the active list read the following tokens, or zeros past the sequence; they are
        // never stored)
        const int tok = p.active[a0] * p.N + (r0 - a0 * p.Np);
#pragma unroll
        for (int hb = 0; hb < C::kHalves; ++hb)
          tma_load_3d_hint(dst + hb * C::kHalfBytes, tmQ128, bar(C::kBarQFull + X), hb * 64,
                           u.h, tok, pol_q);
      } else {
        // a tile across frames: gathered in boxes of 8 rows (frames are padded to 8 rows)
        int tok[BM / 8];
#pragma unroll
        for (int b = 0; b < BM / 8; ++b) {
          const int r = r0 + b * 8;
          const int a = r / p.Np;
          tok[b] = r < sc.R ? p.active[a] * p.N + (r - a * p.Np)
                            : p.S_tok;  // past the active list: out of bounds, zero filled
        }
#pragma unroll
        for (int b = 0; b < BM / 8; ++b)
#pragma unroll
          for (int hb = 0; hb < C::kHalves; ++hb)
            tma_load_3d_hint(dst + hb * C::kHalfBytes + b * 1024, tmQ, bar(C::kBarQFull + X),
                             hb * 64, u.h, tok[b], pol_q);
      }
      ++q_cnt[X];
    }
    // (MASKED, work queue) tiles of this unit still to load; the claim signal goes out once
    int left = 0;
    bool claim_due = false;
    if constexpr (MASKED) {
      left = static_cast<int>(tw[kTLWords]);
      claim_due = claim_jit(p, sc);
      if (claim_due && left <= kClaimAhead) {
        mbar_arrive(tl.claim());
        claim_due = false;
      }
    }
#pragma unroll 1
    for (int j = tile_first<MASKED>(u, tw, nw); j < tile_end<MASKED>(u, p);
         j = tile_next<MASKED>(tw, nw, j)) {
      if constexpr (MASKED) {
        if (claim_due && --left <= kClaimAhead) {
          mbar_arrive(tl.claim());
          claim_due = false;
        }
      }
#pragma unroll
      for (int kv = 0; kv < 2; ++kv) {
        const int s = it % C::kSlots, n = it / C::kSlots;
        if (!mbar_wait(bar(C::kBarKVEmpty + s), (n & 1) ^ 1, abort, kWaitLimitNs)) {
          flag_error(p, 1);
          goto drain;
        }
        mbar_arrive_expect_tx(bar(C::kBarKVFull + s), C::kTileBytes);
        const uint32_t dst = sKV0 + s * C::kTileBytes;
#pragma unroll
        for (int hb = 0; hb < C::kHalves; ++hb)
          tma_load_3d_hint(dst + hb * C::kHalfBytes, kv ? tmV : tmK, bar(C::kBarKVFull + s),
                           hb * 64, u.h, j * BN, pol_kv);
        ++it;
      }
    }
    if constexpr (MASKED) mbar_arrive(tl.empty(k));
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
// Descriptors are built once per buffer; a K step only adds its byte offset / 16 to the start
// address field (bits 0-13), which cannot carry: every shared address is below 256 KB.  (The
// single issuing thread is on the critical path: rebuilding descriptors per MMA cost ~2-4%.)
template <int D>
__device__ __forceinline__ void mma_qk(uint32_t tS, uint64_t dQ, uint64_t dK) {
  constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, 0, 0);
#pragma unroll
  for (int k = 0; k < D / 16; ++k) {
    const uint64_t off = ((k >> 2) * (BM * 128) + (k & 3) * 32) >> 4;
    tc_mma_ss(tS, dQ + off, dK + off, idesc, k > 0);
  }
}

template <int D>
__device__ __forceinline__ void mma_pv(uint32_t tO, uint32_t tP, uint64_t dV, uint32_t acc) {
  constexpr uint32_t idesc = idesc_bf16_f32(BM, D, 0, 1);
#pragma unroll
  for (int k = 0; k < BN / 16; ++k)
    tc_mma_ts(tO, tP + k * 8, dV + ((k * 2048) >> 4), idesc, (acc | k) != 0);
}

template <int D, bool MASKED>
__device__ __forceinline__ void mma_issuer(const AttnParams& p, const Sched& sc, uint32_t tmem,
                                           uint32_t sQ0, uint32_t sKV0, uint32_t bar0,
                                           const TLRing& tl, volatile int* abort) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const uint32_t tS[2] = {tmem, tmem + 128};
  const uint32_t tO[2] = {tmem + 256, tmem + 384};
  const uint64_t dQ[2] = {smem_desc_sw128(sQ0, 16, 1024),
                          smem_desc_sw128(sQ0 + C::kTileBytes, 16, 1024)};
  // K operand: K-major; V operand: MN-major with the two 64-column halves 16 KB apart
  auto dK = [&](int s) { return smem_desc_sw128(sKV0 + s * C::kTileBytes, 16, 1024); };
  auto dV = [&](int s) { return smem_desc_sw128(sKV0 + s * C::kTileBytes, BN * 128, 1024); };
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
  for (int k = 0;; ++k) {  // k: units so far (MASKED: tile-list ring position)
    int w;
    const uint32_t* tw = nullptr;
    if constexpr (MASKED) {
      if (!mbar_wait(tl.full(k), tl.parity(k), abort, kWaitLimitNs)) goto fail;
      w = tl.unit(k);
      if (w < 0) break;
      tw = tl.words(k);
    } else {
      w = blockIdx.x + k * static_cast<int>(gridDim.x);
      if (w >= sc.units) break;
    }
    const Unit u = get_unit(sc, p, w);
    const bool hasB = 2 * u.pr + 1 < sc.tiles;
    // number of KV tiles of the unit: j1 - j0, or (MASKED) the set bits of the builder's
    // bitmap (the issuer needs only the count; the producer walks the bits)
    const int ntiles = MASKED ? static_cast<int>(tw[kTLWords]) : u.j1 - u.j0;
    if (!mbar_wait(bar(C::kBarQFull + 0), q_cnt[0] & 1, abort, kWaitLimitNs)) goto fail;
    ++q_cnt[0];
    if (hasB) {
      if (!mbar_wait(bar(C::kBarQFull + 1), q_cnt[1] & 1, abort, kWaitLimitNs)) goto fail;
      ++q_cnt[1];
    }
    tc_fence_after();
    if (MASKED && ntiles == 0) {
      // no allowed key block: release the queries.  No output barrier is committed: the
      // softmax warps see the same empty tile list and write their result without waiting
      // (a commit here could run two phases ahead of them).
      mbar_arrive(tl.empty(k));
      tc_commit(bar(C::kBarQEmpty + 0));
      if (hasB) tc_commit(bar(C::kBarQEmpty + 1));
      continue;
    }
    int sK, sV;
    if (!next_slot(sK)) goto fail;
    mma_qk<D>(tS[0], dQ[0], dK(sK));
    tc_commit(bar(C::kBarSFull + 0));
    if (hasB) {
      mma_qk<D>(tS[1], dQ[1], dK(sK));
      tc_commit(bar(C::kBarSFull + 1));
    }
    tc_commit(bar(C::kBarKVEmpty + sK));
    if (!next_slot(sV)) goto fail;
    if (!wait_p(0)) goto fail;
    mma_pv<D>(tO[0], tS[0], dV(sV), 0);
    int nj = 1;  // tiles issued so far
#pragma unroll 1
    for (int j = 0;; ++j) {
      if (j + 1 >= ntiles) break;
      ++nj;
      if (!next_slot(sK)) goto fail;
      mma_qk<D>(tS[0], dQ[0], dK(sK));
      tc_commit(bar(C::kBarSFull + 0));
      if (hasB) {
        if (!wait_p(1)) goto fail;
        mma_pv<D>(tO[1], tS[1], dV(sV), j > 0);
      }
      tc_commit(bar(C::kBarKVEmpty + sV));
      if (hasB) {
        mma_qk<D>(tS[1], dQ[1], dK(sK));
        tc_commit(bar(C::kBarSFull + 1));
      }
      tc_commit(bar(C::kBarKVEmpty + sK));
      if (!next_slot(sV)) goto fail;
      if (!wait_p(0)) goto fail;
      mma_pv<D>(tO[0], tS[0], dV(sV), 1);
    }
    if constexpr (MASKED) mbar_arrive(tl.empty(k));
    tc_commit(bar(C::kBarODone + 0));
    tc_commit(bar(C::kBarQEmpty + 0));
    if (hasB) {
      if (!wait_p(1)) goto fail;
      mma_pv<D>(tO[1], tS[1], dV(sV), nj > 1);
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
__device__ __forceinline__ void store_row_bf16(uint16_t* orow, const float* o, float scale) {
  uint4* dst = reinterpret_cast<uint4*>(orow);
#pragma unroll
  for (int q = 0; q < D / 8; ++q) {
    uint4 v;
    v.x = pack_bf16x2(o[8 * q + 0] * scale, o[8 * q + 1] * scale);
    v.y = pack_bf16x2(o[8 * q + 2] * scale, o[8 * q + 3] * scale);
    v.z = pack_bf16x2(o[8 * q + 4] * scale, o[8 * q + 5] * scale);
    v.w = pack_bf16x2(o[8 * q + 6] * scale, o[8 * q + 7] * scale);
    dst[q] = v;
  }
}

template <int D, bool MASKED>
__device__ __forceinline__ void softmax_group(const AttnParams& p, const Sched& sc, int X,
                                              uint32_t tmem, uint32_t bar0, const TLRing& tl,
                                              volatile int* abort, volatile int* merge_flag) {
  using C = Cfg<D>;
  auto bar = [&](int i) { return bar0 + 8u * i; };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3;  // TMEM lanes this warp may access
  const int row = quarter * 32 + lane;
  const uint32_t lane_base = static_cast<uint32_t>(quarter * 32) << 16;
  const uint32_t tS = tmem + lane_base + X * 128;
  const uint32_t tO = tmem + lane_base + 256 + X * 128;
  const float sl2 = p.scale_log2;
  const int nw = (p.nkv + 31) >> 5;
  int s_cnt = 0, o_cnt = 0, g_cnt = 0, split_cnt = 0;
  for (int k = 0;; ++k) {  // k: units so far (MASKED: tile-list ring position)
    int w;
    const uint32_t* tw = nullptr;
    if constexpr (MASKED) {
      // every softmax thread takes every unit's slot, also when its tile is absent, so the
      // slot's release count is the same for all units
      if (!__all_sync(0xffffffffu, mbar_wait(tl.full(k), tl.parity(k), abort, kWaitLimitNs))) {
        flag_error(p, 8);
        return;
      }
      w = tl.unit(k);
      if (w < 0) break;
      tw = tl.words(k);
    } else {
      w = blockIdx.x + k * static_cast<int>(gridDim.x);
      if (w >= sc.units) break;
    }
    const Unit u = get_unit(sc, p, w);
    const int t = 2 * u.pr + X;
    if (t >= sc.tiles) {
      if constexpr (MASKED) mbar_arrive(tl.empty(k));
      continue;
    }
    const bool empty_unit = MASKED && tw[kTLWords] == 0u;
    float m = -INFINITY, l = 0.f;
    // this row's query block (MASKED): rows past the active list or in frame padding are
    // never stored and need no mask
    const uint8_t* mrow = nullptr;
    if constexpr (MASKED) {
      const int r = t * BM + row;
      if (r < sc.R) {
        const int a = r / p.Np, pp = r - a * p.Np;
        if (pp < p.N) {
          const int qb = (p.active[a] * p.N + pp) / BN;
          mrow = p.block_mask + (static_cast<int64_t>(u.h) * p.nkv + qb) * p.nkv;
        }
      }
    }
    // (MASKED) this row's mask entry for the tile, loaded one tile ahead of its use
    int j = tile_first<MASKED>(u, tw, nw);
    const int j_end = tile_end<MASKED>(u, p);
    uint32_t mk = 1u;
    if constexpr (MASKED) mk = (mrow != nullptr && j < j_end) ? mrow[j] : 1u;
    bool first = true;
#pragma unroll 1
    while (j < j_end) {
      const int jn = tile_next<MASKED>(tw, nw, j);
      uint32_t mk_next = 1u;
      if constexpr (MASKED) mk_next = (mrow != nullptr && jn < j_end) ? mrow[jn] : 1u;
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
      // (MASKED) a tile this row may not see leaves its max alone (and gets p = 0 below)
      const float m_new = fmaxf(m, (MASKED && mk == 0u) ? -INFINITY : mx * sl2);
      const bool need = m_new > m + kRescaleLog2;
      const bool rescale = __any_sync(0xffffffffu, need);
      float fac = 1.f;
      if (rescale) {
        // (MASKED) a row that has seen only excluded keys has m = m_new = -inf while another
        // row of its warp asked for the rescale: factor 1, not 2^(-inf + inf)
        fac = (MASKED && m == m_new) ? 1.f : ex2_approx(m - m_new);
        l *= fac;
        m = m_new;
      }
      // p = 2^(s*scale*log2(e) - m) with packed fp32 pairs for the scale/subtract and the
      // row sum (8 independent sum chains in 4 packed accumulators)
      // (MASKED) while every key seen so far was excluded, m is -inf: use 0 so p = 2^-inf = 0;
      // for a tile the row may not see, an offset of -inf gives p = 0 for every key (s is
      // finite or -inf, so s * scale - inf is -inf, never NaN)
      const float nm = (MASKED && mk == 0u) ? -INFINITY : (MASKED && m == -INFINITY) ? 0.f : -m;
      const uint64_t sl2x2 = f2_pack(sl2, sl2), nmx2 = f2_pack(nm, nm);
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
        const uint64_t t2 = fadd2(fadd2(l4[0], l4[1]), fadd2(l4[2], l4[3]));
        float a, b;
        f2_unpack(t2, a, b);
        l += a + b;
      }
      // O was last written by the previous tile's PV, which completed before S(j) was
      // signalled; at the unit's first tile it holds nothing yet
      if (rescale && (MASKED ? !first : j > u.j0)) {
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
      first = false;
      j = jn;
      mk = mk_next;
    }
    if constexpr (MASKED) mbar_arrive(tl.empty(k));
    // epilogue (an empty unit has no accumulator to wait for: l == 0 writes zeros)
    if (!empty_unit) {
      if (!__all_sync(0xffffffffu,
                      mbar_wait(bar(C::kBarODone + X), o_cnt & 1, abort, kWaitLimitNs))) {
        flag_error(p, 4);
        return;
      }
      ++o_cnt;
      tc_fence_after();
    }
    const int r = t * BM + row;
    bool valid = r < sc.R;
    int64_t token = 0;
    if (valid) {
      const int a = r / p.Np, pp = r - a * p.Np;
      valid = pp < p.N;
      token = static_cast<int64_t>(p.active[a]) * p.N + pp;
    }
    uint16_t* orow = p.O + token * p.o_row_stride + static_cast<int64_t>(u.h) * D;
    if (u.part < 0) {
      // whole item: O / l -> bf16.  A row that may attend to no key gets O = 0 and LSE = -inf;
      // its accumulator may never have been written in this unit, so zeros are stored, not
      // 0 * accumulator.
      const bool none = MASKED && l == 0.f;
      const float inv_l = none ? 0.f : 1.0f / l;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + c * 32, o);
        tmem_wait_ld();
        if (none) {
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = 0u;
        }
        if (valid) store_row_bf16<32>(orow + c * 32, reinterpret_cast<const float*>(o), inv_l);
      }
      if (valid && p.lse)
        p.lse[static_cast<int64_t>(u.h) * p.S_tok + token] =
            (MASKED && l == 0.f) ? -INFINITY : (m + __log2f(l)) * 0.69314718055994531f;
      continue;
    }
    // split item: publish this KV range's partial row, then the last range to finish merges
    float* part = p.ws_part + ((static_cast<int64_t>(u.part) * 2 + X) * BM + row) * C::kPartFloats;
#pragma unroll 1
    for (int c = 0; c < D / 32; ++c) {
      uint32_t o[32];
      tmem_ld32(tO + c * 32, o);
      tmem_wait_ld();
      float4* dst = reinterpret_cast<float4*>(part + c * 32);
      const bool none = MASKED && l == 0.f;  // no allowed key in this range: O is not written
#pragma unroll
      for (int q = 0; q < 8; ++q)
        __stcg(dst + q, none ? make_float4(0.f, 0.f, 0.f, 0.f)
                             : make_float4(__uint_as_float(o[4 * q]), __uint_as_float(o[4 * q + 1]),
                                           __uint_as_float(o[4 * q + 2]),
                                           __uint_as_float(o[4 * q + 3])));
    }
    __stcg(reinterpret_cast<float4*>(part + D), make_float4(m, l, 0.f, 0.f));
    __threadfence();
    // two flag slots alternate, so a slot is rewritten only after every thread read it
    volatile int* flag = merge_flag + (split_cnt & 1);
    ++split_cnt;
    if (!group_sync(bar(C::kBarGroup + X), g_cnt, abort)) {  // every row is published
      flag_error(p, 5);
      return;
    }
    if (row == 0) {
      const int old = atomicAdd(p.ws_count + 2 * u.item + X, 1);
      *flag = (old == sc.C - 1);
    }
    if (!group_sync(bar(C::kBarGroup + X), g_cnt, abort)) {  // the flag is visible
      flag_error(p, 6);
      return;
    }
    if (*flag == 0) continue;
    __threadfence();
    if (valid) {
      const float* base =
          p.ws_part + ((static_cast<int64_t>(u.item) * sc.C * 2 + X) * BM + row) * C::kPartFloats;
      const int64_t stride = static_cast<int64_t>(2) * BM * C::kPartFloats;  // next range
      // O = sum_c 2^(m_c - M) O_c / sum_c 2^(m_c - M) l_c, M = max_c m_c
      float M = -INFINITY;
      for (int c = 0; c < sc.C; ++c) M = fmaxf(M, __ldcg(base + c * stride + D));
      float L = 0.f;
      for (int c = 0; c < sc.C; ++c) {
        const float2 ml = __ldcg(reinterpret_cast<const float2*>(base + c * stride + D));
        if (!(MASKED && M == -INFINITY)) L += ml.y * ex2_approx(ml.x - M);
      }
      const bool empty = MASKED && M == -INFINITY;  // no range saw an allowed key
      const float inv_L = empty ? 0.f : 1.0f / L;
#pragma unroll 1
      for (int cc = 0; cc < D / 32; ++cc) {
        float acc[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) acc[e] = 0.f;
        for (int c = 0; c < sc.C; ++c) {
          const float* pc = base + c * stride;
          const float wgt = empty ? 0.f : ex2_approx(__ldcg(pc + D) - M);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 v = __ldcg(reinterpret_cast<const float4*>(pc + cc * 32) + q);
            acc[4 * q] = fmaf(v.x, wgt, acc[4 * q]);
            acc[4 * q + 1] = fmaf(v.y, wgt, acc[4 * q + 1]);
            acc[4 * q + 2] = fmaf(v.z, wgt, acc[4 * q + 2]);
            acc[4 * q + 3] = fmaf(v.w, wgt, acc[4 * q + 3]);
          }
        }
        store_row_bf16<32>(orow + cc * 32, acc, inv_L);
      }
      if (p.lse)
        p.lse[static_cast<int64_t>(u.h) * p.S_tok + token] =
            empty ? -INFINITY : (M + __log2f(L)) * 0.69314718055994531f;
    }
    if (row == 0) p.ws_count[2 * u.item + X] = 0;  // ready for the next launch
  }
}

template <int D, bool MASKED>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQ128,
                const __grid_constant__ CUtensorMap tmK,
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
  volatile int* merge_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 8);  // [2][2]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int X = 0; X < 2; ++X) {
      mbar_init(bar0 + 8 * (C::kBarQFull + X), 1);
      mbar_init(bar0 + 8 * (C::kBarQEmpty + X), 1);
      mbar_init(bar0 + 8 * (C::kBarSFull + X), 1);
      mbar_init(bar0 + 8 * (C::kBarPFull + X), 128);
      mbar_init(bar0 + 8 * (C::kBarODone + X), 1);
      mbar_init(bar0 + 8 * (C::kBarGroup + X), 128);
      merge_flag[2 * X] = 0;
      merge_flag[2 * X + 1] = 0;
    }
    for (int s = 0; s < C::kSlots; ++s) {
      mbar_init(bar0 + 8 * (C::kBarKVFull + s), 1);
      mbar_init(bar0 + 8 * (C::kBarKVEmpty + s), 1);
    }
    mbar_init(bar0 + 8 * C::kBarDrain, 1);
    if constexpr (MASKED) {
      for (int s = 0; s < kTLSlots; ++s) {
        mbar_init(sbase + C::kOffTL + 8 * s, 32);
        mbar_init(sbase + C::kOffTL + 8 * (kTLSlots + s), kTLConsumers);
      }
      mbar_init(sbase + C::kOffTL + 8 * (2 * kTLSlots), 1);
    }
    *abort = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmQ128);
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
  const Sched sc = make_sched(p);
  TLRing tl{};
  if constexpr (MASKED)
    tl = TLRing{sbase + C::kOffTL, reinterpret_cast<uint32_t*>(smem + C::kOffTLSlot)};

  // Every warp of warpgroup 0 gives registers back before any softmax warp asks for more,
  // so the increase below always finds them.
  if (warp < 4) {
    reg_dealloc<kRegsControl>();
    if (warp == 0) {
      if (lane == 0) producer<D, MASKED>(&tmQ, &tmQ128, &tmK, &tmV, p, sc, sQ0, sKV0, bar0, tl, abort);
      __syncwarp();
    } else if (warp == 1) {
      if (lane == 0) mma_issuer<D, MASKED>(p, sc, tmem, sQ0, sKV0, bar0, tl, abort);
      __syncwarp();
    } else if (MASKED && warp == 2) {
      tile_list_builder(p, sc, tl, abort);
    }
  } else {
    reg_alloc<kRegsSoftmax>();
    const int X = (warp - 4) >> 2;
    softmax_group<D, MASKED>(p, sc, X, tmem, bar0, tl, abort, merge_flag + 2 * X);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if constexpr (MASKED) {
    // every CTA that reaches this point has taken its last unit from the queue; the last one
    // to arrive leaves the queue words at zero for the next launch
    if (threadIdx.x == 0 && p.ws_count != nullptr) {
      __threadfence();
      if (atomicAdd(p.ws_count + kQueueDone, 1) == static_cast<int>(gridDim.x) - 1) {
        p.ws_count[kQueueNext] = 0;
        p.ws_count[kQueueDone] = 0;
      }
    }
  }
}

// ---------------------------------------------------------------------------------------
// Longest-first order of block-masked work items (one small launch before the attention
// kernel).  Under a mask, items differ in cost (the number of KV tiles their tile pair may
// see); handing them out from the work queue longest first within each group of heads (LPT
// list scheduling) keeps the CTAs' finishing times close where a round-robin deal or the
// natural order can leave costly items for the end (a causal block mask on 13 x 1560 tokens:
// 1.10 ms dealt round-robin, 0.83 ms longest first).
//
// Groups of consecutive heads (item = head * pairs + pair): the queue hands out the groups one
// after the other, so the CTAs that run together work on the heads of one group.  A group has
// as many heads as fit their K/V in half of L2, and at least enough for six items per CTA
// (from the active count, so on the device): one global order by cost spread the CTAs over
// all 40 heads of a 21 x 3600-token workload (39 MB of K/V per head, 129 MB of L2) and was 5%
// slower than no order at all, while one head per group left 13 x 1560 tokens (80 items per
// head, 152 CTAs) 19% slower than the global order, because each head's costly items started
// late.
__device__ __forceinline__ int lpt_group_heads(const AttnParams& p, const Sched& sc) {
  const int need = (4 * p.lpt_grid + sc.pairs - 1) / max(sc.pairs, 1);
  return min(p.H, max(p.lpt_heads_l2, need));
}
//
// Each CTA covers kPrepassItems items of one head, one warp per item: the item's cost is the
// number of set bits of the bitmap the builder will write, found with each lane loading 32
// independent mask bytes per query block.  The CTA that completes a group (a counter per group
// in the workspace, reset by that CTA) sorts the group by decreasing cost with a counting sort.
// The order among equal costs is arbitrary, which changes no result (every item is computed
// the same way by whichever CTA takes it) and, within an L2-sized group, no locality.
constexpr int kPrepassItems = 8;       // items (warps) per CTA
constexpr int kPrepassThreads = 32 * kPrepassItems;
constexpr int kQueueGroup0 = 2;        // first per-group counter word
constexpr int kMaxLptGroups = kMaxGrid - kQueueGroup0;
constexpr int kCostBins = kTLMaxTiles + 1;
constexpr int kBinsPerThread = (kCostBins + kPrepassThreads - 1) / kPrepassThreads;

__global__ void __launch_bounds__(kPrepassThreads)
    lpt_prepass_kernel(const AttnParams p, int* cost, int* order, int ctas_per_head) {
  __shared__ int start[kBinsPerThread * kPrepassThreads];  // bin b holds cost kTLMaxTiles - b
  __shared__ int warp_sum[kPrepassThreads / 32];
  __shared__ int last;
  const Sched sc = make_sched(p);  // a block-masked launch: no split, so units are items
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int h = blockIdx.x / ctas_per_head, part = blockIdx.x % ctas_per_head;
  const int ctas_head = (sc.pairs + kPrepassItems - 1) / kPrepassItems;
  if (sc.pairs == 0 || part >= ctas_head) return;  // CTA-uniform: no item of this head
  const int gh = lpt_group_heads(p, sc);
  const int group = h / gh;
  const int base = group * gh * sc.pairs;                  // the group's first item
  const int heads = min(gh, p.H - group * gh);
  const int n = heads * sc.pairs;                          // the group's items
  const int item = (h - group * gh) * sc.pairs + part * kPrepassItems + wid;  // in the group
  if (part * kPrepassItems + wid < sc.pairs) {
    const Unit u = get_unit(sc, p, base + item);
    const QRanges q = unit_qranges(p, sc, u);
    const int nw = (p.nkv + 31) >> 5;
    int total = 0;
    for (int k0 = 0; k0 < nw; k0 += 32) {
      uint32_t acc = 0;  // bit l: tile (k0 + l) * 32 + lane allowed
      for (int i = 0; i < q.n; ++i)
        for (int qb = q.lo[i]; qb <= q.hi[i]; ++qb) {
          const uint8_t* mrow = q.mh + static_cast<int64_t>(qb) * p.nkv;
#pragma unroll
          for (int l = 0; l < 32; ++l) {
            const int j = (k0 + l) * 32 + lane;
            if (j < p.nkv && mrow[j] != 0) acc |= 1u << l;
          }
        }
      total += __popc(acc);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) total += __shfl_xor_sync(0xffffffffu, total, off);
    if (lane == 0) {
      cost[base + item] = total;
      __threadfence();  // visible to the CTA that sorts the group
    }
  }
  // the CTA that completes the group sorts it
  const int ctas = heads * ctas_head;
  __syncthreads();
  if (tid == 0) {
    int* counter = p.ws_count + kQueueGroup0 + group;
    last = atomicAdd(counter, 1) == ctas - 1;
    if (last) *counter = 0;  // ready for the next launch
  }
  __syncthreads();
  if (!last) return;
  __threadfence();
  for (int i = tid; i < kBinsPerThread * kPrepassThreads; i += kPrepassThreads) start[i] = 0;
  __syncthreads();
  for (int i = tid; i < n; i += kPrepassThreads)
    atomicAdd(&start[kTLMaxTiles - __ldcg(cost + base + i)], 1);
  __syncthreads();
  // exclusive prefix sum over the bins: kBinsPerThread consecutive bins per thread, then a
  // block-wide scan of the per-thread sums
  int own[kBinsPerThread];
  int sum = 0;
#pragma unroll
  for (int b = 0; b < kBinsPerThread; ++b) {
    own[b] = start[tid * kBinsPerThread + b];
    sum += own[b];
  }
  int incl = sum;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += t;
  }
  if (lane == 31) warp_sum[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int v = lane < kPrepassThreads / 32 ? warp_sum[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, v, off);
      if (lane >= off) v += t;
    }
    if (lane < kPrepassThreads / 32) warp_sum[lane] = v;  // inclusive, over warps
  }
  __syncthreads();
  int run = incl - sum + (wid > 0 ? warp_sum[wid - 1] : 0);
#pragma unroll
  for (int b = 0; b < kBinsPerThread; ++b) {
    start[tid * kBinsPerThread + b] = run;
    run += own[b];
  }
  __syncthreads();
  for (int i = tid; i < n; i += kPrepassThreads)
    order[base + atomicAdd(&start[kTLMaxTiles - __ldcg(cost + base + i)], 1)] = base + i;
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

// Workspace layout: [kMaxGrid] int counters, then (256-byte aligned) the partial rows.
// Unmasked launches use the counters to merge split-KV ranges and the rest for the partials.
// Block-masked launches (which never split) use counters 0 and 1 for the work queue, 2.. for
// the longest-first pre-pass's groups, and the partial-row area for the items' costs and order.
constexpr int64_t kCountBytes = kMaxGrid * 4;
int64_t workspace_bytes(int d, int grid) {
  return kCountBytes + static_cast<int64_t>(grid) * 2 * BM * (d + 4) * 4;
}

template <int D, bool MASKED>
rf_status launch(const CUtensorMap& q, const CUtensorMap& q128, const CUtensorMap& k,
                 const CUtensorMap& v,
                 const AttnParams& p, int grid, const DeviceInfo& di, cudaStream_t stream) {
  using C = Cfg<D>;
  constexpr int smem = MASKED ? C::kSmemBytesMasked : C::kSmemBytes;
  static bool attr_set[64] = {};
  if (smem > di.max_smem_optin) return fail(RF_ERR_UNSUPPORTED, "shared memory");
  if (!attr_set[di.device]) {
    if (cudaError_t e = cudaFuncSetAttribute(
            attn_kernel<D, MASKED>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem))
      return fail(RF_ERR_CUDA, "cudaFuncSetAttribute(attn_kernel)", e);
    attr_set[di.device] = true;
  }
  attn_kernel<D, MASKED><<<grid, kThreads, smem, stream>>>(q, q128, k, v, p);
  return launch_status("attn_kernel launch");
}

// Scratch for rf_attn_noalloc: a file-scope device array, so that callers who cannot allocate
// device memory still get split-KV.  Sized for head dim 128 on up to 160 SMs (20.6 MiB); every
// GPU that loads this library holds it until the process exits.
constexpr int kNoAllocMaxGrid = 160;
constexpr int64_t kNoAllocScratchBytes =
    kCountBytes + static_cast<int64_t>(kNoAllocMaxGrid) * 2 * BM * (128 + 4) * 4;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
std::mutex g_noalloc_mu;
void* g_noalloc_addr[64] = {};  // device address of the array, per device ordinal

}  // namespace
}  // namespace rf

using namespace rf;

extern "C" int64_t rf_attn_workspace_bytes(int d) {
  if (d != 64 && d != 128) return -1;
  DeviceInfo di;
  if (current_device_info(&di) != RF_OK) return -1;
  const int grid = di.sm_count < kMaxGrid ? di.sm_count : kMaxGrid;
  return workspace_bytes(d, grid);
}

namespace {
// Every host-checkable argument error of an attention call, before anything is enqueued.
rf_status check_attn_args(const void* d_O, const void* d_Q, const void* d_K, const void* d_V,
                          int64_t qkv_row_stride, int64_t o_row_stride, int F, int N, int H,
                          int d, const int32_t* d_active, const int32_t* d_counts,
                          float softmax_scale, const uint8_t* d_block_mask,
                          const void* d_workspace, int64_t workspace_bytes_given,
                          DeviceInfo* di) {
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
  if (d_block_mask && (S_tok + BN - 1) / BN > kTLMaxTiles)
    return fail(RF_ERR_UNSUPPORTED, "block mask: more than 4096 key blocks of 128 tokens");
  if (d_workspace) {
    if (workspace_bytes_given < 0) return RF_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(d_workspace) & 255) return RF_ERR_MISALIGNED;
  }
  if (rf_status st = current_device_info(di)) return st;
  if (di->cc_major != 10 || di->cc_minor != 3) return fail(RF_ERR_UNSUPPORTED, "needs sm_103");
  return RF_OK;
}

rf_status attn_impl(void* d_O, float* d_lse, const void* d_Q, const void* d_K, const void* d_V,
                    int64_t qkv_row_stride, int64_t o_row_stride, int F, int N, int H, int d,
                    const int32_t* d_active, const int32_t* d_counts, float softmax_scale,
                    const uint8_t* d_block_mask, void* d_workspace, int64_t workspace_bytes_given,
                    int32_t* d_status, rf_stream_t stream) {
  DeviceInfo di;
  if (rf_status st = check_attn_args(d_O, d_Q, d_K, d_V, qkv_row_stride, o_row_stride, F, N, H,
                                     d, d_active, d_counts, softmax_scale, d_block_mask,
                                     d_workspace, workspace_bytes_given, &di))
    return st;
  const int64_t S_tok = static_cast<int64_t>(F) * N;
  const int64_t Np = (static_cast<int64_t>(N) + 7) / 8 * 8;

  CUtensorMap mq, mq128, mk, mv;
  if (rf_status st = make_map(&mq, d_Q, d, H, static_cast<int>(S_tok), qkv_row_stride, 8)) return st;
  if (rf_status st = make_map(&mq128, d_Q, d, H, static_cast<int>(S_tok), qkv_row_stride, BM))
    return st;
  if (rf_status st = make_map(&mk, d_K, d, H, static_cast<int>(S_tok), qkv_row_stride, BN)) return st;
  if (rf_status st = make_map(&mv, d_V, d, H, static_cast<int>(S_tok), qkv_row_stride, BN)) return st;

  // Persistent grid: one CTA per SM, fewer if the largest possible active set has fewer items.
  const int64_t rows = static_cast<int64_t>(F) * Np;
  const int64_t tiles = (rows + BM - 1) / BM;
  const int64_t max_items = ((tiles + 1) / 2) * H;
  int grid = di.sm_count < kMaxGrid ? di.sm_count : kMaxGrid;
  const bool split = d_workspace != nullptr && workspace_bytes_given >= workspace_bytes(d, grid);
  // without split-KV there is no use for more CTAs than items
  if (!split && max_items < grid) grid = static_cast<int>(max_items);
  if (grid < 1) grid = 1;

  AttnParams p;
  p.O = static_cast<uint16_t*>(d_O);
  p.lse = d_lse;
  p.active = d_active;
  p.counts = d_counts;
  p.status = d_status;
  p.ws_count = split ? static_cast<int*>(d_workspace) : nullptr;
  p.ws_part = split ? reinterpret_cast<float*>(static_cast<char*>(d_workspace) + kCountBytes)
                    : nullptr;
  p.block_mask = d_block_mask;
  p.lpt_order = nullptr;
  p.lpt_heads_l2 = 1;
  p.lpt_grid = 0;
  p.o_row_stride = o_row_stride;
  p.F = F;
  p.N = N;
  p.Np = static_cast<int>(Np);
  p.H = H;
  p.S_tok = static_cast<int>(S_tok);
  p.nkv = static_cast<int>((S_tok + BN - 1) / BN);
  p.scale_log2 = static_cast<float>(static_cast<double>(softmax_scale) * 1.4426950408889634);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (d_block_mask) {
    // With a workspace: costs and the longest-first order of the items in its partial-row
    // area (unused by block-masked launches, which never split), when it holds them.
    // Heads whose K/V fit in half of L2; the kernel makes groups of at least that many heads.
    const int64_t max_pairs = (tiles + 1) / 2;
    const int64_t kv_head = 4 * S_tok * d;  // bytes of one head's K and V
    const int64_t heads_l2 = std::max<int64_t>(1, di.l2_bytes / 2 / kv_head);
    if (split && (H + heads_l2 - 1) / heads_l2 <= kMaxLptGroups &&
        2 * max_items * 4 <= workspace_bytes(d, grid) - kCountBytes) {
      int* cost = reinterpret_cast<int*>(p.ws_part);
      int* order = cost + max_items;
      p.lpt_heads_l2 = static_cast<int>(std::min<int64_t>(heads_l2, H));
      p.lpt_grid = grid;
      const int per_head = static_cast<int>((max_pairs + kPrepassItems - 1) / kPrepassItems);
      lpt_prepass_kernel<<<static_cast<unsigned>(H * per_head), kPrepassThreads, 0, s>>>(
          p, cost, order, per_head);
      if (rf_status st = launch_status("lpt_prepass_kernel launch")) return st;
      p.lpt_order = order;
    }
    return d == 128 ? launch<128, true>(mq, mq128, mk, mv, p, grid, di, s)
                    : launch<64, true>(mq, mq128, mk, mv, p, grid, di, s);
  }
  return d == 128 ? launch<128, false>(mq, mq128, mk, mv, p, grid, di, s)
                  : launch<64, false>(mq, mq128, mk, mv, p, grid, di, s);
}
}  // namespace

extern "C" rf_status rf_attn(void* d_O, float* d_lse, const void* d_Q, const void* d_K,
                             const void* d_V, int64_t qkv_row_stride, int64_t o_row_stride, int F,
                             int N, int H, int d, const int32_t* d_active,
                             const int32_t* d_counts, float softmax_scale, void* d_workspace,
                             int64_t workspace_bytes_given, int32_t* d_status,
                             rf_stream_t stream) {
  return attn_impl(d_O, d_lse, d_Q, d_K, d_V, qkv_row_stride, o_row_stride, F, N, H, d, d_active,
                   d_counts, softmax_scale, nullptr, d_workspace, workspace_bytes_given, d_status,
                   stream);
}

extern "C" rf_status rf_attn_block_masked(void* d_O, float* d_lse, const void* d_Q,
                                          const void* d_K, const void* d_V,
                                          int64_t qkv_row_stride, int64_t o_row_stride, int F,
                                          int N, int H, int d, const int32_t* d_active,
                                          const int32_t* d_counts, float softmax_scale,
                                          const uint8_t* d_block_mask, void* d_workspace,
                                          int64_t workspace_bytes_given, int32_t* d_status,
                                          rf_stream_t stream) {
  if (!d_block_mask) return RF_ERR_INVALID_ARG;
  return attn_impl(d_O, d_lse, d_Q, d_K, d_V, qkv_row_stride, o_row_stride, F, N, H, d, d_active,
                   d_counts, softmax_scale, d_block_mask, d_workspace, workspace_bytes_given,
                   d_status, stream);
}

// rf_attn without any device allocation: the split-KV scratch is the library's own static
// array.  Host code cannot pass the array's name to a kernel (in host code it only stands in
// for the symbol), so its device address is looked up once per device and cached.
extern "C" rf_status rf_attn_noalloc(void* d_O, float* d_lse, const void* d_Q, const void* d_K,
                                     const void* d_V, int64_t qkv_row_stride,
                                     int64_t o_row_stride, int F, int N, int H, int d,
                                     const int32_t* d_active, const int32_t* d_counts,
                                     float softmax_scale, int32_t* d_status, rf_stream_t stream) {
  // Argument errors return before the counter reset below is enqueued.
  DeviceInfo di;
  if (rf_status st = check_attn_args(d_O, d_Q, d_K, d_V, qkv_row_stride, o_row_stride, F, N, H,
                                     d, d_active, d_counts, softmax_scale, nullptr, nullptr, 0,
                                     &di))
    return st;
  int dev = 0;
  if (cudaError_t e = cudaGetDevice(&dev)) return fail(RF_ERR_CUDA, "cudaGetDevice", e);
  if (dev < 0 || dev >= 64) return fail(RF_ERR_UNSUPPORTED, "device ordinal >= 64");
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_addr[dev]) {
      void* ptr = nullptr;
      if (cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch))
        return fail(RF_ERR_CUDA, "cudaGetSymbolAddress(rf_attn_noalloc scratch)", e);
      g_noalloc_addr[dev] = ptr;
    }
    scratch = g_noalloc_addr[dev];
  }
  const int64_t need = rf_attn_workspace_bytes(d);
  if (need < 0) return d != 64 && d != 128 ? RF_ERR_UNSUPPORTED : RF_ERR_CUDA;
  if (need > kNoAllocScratchBytes) {
    char buf[160];
    std::snprintf(buf, sizeof(buf),
                  "rf_attn_noalloc: this device needs %lld bytes of split-KV scratch, the static "
                  "maximum is %lld",
                  static_cast<long long>(need), static_cast<long long>(kNoAllocScratchBytes));
    return fail(RF_ERR_UNSUPPORTED, buf);
  }
  // The array keeps whatever the previous call left; the merge counters must start at zero.
  if (cudaError_t e = cudaMemsetAsync(scratch, 0, kCountBytes, reinterpret_cast<cudaStream_t>(stream)))
    return fail(RF_ERR_CUDA, "cudaMemsetAsync(rf_attn_noalloc counters)", e);
  return rf_attn(d_O, d_lse, d_Q, d_K, d_V, qkv_row_stride, o_row_stride, F, N, H, d, d_active,
                 d_counts, softmax_scale, scratch, kNoAllocScratchBytes, d_status, stream);
}
