// rf_pipeline.cpp -- the step core fed from pinned host memory (host-side runtime).
//
// One asynchronous denoising step (Algorithm 2) per call, with its inputs copied from the host
// and its results copied back, the copies of neighbouring steps overlapped with the compute of
// the current one.  What a step reads from the host: the query, key and value rows of the frames
// active at that step (the fresh ones) and the velocity.  The keys and values of skipped frames
// come from the device-resident rolling cache (Appendix B.2): rf_project_kv writes their Eq. 3
// projection into the step's K/V buffers and shifts the fresh rows into the cache.  What a step
// writes back: the active frames' rows of the attention output, the Eq. 3 latent context and
// the two-slot latent store.  `depth` device buffer sets and three caller streams (compute,
// host->device, device->host) are ordered by events; nothing synchronises the host until
// rf_pipeline_sync.
#include <cuda_runtime.h>

#include <new>
#include <utility>
#include <vector>

#include "rf.h"
#include "rf_host.h"

using rf::fail;

struct rf_pipeline {
  int F = 0, N = 0, H = 0, d = 0, S = 0, depth = 0;
  int64_t E = 0, S_tok = 0, row_bytes = 0;
  cudaStream_t compute = nullptr, h2d = nullptr, d2h = nullptr;
  std::vector<void*> allocs;  // every device allocation, freed by rf_pipeline_destroy
  std::vector<cudaEvent_t> events;
  // the plan, [S][F] on the device, and its mask on the host (for the active rows)
  uint8_t* mask = nullptr;
  float* alpha = nullptr;
  float* beta = nullptr;
  float* dt = nullptr;
  uint8_t* cur_slot = nullptr;
  std::vector<uint8_t> h_mask;
  // state
  float* z2 = nullptr;   // [2][F][E]
  float* ctx = nullptr;  // [F][E]
  void* Kc = nullptr;    // rolling key/value cache, bf16 [2][F][N][H*d]
  void* Vc = nullptr;
  int32_t* active = nullptr;
  int32_t* skipped = nullptr;
  int32_t* counts = nullptr;
  int32_t* status = nullptr;
  void* ws = nullptr;
  int64_t ws_bytes = 0;
  struct Set {
    void *Q, *K, *V, *O;
    float* v;
    float* z;
    float* ctx;
    cudaEvent_t loaded, consumed, drained;
  };
  std::vector<Set> sets;
  int64_t steps = 0, h2d_bytes = 0, d2h_bytes = 0;
};

namespace {

rf_status cuda_fail(const char* what, cudaError_t e) { return fail(RF_ERR_CUDA, what, e); }

rf_status alloc(rf_pipeline* p, void** out, size_t bytes) {
  if (cudaError_t e = cudaMalloc(out, bytes)) return cuda_fail("cudaMalloc (rf_pipeline)", e);
  p->allocs.push_back(*out);
  return RF_OK;
}

rf_status event(rf_pipeline* p, cudaEvent_t* out) {
  if (cudaError_t e = cudaEventCreateWithFlags(out, cudaEventDisableTiming))
    return cuda_fail("cudaEventCreateWithFlags (rf_pipeline)", e);
  p->events.push_back(*out);
  return RF_OK;
}

void release(rf_pipeline* p) {
  for (cudaEvent_t e : p->events) cudaEventDestroy(e);
  for (void* a : p->allocs) cudaFree(a);
  delete p;
}

}  // namespace

#define RF_TRY(x)                      \
  do {                                 \
    if (rf_status st_ = (x)) return st_; \
  } while (0)
#define CUDA_TRY(x, what)                              \
  do {                                                 \
    if (cudaError_t e_ = (x)) return cuda_fail(what, e_); \
  } while (0)

namespace {

rf_status create(rf_pipeline* p, const uint8_t* h_mask, const float* h_alpha,
                 const float* h_beta, const float* h_dt, const uint8_t* h_cur_slot,
                 const float* h_z2, const void* h_K0, const void* h_V0) {
  const size_t SF = static_cast<size_t>(p->S) * p->F;
  const size_t FE = static_cast<size_t>(p->F) * p->E;
  void* v = nullptr;
  RF_TRY(alloc(p, &v, SF)); p->mask = static_cast<uint8_t*>(v);
  RF_TRY(alloc(p, &v, SF * 4)); p->alpha = static_cast<float*>(v);
  RF_TRY(alloc(p, &v, SF * 4)); p->beta = static_cast<float*>(v);
  RF_TRY(alloc(p, &v, SF * 4)); p->dt = static_cast<float*>(v);
  RF_TRY(alloc(p, &v, SF)); p->cur_slot = static_cast<uint8_t*>(v);
  RF_TRY(alloc(p, &v, 2 * FE * 4)); p->z2 = static_cast<float*>(v);
  RF_TRY(alloc(p, &v, FE * 4)); p->ctx = static_cast<float*>(v);
  RF_TRY(alloc(p, &v, static_cast<size_t>(p->F) * 4)); p->active = static_cast<int32_t*>(v);
  RF_TRY(alloc(p, &v, static_cast<size_t>(p->F) * 4)); p->skipped = static_cast<int32_t*>(v);
  RF_TRY(alloc(p, &v, 2 * 4)); p->counts = static_cast<int32_t*>(v);
  RF_TRY(alloc(p, &v, 4)); p->status = static_cast<int32_t*>(v);
  const size_t qkv = static_cast<size_t>(p->S_tok) * p->row_bytes;
  RF_TRY(alloc(p, &p->Kc, 2 * qkv));
  RF_TRY(alloc(p, &p->Vc, 2 * qkv));
  p->ws_bytes = rf_attn_workspace_bytes(p->d);
  if (p->ws_bytes < 0) return fail(RF_ERR_CUDA, "rf_attn_workspace_bytes (rf_pipeline)");
  RF_TRY(alloc(p, &p->ws, static_cast<size_t>(p->ws_bytes)));
  CUDA_TRY(cudaMemcpy(p->mask, h_mask, SF, cudaMemcpyHostToDevice), "plan upload");
  CUDA_TRY(cudaMemcpy(p->alpha, h_alpha, SF * 4, cudaMemcpyHostToDevice), "plan upload");
  CUDA_TRY(cudaMemcpy(p->beta, h_beta, SF * 4, cudaMemcpyHostToDevice), "plan upload");
  CUDA_TRY(cudaMemcpy(p->dt, h_dt, SF * 4, cudaMemcpyHostToDevice), "plan upload");
  CUDA_TRY(cudaMemcpy(p->cur_slot, h_cur_slot, SF, cudaMemcpyHostToDevice), "plan upload");
  CUDA_TRY(cudaMemcpy(p->z2, h_z2, 2 * FE * 4, cudaMemcpyHostToDevice), "state upload");
  // both cache slots of every frame start with the initial keys and values (the identity for
  // a frame projected before its second update, as both latent slots start with z0)
  for (int slot = 0; slot < 2; ++slot) {
    CUDA_TRY(cudaMemcpy(static_cast<char*>(p->Kc) + slot * qkv, h_K0, qkv, cudaMemcpyHostToDevice),
             "cache upload");
    CUDA_TRY(cudaMemcpy(static_cast<char*>(p->Vc) + slot * qkv, h_V0, qkv, cudaMemcpyHostToDevice),
             "cache upload");
  }
  CUDA_TRY(cudaMemset(p->ws, 0, static_cast<size_t>(p->ws_bytes)), "workspace");
  CUDA_TRY(cudaMemset(p->status, 0, 4), "status");
  p->h_mask.assign(h_mask, h_mask + SF);
  p->sets.resize(p->depth);
  for (rf_pipeline::Set& B : p->sets) {
    RF_TRY(alloc(p, &B.Q, qkv));
    RF_TRY(alloc(p, &B.K, qkv));
    RF_TRY(alloc(p, &B.V, qkv));
    RF_TRY(alloc(p, &B.O, qkv));
    RF_TRY(alloc(p, &v, FE * 4)); B.v = static_cast<float*>(v);
    RF_TRY(alloc(p, &v, 2 * FE * 4)); B.z = static_cast<float*>(v);
    RF_TRY(alloc(p, &v, FE * 4)); B.ctx = static_cast<float*>(v);
    RF_TRY(event(p, &B.loaded));
    RF_TRY(event(p, &B.consumed));
    RF_TRY(event(p, &B.drained));
  }
  return RF_OK;
}

}  // namespace

extern "C" rf_status rf_pipeline_create(int F, int N, int H, int d, int64_t E, int S,
                                        const uint8_t* h_mask, const float* h_alpha,
                                        const float* h_beta, const float* h_dt,
                                        const uint8_t* h_cur_slot, const float* h_z2,
                                        const void* h_K0, const void* h_V0, int depth,
                                        rf_stream_t compute, rf_stream_t h2d, rf_stream_t d2h,
                                        rf_pipeline** out) {
  if (!out) return RF_ERR_INVALID_ARG;
  *out = nullptr;
  if (!h_mask || !h_alpha || !h_beta || !h_dt || !h_cur_slot || !h_z2 || !h_K0 || !h_V0)
    return RF_ERR_INVALID_ARG;
  if (F < 1 || F > 65535 || N < 1 || H < 1 || S < 1 || E < 4 || depth < 2 || depth > 8)
    return RF_ERR_INVALID_ARG;
  if (d != 64 && d != 128) return RF_ERR_UNSUPPORTED;
  if (E % 4 != 0) return RF_ERR_MISALIGNED;
  rf_pipeline* p = new (std::nothrow) rf_pipeline;
  if (!p) return fail(RF_ERR_INVALID_ARG, "rf_pipeline_create: out of host memory");
  p->F = F;
  p->N = N;
  p->H = H;
  p->d = d;
  p->S = S;
  p->depth = depth;
  p->E = E;
  p->S_tok = static_cast<int64_t>(F) * N;
  p->row_bytes = static_cast<int64_t>(H) * d * 2;
  p->compute = reinterpret_cast<cudaStream_t>(compute);
  p->h2d = reinterpret_cast<cudaStream_t>(h2d);
  p->d2h = reinterpret_cast<cudaStream_t>(d2h);
  if (rf_status st = create(p, h_mask, h_alpha, h_beta, h_dt, h_cur_slot, h_z2, h_K0, h_V0)) {
    release(p);
    return st;
  }
  *out = p;
  return RF_OK;
}

extern "C" rf_status rf_pipeline_step(rf_pipeline* p, int s, const void* h_Q, const void* h_K,
                                      const void* h_V, const float* h_v, void* h_O, float* h_z2,
                                      float* h_ctx, float softmax_scale) {
  if (!p || !h_Q || !h_K || !h_V || !h_v || !h_O || !h_z2) return RF_ERR_INVALID_ARG;
  if (s < 0 || s >= p->S) return RF_ERR_INVALID_ARG;
  const int F = p->F;
  const int64_t frame_bytes = static_cast<int64_t>(p->N) * p->row_bytes;
  const size_t FE4 = static_cast<size_t>(F) * p->E * 4;
  rf_pipeline::Set& B = p->sets[p->steps % p->depth];
  const bool first_use = p->steps < p->depth;
  // frames active at step s, as runs of consecutive frames (one copy per run)
  std::vector<std::pair<int, int>> runs;
  const uint8_t* m = p->h_mask.data() + static_cast<size_t>(s) * F;
  for (int f = 0; f < F;) {
    if (!m[f]) {
      ++f;
      continue;
    }
    int g = f;
    while (g < F && m[g]) ++g;
    runs.emplace_back(f, g);
    f = g;
  }
  int64_t active_bytes = 0;
  // host -> device: the fresh Q, K and V rows of the active frames, and the velocity
  if (!first_use) CUDA_TRY(cudaStreamWaitEvent(p->h2d, B.consumed, 0), "rf_pipeline h2d wait");
  for (const auto& r : runs) {
    const int64_t off = r.first * frame_bytes, n = (r.second - r.first) * frame_bytes;
    const std::pair<void*, const void*> qkv[3] = {{B.Q, h_Q}, {B.K, h_K}, {B.V, h_V}};
    for (const auto& x : qkv)
      CUDA_TRY(cudaMemcpyAsync(static_cast<char*>(x.first) + off,
                               static_cast<const char*>(x.second) + off, n,
                               cudaMemcpyHostToDevice, p->h2d),
               "rf_pipeline Q/K/V copy");
    active_bytes += n;
  }
  CUDA_TRY(cudaMemcpyAsync(B.v, h_v, FE4, cudaMemcpyHostToDevice, p->h2d), "rf_pipeline v copy");
  CUDA_TRY(cudaEventRecord(B.loaded, p->h2d), "rf_pipeline event");
  // the step core on the compute stream
  CUDA_TRY(cudaStreamWaitEvent(p->compute, B.loaded, 0), "rf_pipeline compute wait");
  if (!first_use)
    CUDA_TRY(cudaStreamWaitEvent(p->compute, B.drained, 0), "rf_pipeline compute wait");
  const rf_stream_t cs = reinterpret_cast<rf_stream_t>(p->compute);
  const size_t o = static_cast<size_t>(s) * F;
  RF_TRY(rf_schedule_compact(p->mask + o, F, p->N, p->active, p->skipped, nullptr, p->counts, cs));
  RF_TRY(rf_project(p->ctx, p->z2, p->cur_slot + o, p->alpha + o, p->beta + o, F, p->E, cs));
  const int64_t hd = static_cast<int64_t>(p->H) * p->d;
  // skipped frames' keys and values: Eq. 3 over the cache; active frames' fresh rows shifted in
  RF_TRY(rf_project_kv(B.K, B.V, hd, p->Kc, p->Vc, p->cur_slot + o, p->alpha + o, p->beta + o,
                       p->active, p->skipped, p->counts, F, p->N, static_cast<int>(hd), cs));
  RF_TRY(rf_attn(B.O, nullptr, B.Q, B.K, B.V, hd, hd, F, p->N, p->H, p->d, p->active, p->counts,
                 softmax_scale, p->ws, p->ws_bytes, p->status, cs));
  RF_TRY(rf_step(p->z2, p->cur_slot + o, B.v, p->dt + o, p->active, p->counts, F, p->E, cs));
  CUDA_TRY(cudaMemcpyAsync(B.z, p->z2, 2 * FE4, cudaMemcpyDeviceToDevice, p->compute),
           "rf_pipeline state snapshot");
  if (h_ctx)
    CUDA_TRY(cudaMemcpyAsync(B.ctx, p->ctx, FE4, cudaMemcpyDeviceToDevice, p->compute),
             "rf_pipeline context snapshot");
  CUDA_TRY(cudaEventRecord(B.consumed, p->compute), "rf_pipeline event");
  // device -> host
  CUDA_TRY(cudaStreamWaitEvent(p->d2h, B.consumed, 0), "rf_pipeline d2h wait");
  for (const auto& r : runs) {
    const int64_t off = r.first * frame_bytes, n = (r.second - r.first) * frame_bytes;
    CUDA_TRY(cudaMemcpyAsync(static_cast<char*>(h_O) + off, static_cast<char*>(B.O) + off, n,
                             cudaMemcpyDeviceToHost, p->d2h),
             "rf_pipeline O copy");
  }
  CUDA_TRY(cudaMemcpyAsync(h_z2, B.z, 2 * FE4, cudaMemcpyDeviceToHost, p->d2h),
           "rf_pipeline state copy");
  if (h_ctx)
    CUDA_TRY(cudaMemcpyAsync(h_ctx, B.ctx, FE4, cudaMemcpyDeviceToHost, p->d2h),
             "rf_pipeline context copy");
  CUDA_TRY(cudaEventRecord(B.drained, p->d2h), "rf_pipeline event");
  ++p->steps;
  p->h2d_bytes += 3 * active_bytes + static_cast<int64_t>(FE4);
  p->d2h_bytes += active_bytes + (h_ctx ? 3 : 2) * static_cast<int64_t>(FE4);
  return RF_OK;
}

extern "C" rf_status rf_pipeline_sync(rf_pipeline* p, int32_t* h_status) {
  if (!p) return RF_ERR_INVALID_ARG;
  CUDA_TRY(cudaStreamSynchronize(p->h2d), "rf_pipeline sync");
  CUDA_TRY(cudaStreamSynchronize(p->compute), "rf_pipeline sync");
  CUDA_TRY(cudaStreamSynchronize(p->d2h), "rf_pipeline sync");
  if (h_status)
    CUDA_TRY(cudaMemcpy(h_status, p->status, 4, cudaMemcpyDeviceToHost), "rf_pipeline status");
  return RF_OK;
}

extern "C" rf_status rf_pipeline_bytes(const rf_pipeline* p, int64_t* h_steps,
                                       int64_t* h_h2d_bytes, int64_t* h_d2h_bytes) {
  if (!p) return RF_ERR_INVALID_ARG;
  if (h_steps) *h_steps = p->steps;
  if (h_h2d_bytes) *h_h2d_bytes = p->h2d_bytes;
  if (h_d2h_bytes) *h_d2h_bytes = p->d2h_bytes;
  return RF_OK;
}

extern "C" void rf_pipeline_destroy(rf_pipeline* p) {
  if (!p) return;
  cudaStreamSynchronize(p->h2d);
  cudaStreamSynchronize(p->compute);
  cudaStreamSynchronize(p->d2h);
  release(p);
}
