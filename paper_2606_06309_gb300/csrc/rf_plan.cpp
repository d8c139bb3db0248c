// rf_plan.cpp -- host planner: per-step active masks, Eq. 3 weights and Euler step sizes.
//
// Algorithm 2 (asynchronous denoising flow scheduling) with Eq. 2's progressive stride given
// as a per-step array.  Each frame carries the step it last jumped from (start) and the step
// its state has reached (due).  A frame is active at step s when it is a keyframe, when s is a
// warm-up step (Sec. 3.2.1), or when due == s; an active keyframe (or any frame in warm-up)
// advances one step, an active non-keyframe stride[s] steps, clamped to the final step.
// Skipped frames are projected with Eq. 3 in sigma units.
#include <cmath>
#include <cstring>
#include <vector>

#include "rf.h"

extern "C" rf_status rf_plan_build(int F, int S, const uint8_t* h_is_key, const int32_t* h_stride,
                                   int T_w, const double* h_sigma, uint8_t* h_mask, float* h_alpha,
                                   float* h_beta, float* h_dt, uint8_t* h_cur_slot) {
  if (F < 1 || S < 1 || T_w < 0 || T_w > S) return RF_ERR_INVALID_ARG;
  if (static_cast<int64_t>(F) * S > 0x7FFFFFFF) return RF_ERR_INVALID_ARG;
  if (!h_is_key || !h_stride || !h_mask || !h_alpha || !h_beta || !h_dt) return RF_ERR_INVALID_ARG;
  for (int s = 0; s < S; ++s)
    if (h_stride[s] < 1) return RF_ERR_INVALID_ARG;

  std::vector<double> sig(S + 1);
  if (h_sigma) {
    for (int s = 0; s <= S; ++s) sig[s] = h_sigma[s];
    if (sig[S] != 0.0) return RF_ERR_INVALID_ARG;
    for (int s = 0; s < S; ++s)
      if (!(sig[s] > sig[s + 1])) return RF_ERR_INVALID_ARG;
  } else {
    for (int s = 0; s <= S; ++s) sig[s] = 1.0 - static_cast<double>(s) / S;
  }

  std::vector<int> from(F, 0), reached(F, 0);
  std::vector<uint8_t> slot(F, 0);
  for (int s = 0; s < S; ++s) {
    const bool warm = s < T_w;
    for (int f = 0; f < F; ++f) {
      const size_t i = static_cast<size_t>(s) * F + f;
      if (h_cur_slot) h_cur_slot[i] = slot[f];
      const bool key = h_is_key[f] != 0;
      if (key || warm || reached[f] == s) {
        const int n = (key || warm) ? 1 : h_stride[s];
        from[f] = s;
        reached[f] = (s + n < S) ? s + n : S;
        h_mask[i] = 1;
        h_alpha[i] = 1.0f;
        h_beta[i] = 0.0f;
        h_dt[i] = static_cast<float>(sig[reached[f]] - sig[s]);
        slot[f] ^= 1;
      } else {
        const double s0 = sig[from[f]], s1 = sig[reached[f]];
        const double a = (s0 == s1) ? 0.0 : (s0 - sig[s]) / (s0 - s1);
        h_mask[i] = 0;
        h_alpha[i] = static_cast<float>(a);
        h_beta[i] = static_cast<float>(1.0 - a);
        h_dt[i] = 0.0f;
      }
    }
  }
  return RF_OK;
}

// Algorithm 1 (dynamic sequential keyframe selection) over the frames' inner products.
// Frame 0 is the first keyframe.  Frames are visited in order; while fewer than M keyframes
// exist, a frame whose cosine similarity to the latest keyframe is below tau becomes a
// keyframe, after tau is moved by -dtau if the gap to the latest keyframe is at least
// F/M + delta_up, or by +dtau if it is at most F/M - delta_down (Algorithm 1 as printed).
extern "C" rf_status rf_keyframe_select(const double* h_G, int F, int M, double tau, double dtau,
                                        double delta_up, double delta_down, uint8_t* h_is_key,
                                        int32_t* h_num_keys) {
  if (!h_G || !h_is_key || F < 1 || M < 1) return RF_ERR_INVALID_ARG;
  for (int f = 0; f < F; ++f) {
    h_is_key[f] = 0;
    if (!(h_G[static_cast<size_t>(f) * F + f] > 0.0)) return RF_ERR_INVALID_ARG;  // zero frame
  }
  h_is_key[0] = 1;
  int keys = 1, last = 0;
  const double L_avg = static_cast<double>(F) / M;
  for (int i = 1; i < F; ++i) {
    if (keys >= M) break;
    const double gii = h_G[static_cast<size_t>(i) * F + i];
    const double gll = h_G[static_cast<size_t>(last) * F + last];
    const double sim = h_G[static_cast<size_t>(i) * F + last] / (std::sqrt(gii) * std::sqrt(gll));
    if (sim < tau) {
      const int gap = i - last;
      if (gap >= L_avg + delta_up)
        tau -= dtau;
      else if (gap <= L_avg - delta_down)
        tau += dtau;
      h_is_key[i] = 1;
      ++keys;
      last = i;
    }
  }
  if (h_num_keys) *h_num_keys = keys;
  return RF_OK;
}
