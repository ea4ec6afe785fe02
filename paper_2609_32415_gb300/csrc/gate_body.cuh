// Algorithm 1's per-block decision on the device: the controller state, the
// launch parameters and the pieces of the decision, shared by refadapt_gate's
// own kernel (one CTA does all of it) and by the Q-change kernel of
// refadapt_q_delta_gate (each cluster leader forms its head's exposure and
// score term, the last leader to finish sums the terms and decides). Both
// take the same arithmetic in the same order, so their results are equal.
//
// Score (paper Eq. 12): g_{t,b,h} = D_{t,b,h} * M_{t-1,b,h}, formed per head
// (or D alone / M alone for the controller ablation of Sec. 5.3);
// aggregate (App. A.2): gbar = mean_h g; cutoff (Eq. 13): the first block with
// gbar >= theta reactivates, deeper blocks compute; bounded-age refresh
// (Sec. 4): t - a_full >= delta_max recomputes every block of the step.
#pragma once
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "refadapt.h"

struct ra_state {
  int32_t magic;
  int32_t B;
  int32_t a_full;      // step of the last full refresh
  int32_t full_step;   // the current step is a full refresh
  int32_t step;        // the step opened at block 0
  int32_t reserved[3];
  // followed by reactivated[B], boundary[B]
};

namespace ra {
namespace gate {

constexpr int32_t kMagic = 0x52414701;
constexpr int THREADS = 256;
constexpr int kMaxBH = 6144;  // B * H limit: the head exposures live in shared memory

struct Params {
  double theta;
  int32_t t, b, B, H, delta_max, forced_boundary, mpl, mass_rows_count, cue;
  const float* qd;
  const float* mp;
  ra_state* st;
  int32_t* mode_out;
  float* gbar_out;
  float* m_out;
};

// (hi, lo) += x with the rounding error of the addition kept in lo (TwoSum;
// the value is hi + lo). The sums stay off the FP64 pipe, which is narrow on
// this GPU, with about the accuracy of fp64 over these few terms.
__device__ __forceinline__ void g_ff_add(float& hi, float& lo, float x) {
  const float s = hi + x;
  const float v = s - hi;
  lo += (hi - (s - v)) + (x - v);
  hi = s;
}

// Thread 0 of the deciding CTA: at block 0 opens step t (t = 0 or an expired
// bounded age forces a full refresh); returns the step's full-refresh flag.
__device__ __forceinline__ int32_t open_step(const Params& p) {
  ra_state* st = p.st;
  if (p.b == 0) {
    if (p.t == 0) {
      st->full_step = 1;
      st->a_full = 0;
    } else if (p.t - st->a_full >= p.delta_max) {
      st->full_step = 1;
      st->a_full = p.t;
    } else {
      st->full_step = 0;
    }
    st->step = p.t;
  }
  return st->full_step;
}

// One warp: M_{t-1,b,h} of (sample, head) row sh from its mass partials
// (lane-strided two-float sums, then a fixed tree over the lanes); the value
// is in lane 0.
__device__ __forceinline__ float head_exposure(const Params& p, int sh) {
  const int lane = threadIdx.x & 31;
  float hi = 0.f, lo = 0.f;
  const float* row = p.mp + int64_t(sh) * p.mpl;
  for (int i = lane; i < p.mpl; i += 32) g_ff_add(hi, lo, row[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float xh = __shfl_down_sync(0xffffffffu, hi, o), xl = __shfl_down_sync(0xffffffffu, lo, o);
    g_ff_add(hi, lo, xh);
    lo += xl;
  }
  return (hi + lo) / float(p.mass_rows_count);
}

// Head h's term of the score sum (Eq. 12 per head, or the ablation cue): g,
// and for the product the product's rounding error e (exact by one fma),
// which joins the low word of the sum.
__device__ __forceinline__ void score_term(int cue, float dh, float mh, float& g, float& e) {
  if (cue == RA_CUE_CHANGE) {
    g = dh;
    e = 0.f;
  } else if (cue == RA_CUE_EXPOSURE) {
    g = mh;
    e = 0.f;
  } else {
    g = dh * mh;
    e = fmaf(dh, mh, -g);
  }
}

// Sample s's decision given its per-head terms term(h, g, e) (have: a score
// exists, t >= 1 with D and M): gbar = mean_h g in two-float sums over the
// heads in order, compared with theta in fp64; mode and latch per Algorithm 1.
template <class Term>
__device__ __forceinline__ void decide_sample(const Params& p, int s, int32_t full_step, bool have, Term term) {
  int32_t* reactivated = reinterpret_cast<int32_t*>(p.st + 1);
  int32_t* boundary = reactivated + p.B;
  if (p.b == 0) {
    reactivated[s] = 0;
    boundary[s] = -1;
  }
  float ghi = 0.f, glo = 0.f;
  if (have) {
    for (int h = 0; h < p.H; ++h) {
      float g, e;
      term(h, g, e);
      g_ff_add(ghi, glo, g);
      if (p.cue == RA_CUE_PRODUCT) glo += e;
    }
  }
  // The comparison with theta (a double) is made in fp64 on hi + lo.
  const double gbar = have ? (double(ghi) + double(glo)) / double(p.H) : NAN;
  if (p.gbar_out) p.gbar_out[s] = float(gbar);
  int32_t mode;
  if (full_step) {
    mode = RA_MODE_FULL;
  } else if (reactivated[s]) {
    mode = RA_MODE_COMPUTE;
  } else {
    const bool cross = (p.forced_boundary >= 0) ? (p.b >= p.forced_boundary) : (have && gbar >= p.theta);
    if (cross) {
      mode = RA_MODE_BOUNDARY;
      reactivated[s] = 1;
      boundary[s] = p.b;
    } else {
      mode = RA_MODE_REUSE;
    }
  }
  p.mode_out[s] = mode;
}

// The whole decision in one CTA (refadapt_gate's kernel): every thread runs
// this (it holds a CTA barrier). Warps compute M for every (sample, head)
// into m_sh [B * H] of shared memory; then thread s takes sample s through
// the decision. The results do not depend on the CTA's size.
__device__ __forceinline__ void decide(const Params& p, float* m_sh, volatile int32_t* full_step_sh) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  if (threadIdx.x == 0) *full_step_sh = open_step(p);
  for (int sh = warp; sh < p.B * p.H; sh += nwarps) {
    const float m = p.mp ? head_exposure(p, sh) : 0.f;
    if (lane == 0) {
      m_sh[sh] = m;
      if (p.m_out && p.mp) p.m_out[sh] = m;
    }
  }
  __syncthreads();
  const int32_t full_step = *full_step_sh;
  const bool have = (p.t >= 1) && p.qd && p.mp;
  for (int s = threadIdx.x; s < p.B; s += blockDim.x)
    decide_sample(p, s, full_step, have, [&](int h, float& g, float& e) {
      score_term(p.cue, p.qd[s * p.H + h], m_sh[s * p.H + h], g, e);
    });
}

// Host side (gate.cu): checks an ra_gate_args and fills Params (RA_EINVAL
// with the reason recorded as `who`); launches refadapt_gate's own kernel.
ra_status make_params(const ra_gate_args* a, const char* who, Params* p);
ra_status launch(const Params& p, cudaStream_t stream, const char* who);

}  // namespace gate
}  // namespace ra
