// refadapt_gate: Algorithm 1's per-block decision on the device, so a whole
// denoising step can be enqueued (or graph-captured) without a host sync.
//
// Score (paper Eq. 12): g_{t,b,h} = D_{t,b,h} * M_{t-1,b,h}, formed per head
// (or D alone / M alone for the controller ablation of Sec. 5.3);
// aggregate (App. A.2): gbar = mean_h g; cutoff (Eq. 13): the first block with
// gbar >= theta reactivates, deeper blocks compute; bounded-age refresh
// (Sec. 4): t - a_full >= delta_max recomputes every block of the step.
#include <cuda_runtime.h>

#include <cmath>

#include "api_common.h"

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

__global__ void init_kernel(ra_state* st, int32_t B) {
  int32_t* extra = reinterpret_cast<int32_t*>(st + 1);
  for (int i = threadIdx.x; i < 2 * B; i += blockDim.x) extra[i] = (i < B) ? 0 : -1;
  if (threadIdx.x == 0) {
    st->magic = kMagic;
    st->B = B;
    st->a_full = 0;
    st->full_step = 1;
    st->step = -1;
  }
}

// (hi, lo) += x with the rounding error of the addition kept in lo (TwoSum;
// the value is hi + lo). The sums stay off the FP64 pipe, which is narrow on
// this GPU, with about the accuracy of fp64 over these few terms.
__device__ __forceinline__ void ff_add(float& hi, float& lo, float x) {
  const float s = hi + x;
  const float v = s - hi;
  lo += (hi - (s - v)) + (x - v);
  hi = s;
}

// One CTA. Warps compute M_{t-1,b,h} for every (sample, head) from the mass
// partials (lane-strided two-float sums, then a fixed tree over the lanes)
// into shared memory; then thread s takes sample s through the decision.
__global__ void __launch_bounds__(THREADS) gate_kernel(const Params p) {
  extern __shared__ float m_sh[];  // [B * H]
  ra_state* st = p.st;
  int32_t* reactivated = reinterpret_cast<int32_t*>(st + 1);
  int32_t* boundary = reactivated + p.B;
  __shared__ int32_t full_step;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = THREADS / 32;
  if (threadIdx.x == 0) {
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
    full_step = st->full_step;
  }
  for (int sh = warp; sh < p.B * p.H; sh += nwarps) {
    float hi = 0.f, lo = 0.f;
    if (p.mp) {
      const float* row = p.mp + int64_t(sh) * p.mpl;
      for (int i = lane; i < p.mpl; i += 32) ff_add(hi, lo, row[i]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float xh = __shfl_down_sync(0xffffffffu, hi, o), xl = __shfl_down_sync(0xffffffffu, lo, o);
        ff_add(hi, lo, xh);
        lo += xl;
      }
    }
    if (lane == 0) {
      const float m = (hi + lo) / float(p.mass_rows_count);
      m_sh[sh] = m;
      if (p.m_out && p.mp) p.m_out[sh] = m;
    }
  }
  __syncthreads();
  for (int s = threadIdx.x; s < p.B; s += blockDim.x) {
    if (p.b == 0) {
      reactivated[s] = 0;
      boundary[s] = -1;
    }
    const bool have = (p.t >= 1) && p.qd && p.mp;
    float ghi = 0.f, glo = 0.f;
    if (have) {
      for (int h = 0; h < p.H; ++h) {
        const float dh = p.qd[s * p.H + h], mh = m_sh[s * p.H + h];
        if (p.cue == RA_CUE_CHANGE) {
          ff_add(ghi, glo, dh);
        } else if (p.cue == RA_CUE_EXPOSURE) {
          ff_add(ghi, glo, mh);
        } else {
          // the product's rounding error joins lo (exact by one fma)
          const float g = dh * mh;
          ff_add(ghi, glo, g);
          glo += fmaf(dh, mh, -g);
        }
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
}

}  // namespace gate
}  // namespace ra

extern "C" size_t refadapt_state_size(int32_t B) {
  if (B < 1) return 0;
  return sizeof(ra_state) + 2 * sizeof(int32_t) * size_t(B);
}

extern "C" ra_status refadapt_state_init(ra_state* state, int32_t B, void* stream) {
  using namespace ra;
  clear_error();
  if (!state || B < 1) {
    set_error("refadapt_state_init: state is NULL or B < 1");
    return RA_EINVAL;
  }
  gate::init_kernel<<<1, 256, 0, static_cast<cudaStream_t>(stream)>>>(state, B);
  return launch_status("refadapt_state_init");
}

extern "C" ra_status refadapt_gate(const ra_gate_args* a, void* stream) {
  using namespace ra;
  clear_error();
  if (!a || !a->state || !a->mode_out) {
    set_error("refadapt_gate: args, state or mode_out is NULL");
    return RA_EINVAL;
  }
  if (a->B < 1 || a->H < 1 || a->t < 0 || a->b < 0) {
    set_error("refadapt_gate: B, H must be >= 1 and t, b >= 0");
    return RA_EINVAL;
  }
  if (a->delta_max < 1) {
    set_error("refadapt_gate: delta_max must be >= 1");
    return RA_EINVAL;
  }
  if (a->t >= 1 && (!a->q_delta || !a->mass_partial_prev)) {
    set_error("refadapt_gate: q_delta and mass_partial_prev are required for t >= 1");
    return RA_EINVAL;
  }
  if (a->mass_partial_prev && (a->mass_partial_len < 1 || a->mass_row_count < 1)) {
    set_error("refadapt_gate: mass_partial_len and mass_row_count must be >= 1");
    return RA_EINVAL;
  }
  if (int64_t(a->B) * a->H > 6144) {
    set_error("refadapt_gate: B * H must be <= 6144");
    return RA_EINVAL;
  }
  if (a->cue != RA_CUE_PRODUCT && a->cue != RA_CUE_CHANGE && a->cue != RA_CUE_EXPOSURE) {
    set_error("refadapt_gate: unknown cue %d", a->cue);
    return RA_EINVAL;
  }
  if (std::isnan(a->theta)) {
    set_error("refadapt_gate: theta is NaN");
    return RA_EINVAL;
  }
  gate::Params p;
  p.theta = a->theta;
  p.t = a->t;
  p.b = a->b;
  p.B = a->B;
  p.H = a->H;
  p.delta_max = a->delta_max;
  p.forced_boundary = a->forced_boundary;
  p.mpl = a->mass_partial_len;
  p.mass_rows_count = a->mass_row_count;
  p.cue = a->cue;
  p.qd = a->q_delta;
  p.mp = a->mass_partial_prev;
  p.st = a->state;
  p.mode_out = a->mode_out;
  p.gbar_out = a->gbar_out;
  p.m_out = a->m_out;
  const size_t sh_bytes = size_t(a->B) * a->H * sizeof(float);
  gate::gate_kernel<<<1, gate::THREADS, sh_bytes, static_cast<cudaStream_t>(stream)>>>(p);
  return launch_status("refadapt_gate");
}
