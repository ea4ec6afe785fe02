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
#include "gate_body.cuh"

namespace ra {
namespace gate {

__global__ void init_kernel(ra_state* st, int32_t B) {
  int32_t* extra = reinterpret_cast<int32_t*>(st + 1);
  for (int i = threadIdx.x; i < 2 * B; i += blockDim.x) extra[i] = (i < B) ? 0 : -1;
  if (threadIdx.x == 0) {
    st->magic = kMagic;
    st->B = B;
    st->a_full = 0;
    st->full_step = 1;
    st->step = -1;
    for (int i = 0; i < 3; ++i) st->reserved[i] = 0;
  }
}

// One CTA runs the decision (decide() in gate_body.cuh).
__global__ void __launch_bounds__(THREADS) gate_kernel(const Params p) {
  extern __shared__ float m_sh[];  // [B * H]
  __shared__ int32_t full_step;
  decide(p, m_sh, &full_step);
}

ra_status make_params(const ra_gate_args* a, const char* who, Params* p) {
  if (!a || !a->state || !a->mode_out) {
    set_error("%s: args, state or mode_out is NULL", who);
    return RA_EINVAL;
  }
  if (a->B < 1 || a->H < 1 || a->t < 0 || a->b < 0) {
    set_error("%s: B, H must be >= 1 and t, b >= 0", who);
    return RA_EINVAL;
  }
  if (a->delta_max < 1) {
    set_error("%s: delta_max must be >= 1", who);
    return RA_EINVAL;
  }
  if (a->t >= 1 && (!a->q_delta || !a->mass_partial_prev)) {
    set_error("%s: q_delta and mass_partial_prev are required for t >= 1", who);
    return RA_EINVAL;
  }
  if (a->mass_partial_prev && (a->mass_partial_len < 1 || a->mass_row_count < 1)) {
    set_error("%s: mass_partial_len and mass_row_count must be >= 1", who);
    return RA_EINVAL;
  }
  if (int64_t(a->B) * a->H > kMaxBH) {
    set_error("%s: B * H must be <= %d", who, kMaxBH);
    return RA_EINVAL;
  }
  if (a->cue != RA_CUE_PRODUCT && a->cue != RA_CUE_CHANGE && a->cue != RA_CUE_EXPOSURE) {
    set_error("%s: unknown cue %d", who, a->cue);
    return RA_EINVAL;
  }
  if (std::isnan(a->theta)) {
    set_error("%s: theta is NaN", who);
    return RA_EINVAL;
  }
  p->theta = a->theta;
  p->t = a->t;
  p->b = a->b;
  p->B = a->B;
  p->H = a->H;
  p->delta_max = a->delta_max;
  p->forced_boundary = a->forced_boundary;
  p->mpl = a->mass_partial_len;
  p->mass_rows_count = a->mass_row_count;
  p->cue = a->cue;
  p->qd = a->q_delta;
  p->mp = a->mass_partial_prev;
  p->st = a->state;
  p->mode_out = a->mode_out;
  p->gbar_out = a->gbar_out;
  p->m_out = a->m_out;
  return RA_OK;
}

ra_status launch(const Params& p, cudaStream_t stream, const char* who) {
  const size_t sh_bytes = size_t(p.B) * p.H * sizeof(float);
  gate_kernel<<<1, THREADS, sh_bytes, stream>>>(p);
  return launch_status(who);
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
  gate::Params p;
  const ra_status v = gate::make_params(a, "refadapt_gate", &p);
  if (v != RA_OK) return v;
  return gate::launch(p, static_cast<cudaStream_t>(stream), "refadapt_gate");
}
