// refadapt_ref_cache_update: materialise a block's reference K/V (and an
// optional hidden-state tensor) into its cache slot for every sample whose mode
// is COMPUTE or FULL, and record a_b = t (paper Eq. 11; Algorithm 1).
//
// HBM-bound copy: one grid-stride loop of 16-byte vectors per (tensor, sample);
// the mode is read on the device, so no host sync is needed.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "api_common.h"

namespace ra {
namespace cu {

constexpr int THREADS = 256;
constexpr int UNROLL = 4;

struct Tensor {
  const __nv_bfloat16* src;
  __nv_bfloat16* dst;
  int64_t s_sb, s_sh, s_sn, d_sb, d_sh, d_sn;
  int32_t heads, vec_per_row;
};

struct Params {
  Tensor t[3];
  int32_t n_tensors;
  int32_t n;
  const int32_t* mode;
  int32_t step;
  int32_t* a_b;
};

__device__ __forceinline__ bool refreshes(int32_t m) { return m == RA_MODE_COMPUTE || m == RA_MODE_FULL; }

// grid.y = tensor * B + sample
__global__ void __launch_bounds__(THREADS) copy_kernel(const Params p, int B) {
  const int ti = blockIdx.y / B;
  const int s = blockIdx.y % B;
  const int32_t m = __ldg(p.mode + s);
  if (!refreshes(m)) return;
  if (ti == 0 && blockIdx.x == 0 && threadIdx.x == 0 && p.a_b) p.a_b[s] = p.step;
  const Tensor& T = p.t[ti];
  if (T.src == T.dst) return;
  const int64_t per_head = int64_t(p.n) * T.vec_per_row;
  const int64_t total = per_head * T.heads;
  const int64_t stride = int64_t(gridDim.x) * THREADS;
  int64_t i = int64_t(blockIdx.x) * THREADS + threadIdx.x;
  for (; i + (UNROLL - 1) * stride < total; i += UNROLL * stride) {
    uint4 v[UNROLL];
    int64_t dofs[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int64_t idx = i + u * stride;
      const int64_t h = idx / per_head;
      const int64_t rem = idx - h * per_head;
      const int64_t row = rem / T.vec_per_row;
      const int64_t c = rem - row * T.vec_per_row;
      v[u] = __ldg(reinterpret_cast<const uint4*>(T.src + s * T.s_sb + h * T.s_sh + row * T.s_sn) + c);
      dofs[u] = s * T.d_sb + h * T.d_sh + row * T.d_sn + c * 8;
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) *reinterpret_cast<uint4*>(T.dst + dofs[u]) = v[u];
  }
  for (; i < total; i += stride) {
    const int64_t h = i / per_head;
    const int64_t rem = i - h * per_head;
    const int64_t row = rem / T.vec_per_row;
    const int64_t c = rem - row * T.vec_per_row;
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(T.src + s * T.s_sb + h * T.s_sh + row * T.s_sn) + c);
    *reinterpret_cast<uint4*>(T.dst + s * T.d_sb + h * T.d_sh + row * T.d_sn + c * 8) = v;
  }
}

__global__ void stamp_kernel(const int32_t* mode, int32_t step, int32_t* a_b, int B) {
  for (int s = threadIdx.x; s < B; s += blockDim.x)
    if (refreshes(mode[s])) a_b[s] = step;
}

}  // namespace cu
}  // namespace ra

extern "C" ra_status refadapt_ref_cache_update(const ra_seg* k_src, const ra_seg* v_src, const ra_seg* k_cache,
                                               const ra_seg* v_cache, int32_t B, int32_t H, int32_t d,
                                               const ra_seg* x_src, const ra_seg* x_cache, int32_t x_heads,
                                               int32_t x_width, const int32_t* mode, int32_t t, int32_t* a_b,
                                               void* stream) {
  using namespace ra;
  clear_error();
  if (!k_src || !v_src || !k_cache || !v_cache || !mode) {
    set_error("refadapt_ref_cache_update: NULL argument");
    return RA_EINVAL;
  }
  if (d != 64 && d != 128) {
    set_error("refadapt_ref_cache_update: d = %d (supported: 64, 128)", d);
    return RA_EINVAL;
  }
  if (B < 1 || H < 1 || B > 4096 || H > 65535) {
    set_error("refadapt_ref_cache_update: B = %d, H = %d out of range", B, H);
    return RA_EINVAL;
  }
  const int n = k_src->n;
  if (v_src->n != n || k_cache->n != n || v_cache->n != n) {
    set_error("refadapt_ref_cache_update: segments disagree on n");
    return RA_EINVAL;
  }
  if (!check_seg(*k_src, "refadapt_ref_cache_update: k_src") || !check_seg(*v_src, "refadapt_ref_cache_update: v_src") ||
      !check_seg(*k_cache, "refadapt_ref_cache_update: k_cache") ||
      !check_seg(*v_cache, "refadapt_ref_cache_update: v_cache"))
    return RA_EINVAL;
  const bool with_x = (x_src != nullptr) || (x_cache != nullptr);
  if (with_x) {
    if (!x_src || !x_cache) {
      set_error("refadapt_ref_cache_update: x_src and x_cache must both be set or both be NULL");
      return RA_EINVAL;
    }
    if (x_src->n != n || x_cache->n != n || x_heads < 1 || x_width < 8 || x_width % 8) {
      set_error("refadapt_ref_cache_update: x tensors need n = n_ref, x_heads >= 1, x_width a multiple of 8");
      return RA_EINVAL;
    }
    if (!check_seg(*x_src, "refadapt_ref_cache_update: x_src") ||
        !check_seg(*x_cache, "refadapt_ref_cache_update: x_cache"))
      return RA_EINVAL;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n == 0) {
    if (a_b) {
      cu::stamp_kernel<<<1, 128, 0, st>>>(mode, t, a_b, B);
      return launch_status("refadapt_ref_cache_update");
    }
    return RA_OK;
  }
  cu::Params p;
  auto fill = [&](cu::Tensor& T, const ra_seg* s, const ra_seg* dst, int heads, int width) {
    T.src = static_cast<const __nv_bfloat16*>(s->ptr);
    T.dst = static_cast<__nv_bfloat16*>(dst->ptr);
    T.s_sb = s->stride_b;
    T.s_sh = s->stride_h;
    T.s_sn = s->stride_n;
    T.d_sb = dst->stride_b;
    T.d_sh = dst->stride_h;
    T.d_sn = dst->stride_n;
    T.heads = heads;
    T.vec_per_row = width / 8;
  };
  fill(p.t[0], k_src, k_cache, H, d);
  fill(p.t[1], v_src, v_cache, H, d);
  p.n_tensors = 2;
  if (with_x) {
    fill(p.t[2], x_src, x_cache, x_heads, x_width);
    p.n_tensors = 3;
  }
  p.n = n;
  p.mode = mode;
  p.step = t;
  p.a_b = a_b;
  // About four CTAs per SM over all (tensor, sample) pairs.
  const int pairs = p.n_tensors * B;
  int per = (4 * num_sms() + pairs - 1) / pairs;
  const int64_t vecs = int64_t(n) * H * (d / 8);
  const int64_t max_useful = (vecs + cu::THREADS - 1) / cu::THREADS;
  if (per > max_useful) per = int(max_useful);
  if (per < 1) per = 1;
  dim3 grid(per, pairs);
  cu::copy_kernel<<<grid, cu::THREADS, 0, st>>>(p, B);
  return launch_status("refadapt_ref_cache_update");
}
