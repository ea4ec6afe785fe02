// refadapt_ln_modulate: the DiT block's modulated LayerNorm,
//   x = (h - mean(h)) / sqrt(var(h) + eps) * (1 + scale[sample]) + shift[sample]
// over the C features of every row (no affine of its own; the AdaLN shift and
// scale of the block, stream and sample modulate it). HBM-bound: one warp per
// row, 16-byte loads and stores, the row held in registers, mean and variance
// in fp32 in two passes over the registers. Reference segments may be gated on
// the per-sample mode (skipped when REUSE).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstring>

#include "api_common.h"
#include "tc_ptx.cuh"

namespace ra {
namespace lnmod {

constexpr int WARPS = 8;
constexpr int MAX_GROUPS = 16;  // 8 features per lane per group: C <= 4096

struct Seg {
  const __nv_bfloat16* h;
  int64_t h_ss, h_sr;
  __nv_bfloat16* x;
  int64_t x_ss, x_sr;
  const float* shift;
  const float* scale;
  int64_t mod_ss;
  int32_t rows, gated;
  int64_t row_begin;  // first global row index of this segment
};

struct Params {
  Seg seg[3];
  int32_t n_seg, B, C, groups;
  int64_t total_rows;
  float eps;
  const int32_t* mode;
};

template <int G>  // 8-feature groups per lane: C = 256 G
__global__ void __launch_bounds__(32 * WARPS) ln_mod_kernel(const __grid_constant__ Params p) {
  const int lane = threadIdx.x & 31;
  const int64_t gr = int64_t(blockIdx.x) * WARPS + (threadIdx.x >> 5);
  if (gr >= p.total_rows) return;
  int g = 0;
  while (g + 1 < p.n_seg && gr >= p.seg[g + 1].row_begin) ++g;
  const Seg& sg = p.seg[g];
  const int64_t local = gr - sg.row_begin;
  const int s = int(local / sg.rows), r = int(local % sg.rows);
  if (sg.gated && __ldg(p.mode + s) == RA_MODE_REUSE) return;
  const uint4* src = reinterpret_cast<const uint4*>(sg.h + s * sg.h_ss + int64_t(r) * sg.h_sr);
  float v[G][8];
  float sum = 0.f;
#pragma unroll
  for (int q = 0; q < G; ++q) {
    const uint4 u = __ldg(src + q * 32 + lane);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[q][2 * e] = __uint_as_float(w[e] << 16);
      v[q][2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
      sum += v[q][2 * e] + v[q][2 * e + 1];
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  const float mean = sum / float(p.C);
  float sq = 0.f;
#pragma unroll
  for (int q = 0; q < G; ++q)
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float dv = v[q][e] - mean;
      sq = fmaf(dv, dv, sq);
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  const float rstd = rsqrtf(sq / float(p.C) + p.eps);
  const float* shift = sg.shift + s * sg.mod_ss;
  const float* scale = sg.scale + s * sg.mod_ss;
  uint4* dst = reinterpret_cast<uint4*>(sg.x + s * sg.x_ss + int64_t(r) * sg.x_sr);
#pragma unroll
  for (int q = 0; q < G; ++q) {
    const int c = (q * 32 + lane) * 8;
      const float4 sh0 = __ldg(reinterpret_cast<const float4*>(shift + c));
      const float4 sh1 = __ldg(reinterpret_cast<const float4*>(shift + c + 4));
      const float4 sc0 = __ldg(reinterpret_cast<const float4*>(scale + c));
      const float4 sc1 = __ldg(reinterpret_cast<const float4*>(scale + c + 4));
      const float shv[8] = {sh0.x, sh0.y, sh0.z, sh0.w, sh1.x, sh1.y, sh1.z, sh1.w};
      const float scv[8] = {sc0.x, sc0.y, sc0.z, sc0.w, sc1.x, sc1.y, sc1.z, sc1.w};
      uint32_t pk[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float y0 = fmaf((v[q][2 * e] - mean) * rstd, 1.f + scv[2 * e], shv[2 * e]);
        const float y1 = fmaf((v[q][2 * e + 1] - mean) * rstd, 1.f + scv[2 * e + 1], shv[2 * e + 1]);
        pk[e] = pack_bf16x2(y0, y1);
      }
      dst[q * 32 + lane] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  }
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace lnmod
}  // namespace ra

extern "C" ra_status refadapt_ln_modulate(const ra_lnmod_args* a, void* stream) {
  using namespace ra;
  using namespace ra::lnmod;
  clear_error();
  if (!a) {
    set_error("refadapt_ln_modulate: args is NULL");
    return RA_EINVAL;
  }
  if (a->B < 1 || a->n_seg < 1 || a->n_seg > 3 || a->C < 256 || a->C % 256 != 0 || a->C > 256 * MAX_GROUPS ||
      !(a->eps >= 0.f)) {
    set_error("refadapt_ln_modulate: need B >= 1, 1 <= n_seg <= 3, C a multiple of 256 in [256, 4096], "
              "eps >= 0 (B=%d n_seg=%d C=%d)", a->B, a->n_seg, a->C);
    return RA_EINVAL;
  }
  Params p;
  std::memset(&p, 0, sizeof(p));
  p.n_seg = a->n_seg;
  p.B = a->B;
  p.C = a->C;
  p.groups = a->C / 256;
  p.eps = a->eps;
  p.mode = a->mode;
  int64_t rows = 0;
  for (int g = 0; g < a->n_seg; ++g) {
    const ra_lnmod_seg& s = a->seg[g];
    Seg& d = p.seg[g];
    if (s.rows < 0) {
      set_error("refadapt_ln_modulate: seg %d rows < 0", g);
      return RA_EINVAL;
    }
    d.row_begin = rows;
    d.rows = s.rows;
    d.gated = s.gated ? 1 : 0;
    if (s.gated && !a->mode) {
      set_error("refadapt_ln_modulate: seg %d is gated but mode is NULL", g);
      return RA_EINVAL;
    }
    if (s.rows == 0) continue;
    if (!s.h || !s.x || !s.shift || !s.scale || !aligned16(s.h) || !aligned16(s.x) || !aligned16(s.shift) ||
        !aligned16(s.scale) || s.h_stride_r % 8 || s.h_stride_s % 8 || s.x_stride_r % 8 || s.x_stride_s % 8 ||
        s.mod_stride_s % 4 || s.h_stride_r < a->C || s.x_stride_r < a->C) {
      set_error("refadapt_ln_modulate: seg %d: pointers must be 16-byte aligned, row strides >= C and "
                "multiples of 8 elements (mod_stride_s of 4)", g);
      return RA_EINVAL;
    }
    d.h = static_cast<const __nv_bfloat16*>(s.h);
    d.h_ss = s.h_stride_s;
    d.h_sr = s.h_stride_r;
    d.x = static_cast<__nv_bfloat16*>(s.x);
    d.x_ss = s.x_stride_s;
    d.x_sr = s.x_stride_r;
    d.shift = s.shift;
    d.scale = s.scale;
    d.mod_ss = s.mod_stride_s;
    rows += int64_t(a->B) * s.rows;
  }
  p.total_rows = rows;
  if (rows == 0) return RA_OK;
  const int64_t blocks = (rows + WARPS - 1) / WARPS;
  if (blocks > 2147483647) {
    set_error("refadapt_ln_modulate: too many rows");
    return RA_EINVAL;
  }
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  switch (p.groups) {
#define RA_LNMOD_CASE(G) \
  case G: ln_mod_kernel<G><<<unsigned(blocks), 32 * WARPS, 0, st>>>(p); break;
    RA_LNMOD_CASE(1) RA_LNMOD_CASE(2) RA_LNMOD_CASE(3) RA_LNMOD_CASE(4) RA_LNMOD_CASE(5) RA_LNMOD_CASE(6)
    RA_LNMOD_CASE(7) RA_LNMOD_CASE(8) RA_LNMOD_CASE(9) RA_LNMOD_CASE(10) RA_LNMOD_CASE(11) RA_LNMOD_CASE(12)
    RA_LNMOD_CASE(13) RA_LNMOD_CASE(14) RA_LNMOD_CASE(15) RA_LNMOD_CASE(16)
#undef RA_LNMOD_CASE
    default: break;
  }
  return launch_status("refadapt_ln_modulate");
}
