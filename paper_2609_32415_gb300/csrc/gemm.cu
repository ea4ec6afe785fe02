// refadapt_gemm: the linear layers of the DiT block around the attention
// (QKV projection, output projection, MLP), bf16 in, fp32 accumulate in TMEM,
// with the elementwise work that follows each layer fused into the epilogue.
//
//   D[r, n] = sum_k A[r, k] W[n, k]        (A rows of one segment and sample,
//                                           W in nn.Linear layout [N][K])
//
// Two kernels: CTA pairs on 256 x 256 output tiles (gemm_pair_kernel, below,
// used when a call has at least a wave of such tiles) and one CTA per SM on
// 128 x 256 tiles (gemm_kernel), both persistent, K in 64-column steps. Tiles
// are numbered segment-major, then sample, then in bands of GROUP_M row tiles,
// rows fastest inside a band (so the CTAs that run at once share a few A row
// blocks and a few W column blocks, both held in L2); CTA c takes tiles c,
// c + G, c + 2G, ...
//   warp 0      TMA producer: per K step one 128 x 64 A box and one 256 x 64 W
//               box (128-byte swizzle, rows past a segment's end read as
//               zeros) into a 4-stage ring.
//   warp 1      TMEM allocator (512 columns: two 256-column accumulators) and
//               MMA issuer: tcgen05.mma kind::f16, M = 128, N = 256, K = 16,
//               four per stage; commits free the stage and, after a tile's
//               last step, hand the accumulator to the epilogue.
//   warps 2..5  epilogue: thread = output row = TMEM lane (quarter = warp % 4),
//               32 columns per tcgen05.ld; the next tile's MMAs run into the
//               other accumulator meanwhile.
// Epilogues (fp32 until the final bf16 rounding):
//   STORE  out = acc + bias
//   GELU   out = gelu_tanh(acc + bias)
//   RESID  out = resid + gate[sample] * (acc + bias)        (gated residual)
//   QKV    columns [q | k | v] of H heads of width d: q and k RMS-normalised
//          per head with a [d] weight, then rotated by RoPE on interleaved
//          pairs at the row's joint position; written head-major.
// Reference segments may be gated on the per-sample mode: their tiles are
// skipped when the mode is REUSE (Algorithm 1 skips reference rows) and, for
// QKV, the K and V column tiles also when it is BOUNDARY (the block keeps its
// cached reference K/V). Every mbarrier wait is bounded; on a timeout the CTA
// drains its own TMA and MMA work, frees TMEM, flags the error word and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "api_common.h"
#include "tc_ptx.cuh"

namespace ra {
namespace gemm {

constexpr int BM = 128, BN = 256, BK = 64;
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int OFF_BAR = STAGES * STAGE_BYTES;
constexpr int NUM_BARS = 2 * STAGES + 2 + 2 + 1;  // full, empty, tfull[2], tempty[2], drain
constexpr int OFF_MISC = OFF_BAR + NUM_BARS * 8;
constexpr int SMEM_BYTES = OFF_MISC + 16;
constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;
constexpr int THREADS = 192;
constexpr int TMEM_COLS = 512;
static_assert(SMEM_ALLOC <= 232448, "shared memory budget");

// CTA-pair kernel: 256 x 256 output tiles; each CTA stages its 128 rows of A
// and its 128-column half of the W tile, 128 of K per stage (two 128-byte
// swizzle chunks per operand, 64 KB per stage, 3 stages): half the stage
// hand-offs of 64-wide stages, which the fused epilogues gained from (GELU
// +3 %); a K % 128 == 64 tail is a half stage.
constexpr int P_TM = 256;
constexpr int P_STAGES = 3;
constexpr int P_BK = 128;              // K per stage: two 64-column chunks per operand
constexpr int P_CHUNK = 128 * 64 * 2;  // 128 rows x 64 K of one operand (one 128-byte swizzle span)
constexpr int P_A_BYTES = 128 * P_BK * 2;
constexpr int P_B_BYTES = 128 * P_BK * 2;
constexpr int P_STAGE_BYTES = P_A_BYTES + P_B_BYTES;
constexpr int P_OFF_BAR = P_STAGES * P_STAGE_BYTES;
constexpr int P_NUM_BARS = 2 * P_STAGES + 2 + 2 + 1;
constexpr int P_OFF_MISC = P_OFF_BAR + P_NUM_BARS * 8;
constexpr int P_SMEM_BYTES = P_OFF_MISC + 16;
constexpr int P_SMEM_ALLOC = P_SMEM_BYTES + 1024;
static_assert(P_SMEM_ALLOC <= 232448, "shared memory budget");

struct Seg {
  int64_t tile_begin;
  int32_t rows, m_tiles, gated, pos_offset;
  const float* bias;
  __nv_bfloat16* out;
  int64_t out_ss, out_sr;
  const __nv_bfloat16* resid;
  int64_t res_ss, res_sr;
  const float* gate;
  int64_t gate_ss;
  __nv_bfloat16* dst[3];  // QKV: q, k, v, head-major
  int64_t dst_sb[3], dst_sh[3], dst_sn[3];
  const float* norm_w[2];  // QKV: q, k
};

struct Params {
  CUtensorMap tm_a[3], tm_w[3];
  Seg seg[3];
  int32_t n_seg, B, N, K, epi, H, d, C, n_tiles_n, kblocks;
  int64_t total_tiles;
  const int32_t* mode;
  const float4* rope;  // [pos][d/4]: (cos, sin) of two consecutive pairs
  int32_t rope_len;
  float norm_eps;
  int32_t* err_word;
  uint64_t budget_ns;
};

struct Tile {
  int seg, s, m0, n0;
  bool live;
};

constexpr int GROUP_M = 16;  // tile rows per band of the tile order

template <int TM>  // output rows per tile: 128 (one CTA) or 256 (a CTA pair)
__device__ __forceinline__ Tile decode(const Params& p, int64_t t) {
  Tile r;
  int g = 0;
  while (g + 1 < p.n_seg && t >= p.seg[g + 1].tile_begin) ++g;
  const Seg& sg = p.seg[g];
  const int64_t local = t - sg.tile_begin;
  const int64_t per_sample = int64_t(sg.m_tiles) * p.n_tiles_n;
  r.seg = g;
  r.s = int(local / per_sample);
  const int64_t rem = local - int64_t(r.s) * per_sample;
  // Grouped order: bands of GROUP_M tile rows, rows fastest inside a band, so
  // the tiles in flight at once (one per CTA pair) share a few A row blocks
  // and a few W column blocks that stay in L2, and W streams from HBM once per
  // band instead of once per wave.
  const int64_t band_tiles = int64_t(GROUP_M) * p.n_tiles_n;
  const int band = int(rem / band_tiles);
  const int m_first = band * GROUP_M;
  const int rows = min(GROUP_M, sg.m_tiles - m_first);
  const int idx = int(rem - int64_t(band) * band_tiles);
  r.m0 = (m_first + idx % rows) * TM;
  r.n0 = (idx / rows) * BN;
  r.live = true;
  if (sg.gated) {
    const int m = __ldg(p.mode + r.s);
    if (m == RA_MODE_REUSE) r.live = false;
    if (p.epi == RA_EPI_QKV && m == RA_MODE_BOUNDARY && r.n0 >= p.C) r.live = false;
  }
  return r;
}

// GELU, tanh form, through the identity 0.5 x (1 + tanh(u)) = x / (1 + e^(-2u)),
// u = sqrt(2/pi) (x + 0.044715 x^3): one exponential and one division instead
// of tanhf (e^(-2u) overflowing to +inf for very negative x gives -0).
__device__ __forceinline__ float gelu_tanh(float x) {
  const float u = 0.7978845608028654f * fmaf(0.044715f * x * x, x, x);
  return __fdividef(x, 1.f + __expf(-2.f * u));
}

__device__ __forceinline__ void store32(__nv_bfloat16* dst, const float (&x)[32]) {
  uint32_t pk[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2(x[2 * i], x[2 * i + 1]);
  uint4* d = reinterpret_cast<uint4*>(dst);
  d[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  d[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
  d[2] = make_uint4(pk[8], pk[9], pk[10], pk[11]);
  d[3] = make_uint4(pk[12], pk[13], pk[14], pk[15]);
}

__device__ __forceinline__ void load_acc(uint32_t taddr, const float* bias, int n, float (&x)[32]) {
  uint32_t v[32];
  tmem_ld32(taddr, v);
  tmem_ld_wait();
  if (bias) {
    const float4* b4 = reinterpret_cast<const float4*>(bias + n);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 b = __ldg(b4 + i);
      x[4 * i] = __uint_as_float(v[4 * i]) + b.x;
      x[4 * i + 1] = __uint_as_float(v[4 * i + 1]) + b.y;
      x[4 * i + 2] = __uint_as_float(v[4 * i + 2]) + b.z;
      x[4 * i + 3] = __uint_as_float(v[4 * i + 3]) + b.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) x[i] = __uint_as_float(v[i]);
  }
}

// Epilogue of one output tile for the calling thread's row r (within the
// segment's sample): 256 accumulator columns at TMEM address `base`.
__device__ __forceinline__ void epilogue_tile(const Params& p, const Tile& tl, int r, uint32_t base) {
  const Seg& sg = p.seg[tl.seg];
  const bool valid = r < sg.rows;
  if (p.epi == RA_EPI_QKV) {
    const int part = tl.n0 / p.C;               // 0 q, 1 k, 2 v
    const int h0 = (tl.n0 - part * p.C) / p.d;  // first head of the tile
    const int pos = sg.pos_offset + r;
    for (int hh = 0; hh < BN / p.d; ++hh) {
      const int cb = hh * p.d;                  // tile column of the head
      const int h = h0 + hh;
      __nv_bfloat16* drow = sg.dst[part] + tl.s * sg.dst_sb[part] + h * sg.dst_sh[part] +
                            int64_t(valid ? r : 0) * sg.dst_sn[part];
      if (part == 2) {
        for (int c0 = 0; c0 < p.d; c0 += 32) {
          float x[32];
          load_acc(base + cb + c0, sg.bias, tl.n0 + cb + c0, x);
          if (valid) store32(drow + c0, x);
        }
        continue;
      }
      float ss = 0.f;
      for (int c0 = 0; c0 < p.d; c0 += 32) {
        float x[32];
        load_acc(base + cb + c0, sg.bias, tl.n0 + cb + c0, x);
#pragma unroll
        for (int j = 0; j < 32; ++j) ss = fmaf(x[j], x[j], ss);
      }
      const float rstd = rsqrtf(ss / float(p.d) + p.norm_eps);
      const float* w = sg.norm_w[part];
      const float4* cs = p.rope + int64_t(valid ? pos : 0) * (p.d / 4);
      for (int c0 = 0; c0 < p.d; c0 += 32) {
        float x[32];
        load_acc(base + cb + c0, sg.bias, tl.n0 + cb + c0, x);
        const float4* w4 = reinterpret_cast<const float4*>(w + c0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 wv = __ldg(w4 + q);
          const float4 rc = valid ? __ldg(cs + c0 / 4 + q) : make_float4(1.f, 0.f, 1.f, 0.f);
          const float a0 = x[4 * q] * rstd * wv.x, a1 = x[4 * q + 1] * rstd * wv.y;
          const float b0 = x[4 * q + 2] * rstd * wv.z, b1 = x[4 * q + 3] * rstd * wv.w;
          x[4 * q] = a0 * rc.x - a1 * rc.y;
          x[4 * q + 1] = a0 * rc.y + a1 * rc.x;
          x[4 * q + 2] = b0 * rc.z - b1 * rc.w;
          x[4 * q + 3] = b0 * rc.w + b1 * rc.z;
        }
        if (valid) store32(drow + c0, x);
      }
    }
  } else {
    const int64_t orow = int64_t(tl.s) * sg.out_ss + int64_t(valid ? r : 0) * sg.out_sr;
    // RESID: the row's residual for the next 32 columns is loaded while the
    // current 32 are computed (one global-load latency per tile, not per chunk).
    const bool resid = p.epi == RA_EPI_RESID && valid;
    const uint4* rrow = resid ? reinterpret_cast<const uint4*>(sg.resid + int64_t(tl.s) * sg.res_ss +
                                                               int64_t(r) * sg.res_sr + tl.n0)
                              : nullptr;
    uint4 rnext[4];
    if (resid) {
#pragma unroll
      for (int q = 0; q < 4; ++q) rnext[q] = rrow[q];
    }
    for (int c0 = 0; c0 < BN; c0 += 32) {
      const int n = tl.n0 + c0;
      uint4 rcur[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) rcur[q] = rnext[q];
      if (resid && c0 + 32 < BN) {
#pragma unroll
        for (int q = 0; q < 4; ++q) rnext[q] = rrow[(c0 + 32) / 8 + q];
      }
      float x[32];
      load_acc(base + c0, sg.bias, n, x);
      if (p.epi == RA_EPI_GELU) {
#pragma unroll
        for (int j = 0; j < 32; ++j) x[j] = gelu_tanh(x[j]);
      } else if (resid) {
        const float4* gp = reinterpret_cast<const float4*>(sg.gate + int64_t(tl.s) * sg.gate_ss + n);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 rv = rcur[q];
          const uint32_t w4[4] = {rv.x, rv.y, rv.z, rv.w};
          const float4 g0 = __ldg(gp + 2 * q), g1 = __ldg(gp + 2 * q + 1);
          const float gv[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float lo = __uint_as_float(w4[e] << 16), hi = __uint_as_float(w4[e] & 0xFFFF0000u);
            x[8 * q + 2 * e] = fmaf(gv[2 * e], x[8 * q + 2 * e], lo);
            x[8 * q + 2 * e + 1] = fmaf(gv[2 * e + 1], x[8 * q + 2 * e + 1], hi);
          }
        }
      }
      if (valid) store32(sg.out + orow + n, x);
    }
  }}

__global__ void __launch_bounds__(THREADS, 1) gemm_kernel(const __grid_constant__ Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* tfull = bars + 2 * STAGES;
  uint64_t* tempty = bars + 2 * STAGES + 2;
  uint64_t* drain = bars + 2 * STAGES + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err_word, p.budget_ns};

  if (warp == 0) {
    if (lane == 0) {
      // -------------------------------------------------------------- producer
      for (int g = 0; g < p.n_seg; ++g)
        if (p.seg[g].rows > 0) {
          tma_prefetch_desc(&p.tm_a[g]);
          tma_prefetch_desc(&p.tm_w[g]);
        }
      int64_t it = 0;  // K steps issued
      bool ok = true;
      for (int64_t t = blockIdx.x; ok && t < p.total_tiles; t += gridDim.x) {
        const Tile tl = decode<BM>(p, t);
        if (!tl.live) continue;
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int st = int(it % STAGES);
          if (it >= STAGES && !(ok = mbar_wait(empty + st, uint32_t((it / STAGES - 1) & 1), ctl))) break;
          uint8_t* sa = smem + st * STAGE_BYTES;
          mbar_arrive_expect_tx(full + st, STAGE_BYTES);
          tma_load_4d(sa, &p.tm_a[tl.seg], full + st, kb * BK, tl.m0, 0, tl.s);
          tma_load_4d(sa + A_BYTES, &p.tm_w[tl.seg], full + st, kb * BK, tl.n0, 0, 0);
        }
      }
      if (*abort_flag) {
        for (int st = 0; st < STAGES; ++st) {
          const int64_t n_s = (it > st) ? (it - st + STAGES - 1) / STAGES : 0;
          if (n_s > 0) mbar_wait_drain(full + st, uint32_t((n_s - 1) & 1), p.budget_ns);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // -------------------------------------------------------------- MMA issuer
      constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN, 0, 0);
      const uint32_t s0 = smem_u32(smem);
      int64_t it = 0;
      int i = 0;
      bool ok = true, issued = false;
      for (int64_t t = blockIdx.x; ok && t < p.total_tiles; t += gridDim.x) {
        const Tile tl = decode<BM>(p, t);
        if (!tl.live) continue;
        const int buf = i & 1, use = i >> 1;
        if (use > 0 && !(ok = mbar_wait(tempty + buf, uint32_t((use - 1) & 1), ctl))) break;
        tc_fence_after();
        const uint32_t d_t = tmem + uint32_t(buf * BN);
        for (int kb = 0; kb < p.kblocks; ++kb, ++it) {
          const int st = int(it % STAGES);
          if (!(ok = mbar_wait(full + st, uint32_t((it / STAGES) & 1), ctl))) break;
          tc_fence_after();
          const uint32_t sa = s0 + st * STAGE_BYTES, sb = sa + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_ss(d_t, sdesc_sw128(sa + kk * 32, 16, 1024), sdesc_sw128(sb + kk * 32, 16, 1024), IDESC,
                    (kb > 0 || kk > 0) ? 1u : 0u);
          umma_commit(empty + st);
          issued = true;
        }
        if (!ok) break;
        umma_commit(tfull + buf);
        ++i;
      }
      if (!ok && issued) {
        umma_commit(drain);
        mbar_wait_drain(drain, 0, p.budget_ns);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    int i = 0;
    for (int64_t t = blockIdx.x; t < p.total_tiles; t += gridDim.x) {
      const Tile tl = decode<BM>(p, t);
      if (!tl.live) continue;
      const int buf = i & 1, use = i >> 1;
      if (!__all_sync(0xffffffffu, mbar_wait(tfull + buf, uint32_t(use & 1), ctl))) break;
      tc_fence_after();
      epilogue_tile(p, tl, tl.m0 + row, tmem + lane_off + uint32_t(buf * BN));
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty + buf);
      ++i;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}


// CTA-pair variant (cluster of two, cta_group::2). Both CTAs walk the same
// tile sequence (cluster c takes tiles c, c + G/2, ...); per K step each CTA's
// producer loads its own 128 A rows and its half of the W tile, and both
// loads complete on rank 0's full barrier (rank 0 arms it for both CTAs'
// bytes). Rank 0's MMA thread issues M = 256, N = 256 MMAs; commits are
// multicast to both CTAs (stage free, accumulator ready). Each CTA's epilogue
// reads its own TMEM rows and arrives on rank 0's accumulator-free barrier
// (count 8). The two CTAs meet at a cluster barrier before TMEM is freed and
// before either exits, so no remote arrive or MMA outlives its target.
__global__ void __launch_bounds__(THREADS, 1) gemm_pair_kernel(const __grid_constant__ Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + P_OFF_BAR);
  uint64_t* full = bars;
  uint64_t* empty = bars + P_STAGES;
  uint64_t* tfull = bars + 2 * P_STAGES;
  uint64_t* tempty = bars + 2 * P_STAGES + 2;
  uint64_t* drain = bars + 2 * P_STAGES + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + P_OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + P_OFF_MISC + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int64_t cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;
  if (threadIdx.x == 0) {
    for (int s = 0; s < P_STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, 8);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc_pair(tmem_slot, TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers and TMEM exist before any cross-CTA use
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err_word, p.budget_ns};

  if (warp == 0) {
    if (lane == 0) {
      // -------------------------------------------------------------- producer (both CTAs)
      for (int g = 0; g < p.n_seg; ++g)
        if (p.seg[g].rows > 0) {
          tma_prefetch_desc(&p.tm_a[g]);
          tma_prefetch_desc(&p.tm_w[g]);
        }
      const uint32_t full0 = mapa_shared(smem_u32(full), 0);  // rank 0's full barriers
      int64_t it = 0;
      bool ok = true;
      for (int64_t t = cid; ok && t < p.total_tiles; t += ncl) {
        const Tile tl = decode<P_TM>(p, t);
        if (!tl.live) continue;
        for (int kb = 0; kb < (p.kblocks + 1) / 2; ++kb, ++it) {
          const int st = int(it % P_STAGES);
          if (it >= P_STAGES && !(ok = mbar_wait(empty + st, uint32_t((it / P_STAGES - 1) & 1), ctl))) break;
          uint8_t* sa = smem + st * P_STAGE_BYTES;
          const int chunks = (2 * kb + 1 < p.kblocks) ? 2 : 1;  // K % 128 == 64: the last stage is half
          if (rank == 0) mbar_arrive_expect_tx(full + st, 4 * chunks * P_CHUNK);
          for (int c = 0; c < chunks; ++c) {
            tma_load_4d_pair(sa + c * P_CHUNK, &p.tm_a[tl.seg], full0 + 8u * st, kb * P_BK + c * 64,
                             tl.m0 + int(rank) * 128, 0, tl.s);
            tma_load_4d_pair(sa + P_A_BYTES + c * P_CHUNK, &p.tm_w[tl.seg], full0 + 8u * st, kb * P_BK + c * 64,
                             tl.n0 + int(rank) * 128, 0, 0);
          }
        }
      }
      if (*abort_flag) {
        if (rank == 0) {
          // rank 0's full barriers count both CTAs' bytes of every phase it armed
          for (int st = 0; st < P_STAGES; ++st) {
            const int64_t n_s = (it > st) ? (it - st + P_STAGES - 1) / P_STAGES : 0;
            if (n_s > 0) mbar_wait_drain(full + st, uint32_t((n_s - 1) & 1), p.budget_ns);
          }
        } else {
          // this CTA cannot observe its own loads' completion: give them time to land
          const uint64_t t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 200000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // -------------------------------------------------------------- MMA issuer (rank 0)
      constexpr uint32_t IDESC = idesc_bf16_f32(P_TM, BN, 0, 0);
      const uint32_t s0 = smem_u32(smem);
      int64_t it = 0;
      int i = 0;
      bool ok = true, issued = false;
      for (int64_t t = cid; ok && t < p.total_tiles; t += ncl) {
        const Tile tl = decode<P_TM>(p, t);
        if (!tl.live) continue;
        const int buf = i & 1, use = i >> 1;
        if (use > 0 && !(ok = mbar_wait_cluster(tempty + buf, uint32_t((use - 1) & 1), ctl))) break;
        tc_fence_after();
        const uint32_t d_t = tmem + uint32_t(buf * BN);
        for (int kb = 0; kb < (p.kblocks + 1) / 2; ++kb, ++it) {
          const int st = int(it % P_STAGES);
          if (!(ok = mbar_wait(full + st, uint32_t((it / P_STAGES) & 1), ctl))) break;
          tc_fence_after();
          const uint32_t sa = s0 + st * P_STAGE_BYTES, sb = sa + P_A_BYTES;
          const int ksteps = (2 * kb + 1 < p.kblocks) ? P_BK / 16 : 64 / 16;
#pragma unroll
          for (int kk = 0; kk < P_BK / 16; ++kk) {
            if (kk >= ksteps) break;
            const uint32_t o = uint32_t((kk >> 2) * P_CHUNK + (kk & 3) * 32);
            umma_ss_pair(d_t, sdesc_sw128(sa + o, 16, 1024), sdesc_sw128(sb + o, 16, 1024), IDESC,
                         (kb > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit_pair(empty + st, 0x3);
          issued = true;
        }
        if (!ok) break;
        umma_commit_pair(tfull + buf, 0x3);
        ++i;
      }
      if (!ok && issued) {
        umma_commit_pair(drain, 0x1);
        mbar_wait_drain(drain, 0, p.budget_ns);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue (both CTAs)
    const int quarter = warp & 3;
    const int row = int(rank) * 128 + quarter * 32 + lane;
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    const uint32_t tempty0 = mapa_shared(smem_u32(tempty), 0);
    int i = 0;
    for (int64_t t = cid; t < p.total_tiles; t += ncl) {
      const Tile tl = decode<P_TM>(p, t);
      if (!tl.live) continue;
      const int buf = i & 1, use = i >> 1;
      if (!__all_sync(0xffffffffu, mbar_wait(tfull + buf, uint32_t(use & 1), ctl))) break;
      tc_fence_after();
      epilogue_tile(p, tl, tl.m0 + row, tmem + lane_off + uint32_t(buf * BN));
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0)
          mbar_arrive(tempty + buf);
        else
          mbar_arrive_remote(tempty0 + 8u * buf);
      }
      ++i;
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, TMEM_COLS);
}

__global__ void rope_table_kernel(float* table, int32_t n_pos, int32_t d, double base) {
  const int64_t n = int64_t(n_pos) * (d / 2);
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x) {
    const int64_t pos = i / (d / 2);
    const int pair = int(i % (d / 2));
    const double ang = double(pos) * pow(base, -2.0 * pair / double(d));
    double s, c;
    sincos(ang, &s, &c);
    table[2 * i] = float(c);
    table[2 * i + 1] = float(s);
  }
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

}  // namespace gemm
}  // namespace ra

extern "C" ra_status refadapt_rope_table(float* table, int32_t n_pos, int32_t d, double base, void* stream) {
  using namespace ra;
  clear_error();
  if (!table || n_pos < 1 || d < 2 || d % 4 != 0 || !(base > 1.0)) {
    set_error("refadapt_rope_table: table NULL, n_pos < 1, d not a multiple of 4 or base <= 1");
    return RA_EINVAL;
  }
  const int64_t n = int64_t(n_pos) * (d / 2);
  const int blocks = int((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  gemm::rope_table_kernel<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(table, n_pos, d, base);
  return launch_status("refadapt_rope_table");
}

extern "C" ra_status refadapt_gemm(const ra_gemm_args* a, void* stream) {
  using namespace ra;
  using namespace ra::gemm;
  clear_error();
  if (!a) {
    set_error("refadapt_gemm: args is NULL");
    return RA_EINVAL;
  }
  if (a->B < 1 || a->n_seg < 1 || a->n_seg > 3 || a->K < BK || a->K % BK != 0 || a->N < BN || a->N % BN != 0) {
    set_error("refadapt_gemm: need B >= 1, 1 <= n_seg <= 3, K a positive multiple of 64, N of 256 "
              "(B=%d n_seg=%d N=%d K=%d)", a->B, a->n_seg, a->N, a->K);
    return RA_EINVAL;
  }
  if (a->epilogue < RA_EPI_STORE || a->epilogue > RA_EPI_QKV) {
    set_error("refadapt_gemm: unknown epilogue %d", a->epilogue);
    return RA_EINVAL;
  }
  Params p;
  std::memset(&p, 0, sizeof(p));
  p.n_seg = a->n_seg;
  p.B = a->B;
  p.N = a->N;
  p.K = a->K;
  p.epi = a->epilogue;
  p.n_tiles_n = a->N / BN;
  p.kblocks = a->K / BK;
  p.mode = a->mode;
  p.err_word = a->err_word;
  p.budget_ns = wait_budget_ns();
  p.norm_eps = a->norm_eps;
  if (a->epilogue == RA_EPI_QKV) {
    if ((a->d != 64 && a->d != 128) || a->H < 1 || int64_t(3) * a->H * a->d != a->N || (a->H * a->d) % BN != 0) {
      set_error("refadapt_gemm: QKV needs d in {64, 128}, N = 3 H d and H d a multiple of 256");
      return RA_EINVAL;
    }
    if (!a->rope || !aligned16(a->rope) || a->rope_len < 1 || !(a->norm_eps >= 0.f)) {
      set_error("refadapt_gemm: QKV needs a 16-byte aligned rope table, rope_len >= 1 and norm_eps >= 0");
      return RA_EINVAL;
    }
    p.H = a->H;
    p.d = a->d;
    p.C = a->H * a->d;
    p.rope = reinterpret_cast<const float4*>(a->rope);
    p.rope_len = a->rope_len;
  }
  if (a->tile_mode < 0 || a->tile_mode > 2) {
    set_error("refadapt_gemm: tile_mode %d (0 auto, 1 one CTA per tile, 2 CTA pairs)", a->tile_mode);
    return RA_EINVAL;
  }
  // One CTA per 128-row tile, or CTA pairs on 256-row tiles when there is a
  // full wave of pair tiles (auto) or when asked.
  int64_t pair_tiles = 0;
  for (int g = 0; g < a->n_seg; ++g)
    if (a->seg[g].rows > 0) pair_tiles += int64_t(a->B) * ((a->seg[g].rows + P_TM - 1) / P_TM) * p.n_tiles_n;
  const int sms = num_sms();
  const bool pair = a->tile_mode == 2 || (a->tile_mode == 0 && sms >= 2 && pair_tiles >= sms / 2);
  const int tm = pair ? P_TM : BM;
  int64_t tiles = 0;
  for (int g = 0; g < a->n_seg; ++g) {
    const ra_gemm_seg& s = a->seg[g];
    Seg& d = p.seg[g];
    if (s.rows < 0) {
      set_error("refadapt_gemm: seg %d rows < 0", g);
      return RA_EINVAL;
    }
    d.tile_begin = tiles;
    d.rows = s.rows;
    d.m_tiles = (s.rows + tm - 1) / tm;
    d.gated = s.gated ? 1 : 0;
    d.pos_offset = s.pos_offset;
    d.bias = s.bias;
    if (s.gated && !a->mode) {
      set_error("refadapt_gemm: seg %d is gated but mode is NULL", g);
      return RA_EINVAL;
    }
    if (s.rows == 0) continue;
    if (!s.a || !s.w || !aligned16(s.a) || !aligned16(s.w) || s.a_stride_r % 8 != 0 || s.a_stride_s % 8 != 0 ||
        s.a_stride_r < a->K || s.a_stride_s < 0) {
      set_error("refadapt_gemm: seg %d: A and W must be 16-byte aligned, strides multiples of 8 elements, "
                "a_stride_r >= K", g);
      return RA_EINVAL;
    }
    if (s.bias && !aligned16(s.bias)) {
      set_error("refadapt_gemm: seg %d: bias must be 16-byte aligned", g);
      return RA_EINVAL;
    }
    if (a->epilogue == RA_EPI_QKV) {
      const ra_seg* dst[3] = {&s.q_out, &s.k_out, &s.v_out};
      const char* nm[3] = {"q_out", "k_out", "v_out"};
      for (int z = 0; z < 3; ++z) {
        if (dst[z]->n != s.rows || !check_seg(*dst[z], nm[z], false)) {
          if (dst[z]->n != s.rows) set_error("refadapt_gemm: seg %d: %s.n must equal rows", g, nm[z]);
          return RA_EINVAL;
        }
        d.dst[z] = static_cast<__nv_bfloat16*>(dst[z]->ptr);
        d.dst_sb[z] = dst[z]->stride_b;
        d.dst_sh[z] = dst[z]->stride_h;
        d.dst_sn[z] = dst[z]->stride_n;
      }
      if (!s.q_norm || !s.k_norm || !aligned16(s.q_norm) || !aligned16(s.k_norm)) {
        set_error("refadapt_gemm: seg %d: QKV needs 16-byte aligned q_norm and k_norm", g);
        return RA_EINVAL;
      }
      if (s.pos_offset < 0 || int64_t(s.pos_offset) + s.rows > a->rope_len) {
        set_error("refadapt_gemm: seg %d: positions [%d, %d) outside the rope table (%d)", g, s.pos_offset,
                  s.pos_offset + s.rows, a->rope_len);
        return RA_EINVAL;
      }
      d.norm_w[0] = s.q_norm;
      d.norm_w[1] = s.k_norm;
    } else {
      if (!s.out || !aligned16(s.out) || s.out_stride_r % 8 != 0 || s.out_stride_s % 8 != 0 ||
          s.out_stride_r < a->N) {
        set_error("refadapt_gemm: seg %d: out must be 16-byte aligned with strides multiples of 8 elements, "
                  "out_stride_r >= N", g);
        return RA_EINVAL;
      }
      d.out = static_cast<__nv_bfloat16*>(s.out);
      d.out_ss = s.out_stride_s;
      d.out_sr = s.out_stride_r;
      if (a->epilogue == RA_EPI_RESID) {
        if (!s.resid || !s.gate || !aligned16(s.resid) || !aligned16(s.gate) || s.resid_stride_r % 8 != 0 ||
            s.resid_stride_s % 8 != 0 || s.gate_stride_s % 4 != 0) {
          set_error("refadapt_gemm: seg %d: RESID needs 16-byte aligned resid and gate, resid strides "
                    "multiples of 8 elements, gate_stride_s of 4", g);
          return RA_EINVAL;
        }
        d.resid = static_cast<const __nv_bfloat16*>(s.resid);
        d.res_ss = s.resid_stride_s;
        d.res_sr = s.resid_stride_r;
        d.gate = s.gate;
        d.gate_ss = s.gate_stride_s;
      }
    }
    ra_seg as{const_cast<void*>(s.a), s.a_stride_s, 0, s.a_stride_r, s.rows, 0};
    ra_seg ws{const_cast<void*>(s.w), 0, 0, a->K, a->N, 0};
      // The pair kernel loads 128-row boxes of A and of W (each CTA its half).
    if (!encode_seg(&p.tm_a[g], as, a->B, 1, a->K, BK, BM, true) ||
        !encode_seg(&p.tm_w[g], ws, 1, 1, a->K, BK, pair ? 128 : BN, true))
      return RA_EINVAL;
    tiles += int64_t(a->B) * d.m_tiles * p.n_tiles_n;
  }
  p.total_tiles = tiles;
  if (tiles == 0) return RA_OK;
  ra_status as = ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_kernel), SMEM_ALLOC, "refadapt_gemm");
  if (as == RA_OK)
    as = ensure_dynamic_smem(reinterpret_cast<const void*>(gemm_pair_kernel), P_SMEM_ALLOC, "refadapt_gemm");
  if (as != RA_OK) return as;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (!pair) {
    const int64_t grid = tiles < sms ? tiles : sms;
    gemm_kernel<<<unsigned(grid), THREADS, SMEM_ALLOC, st>>>(p);
    return launch_status("refadapt_gemm");
  }
  const int64_t clusters = tiles < sms / 2 ? tiles : (sms / 2 > 0 ? sms / 2 : 1);
  cudaLaunchConfig_t cfg;
  std::memset(&cfg, 0, sizeof(cfg));
  cfg.gridDim = dim3(unsigned(2 * clusters), 1, 1);
  cfg.blockDim = dim3(THREADS, 1, 1);
  cfg.dynamicSmemBytes = P_SMEM_ALLOC;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, gemm_pair_kernel, p);
  if (e != cudaSuccess) {
    set_error("refadapt_gemm: pair launch failed: %s", cudaGetErrorString(e));
    cudaGetLastError();
    return RA_ECUDA;
  }
  return launch_status("refadapt_gemm");
}
