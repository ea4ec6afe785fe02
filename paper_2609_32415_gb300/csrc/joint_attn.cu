// refadapt_joint_attn: joint [text; reference; target] attention with the
// per-tile reference mass, on tcgen05 tensor cores (sm_103a).
//
// One CTA computes one 128-row Q tile of one role for one (sample, head):
//   warp 0      TMA producer: the Q tile once, then K and V tiles of the text,
//               reference (cache slot) and target segments in that order,
//               into a STAGES-deep ring of 128-byte-swizzled shared buffers.
//   warp 1      TMEM allocator and MMA issuer (one thread): S_j = Q K_j^T into
//               one of two TMEM S buffers (kind::f16, fp32 accumulate), then
//               O += P_j V_j with P_j read from TMEM (it overwrites the first
//               64 columns of S_j as packed bf16). S_{j+1} is issued before
//               O += P_j V_j so the tensor core works while softmax j runs.
//   warps 2..5  softmax / epilogue: thread = query row = TMEM lane. Online
//               softmax in log2 units with a lazy rescale (the running max is
//               only moved when a tile's max exceeds it by more than 2^8), the
//               row sum l and the reference-only row sum l_ref (paper Eq. 4's
//               inner sum is l_ref / l), then O / l -> bf16 global, and the
//               tile's sum of l_ref / l over mass rows -> mass_partial.
// Segment tails: TMA zero-fills rows past a segment's end; the softmax masks
// those key columns to probability 0 and the epilogue skips those query rows.
// Every mbarrier wait is bounded (WaitCtl); on a timeout the CTA drains its own
// TMA and MMA work, frees TMEM, flags the caller's error word and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "api_common.h"
#include "tc_ptx.cuh"

namespace ra {
namespace attn {

constexpr int BM = 128;  // query rows per tile (= TMEM lanes)
constexpr int BN = 128;  // keys per tile
constexpr int NUM_THREADS = 192;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleThresh = 8.0f;  // log2 units: p <= 2^8 between rescales

template <int D>
struct Cfg {
  static constexpr int CHUNKS = D / 64;           // 64-element (128-byte) swizzle chunks per row
  static constexpr int CHUNK_BYTES = BM * 128;    // one chunk of a 128-row tile
  static constexpr int TILE_BYTES = BM * D * 2;   // Q, K or V tile (BN == BM)
  static constexpr int STAGES = (D == 128) ? 2 : 4;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + TILE_BYTES;
  static constexpr int OFF_V = OFF_K + STAGES * TILE_BYTES;
  static constexpr int OFF_BAR = OFF_V + STAGES * TILE_BYTES;
  // q_full, k_full[S], k_empty[S], v_full[S], v_empty[S], s_full[2], p_ready[2], o_done, drain
  static constexpr int NUM_BARS = 1 + 4 * STAGES + 2 + 2 + 1 + 1;
  static constexpr int OFF_MISC = OFF_BAR + NUM_BARS * 8;  // tmem slot, abort flag, 4 floats
  static constexpr int SMEM_BYTES = OFF_MISC + 64;
  static constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;  // slack for 1024-byte alignment
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t TM_S0 = 0, TM_S1 = 128, TM_O = 256;
  static_assert(SMEM_ALLOC <= 232448, "shared memory budget");
};

struct alignas(64) Params {
  CUtensorMap tm_q[3];
  CUtensorMap tm_k[3];
  CUtensorMap tm_v[3];
  __nv_bfloat16* o_ptr[3];
  int64_t o_sb[3], o_sh[3], o_sn[3];
  int32_t n[3];
  int32_t q_tiles[3];
  int32_t kv_tiles[3];
  int32_t B, H;
  int32_t mass_rows;
  int32_t mpl;
  float scale_log2;
  const float* bias;
  const int32_t* mode;
  float* mass_partial;
  int32_t* err_word;
  uint64_t budget_ns;
};

__device__ __forceinline__ void kv_tile(const Params& p, int j, int& r, int& row0) {
  if (j < p.kv_tiles[0]) {
    r = 0;
    row0 = j * BN;
  } else if (j < p.kv_tiles[0] + p.kv_tiles[1]) {
    r = 1;
    row0 = (j - p.kv_tiles[0]) * BN;
  } else {
    r = 2;
    row0 = (j - p.kv_tiles[0] - p.kv_tiles[1]) * BN;
  }
}

template <int D>
__global__ void __launch_bounds__(NUM_THREADS, 1) joint_attn_kernel(const __grid_constant__ Params p) {
  using C = Cfg<D>;
  constexpr int S = C::STAGES;
  const int b = blockIdx.z, h = blockIdx.y;
  int qt = blockIdx.x, role;
  if (qt < p.q_tiles[0]) {
    role = 0;
  } else if (qt - p.q_tiles[0] < p.q_tiles[1]) {
    qt -= p.q_tiles[0];
    role = 1;
  } else {
    qt -= p.q_tiles[0] + p.q_tiles[1];
    role = 2;
  }
  const int mode = p.mode ? __ldg(p.mode + b) : int(RA_MODE_FULL);
  if (role == 1 && mode == RA_MODE_REUSE) return;  // reference rows skipped (uniform exit)

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;
  uint64_t* k_empty = bars + 1 + S;
  uint64_t* v_full = bars + 1 + 2 * S;
  uint64_t* v_empty = bars + 1 + 3 * S;
  uint64_t* s_full = bars + 1 + 4 * S;
  uint64_t* p_ready = bars + 3 + 4 * S;
  uint64_t* o_done = bars + 5 + 4 * S;
  uint64_t* drain = bars + 6 + 4 * S;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  float* red = reinterpret_cast<float*>(smem + C::OFF_MISC + 16);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < S; ++s) {
      mbar_init(k_full + s, 1);
      mbar_init(k_empty + s, 1);
      mbar_init(v_full + s, 1);
      mbar_init(v_empty + s, 1);
    }
    mbar_init(s_full, 1);
    mbar_init(s_full + 1, 1);
    mbar_init(p_ready, 128);
    mbar_init(p_ready + 1, 128);
    mbar_init(o_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const WaitCtl ctl{abort_flag, p.err_word, p.budget_ns};
  const int nkv = p.kv_tiles[0] + p.kv_tiles[1] + p.kv_tiles[2];

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      tma_prefetch_desc(&p.tm_q[role]);
      for (int r = 0; r < 3; ++r)
        if (p.kv_tiles[r] > 0) {
          tma_prefetch_desc(&p.tm_k[r]);
          tma_prefetch_desc(&p.tm_v[r]);
        }
      int k_issued[S], v_issued[S];
      for (int s = 0; s < S; ++s) k_issued[s] = v_issued[s] = 0;
      mbar_arrive_expect_tx(q_full, C::TILE_BYTES);
      for (int c = 0; c < C::CHUNKS; ++c)
        tma_load_4d(smem + C::OFF_Q + c * C::CHUNK_BYTES, &p.tm_q[role], q_full, c * 64, qt * BM, h, b);
      for (int j = 0; j < nkv; ++j) {
        const int s = j % S;
        const uint32_t ph = (j / S) & 1;
        int r, row0;
        kv_tile(p, j, r, row0);
        if (j >= S && !mbar_wait(k_empty + s, ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(k_full + s, C::TILE_BYTES);
        for (int c = 0; c < C::CHUNKS; ++c)
          tma_load_4d(smem + C::OFF_K + s * C::TILE_BYTES + c * C::CHUNK_BYTES, &p.tm_k[r], k_full + s,
                      c * 64, row0, h, b);
        ++k_issued[s];
        if (j >= S && !mbar_wait(v_empty + s, ph ^ 1, ctl)) break;
        mbar_arrive_expect_tx(v_full + s, C::TILE_BYTES);
        for (int c = 0; c < C::CHUNKS; ++c)
          tma_load_4d(smem + C::OFF_V + s * C::TILE_BYTES + c * C::CHUNK_BYTES, &p.tm_v[r], v_full + s,
                      c * 64, row0, h, b);
        ++v_issued[s];
      }
      if (*abort_flag) {
        // Let every load this thread issued land before the CTA exits.
        mbar_wait_drain(q_full, 0, p.budget_ns);
        for (int s = 0; s < S; ++s) {
          if (k_issued[s] > 0) mbar_wait_drain(k_full + s, (k_issued[s] - 1) & 1, p.budget_ns);
          if (v_issued[s] > 0) mbar_wait_drain(v_full + s, (v_issued[s] - 1) & 1, p.budget_ns);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      constexpr uint32_t IDESC_QK = idesc_bf16_f32(BM, BN, 0, 0);  // Q, K both K-major
      constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, D, 0, 1);   // P K-major (TMEM), V MN-major
      const uint32_t sq = smem_u32(smem + C::OFF_Q);
      const uint32_t sk = smem_u32(smem + C::OFF_K);
      const uint32_t sv = smem_u32(smem + C::OFF_V);
      bool issued_any = false;
      auto issue_qk = [&](int j) -> bool {
        const int s = j % S;
        if (!mbar_wait(k_full + s, (j / S) & 1, ctl)) return false;
        tc_fence_after();
        const uint32_t d_t = tmem + ((j & 1) ? C::TM_S1 : C::TM_S0);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * C::CHUNK_BYTES + (kk & 3) * 32;
          umma_ss(d_t, sdesc_sw128(sq + off, 16, 1024), sdesc_sw128(sk + s * C::TILE_BYTES + off, 16, 1024),
                  IDESC_QK, kk > 0 ? 1u : 0u);
        }
        issued_any = true;
        umma_commit(s_full + (j & 1));
        umma_commit(k_empty + s);
        return true;
      };
      bool ok = mbar_wait(q_full, 0, ctl);
      if (ok) {
        tc_fence_after();
        ok = issue_qk(0);
      }
      for (int j = 0; ok && j < nkv; ++j) {
        if (j + 1 < nkv && !(ok = issue_qk(j + 1))) break;
        if (!(ok = mbar_wait(p_ready + (j & 1), (j >> 1) & 1, ctl))) break;
        const int s = j % S;
        if (!(ok = mbar_wait(v_full + s, (j / S) & 1, ctl))) break;
        tc_fence_after();
        const uint32_t p_t = tmem + ((j & 1) ? C::TM_S1 : C::TM_S0);
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk) {
          umma_ts(tmem + C::TM_O, p_t + kk * 8,
                  sdesc_sw128(sv + s * C::TILE_BYTES + kk * 16 * 128, C::CHUNK_BYTES, 1024), IDESC_PV,
                  (j > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(v_empty + s);
        umma_commit(o_done);
      }
      if (!ok && issued_any) {
        umma_commit(drain);
        mbar_wait_drain(drain, 0, p.budget_ns);
      }
    }
  } else {
    // -------------------------------------------------------------- softmax
    const int quarter = warp & 3;  // TMEM lane quarter this warp may access
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    const float sl2 = p.scale_log2;
    const float bias_l2 = (role == 2 && p.bias) ? __ldg(p.bias + h) * kLog2e : 0.f;
    float m = -INFINITY, l = 0.f, lref = 0.f;
    bool ok = true;
    for (int j = 0; j < nkv; ++j) {
      int r, row0;
      kv_tile(p, j, r, row0);
      const int nvalid = min(BN, p.n[r] - row0);
      const float badd = (r == 1) ? bias_l2 : 0.f;
      ok = __all_sync(0xffffffffu, mbar_wait(s_full + (j & 1), (j >> 1) & 1, ctl));
      if (!ok) break;
      tc_fence_after();
      const uint32_t s_t = tmem + lane_off + ((j & 1) ? C::TM_S1 : C::TM_S0);
      uint32_t sa[32], sb[32], sc[32], sd[32];
      tmem_ld32(s_t + 0, sa);
      tmem_ld32(s_t + 32, sb);
      tmem_ld32(s_t + 64, sc);
      tmem_ld32(s_t + 96, sd);
      tmem_ld_wait();
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        if (c < nvalid) mx = fmaxf(mx, __uint_as_float(sa[c]));
        if (c + 32 < nvalid) mx = fmaxf(mx, __uint_as_float(sb[c]));
        if (c + 64 < nvalid) mx = fmaxf(mx, __uint_as_float(sc[c]));
        if (c + 96 < nvalid) mx = fmaxf(mx, __uint_as_float(sd[c]));
      }
      const float mt = fmaf(mx, sl2, badd);  // tile max, log2 units
      float alpha = 1.f;
      bool resc = false;
      if (mt > m + kRescaleThresh) {
        alpha = ex2_approx(m - mt);  // 0 when m = -inf
        resc = (j > 0);
        l *= alpha;
        lref *= alpha;
        m = mt;
      }
      const float negm = badd - m;
      float rs = 0.f;
      uint32_t pa[32], pb[32];
#pragma unroll
      for (int c = 0; c < 16; ++c) {
        const float x0 = (2 * c < nvalid) ? ex2_approx(fmaf(__uint_as_float(sa[2 * c]), sl2, negm)) : 0.f;
        const float x1 = (2 * c + 1 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sa[2 * c + 1]), sl2, negm)) : 0.f;
        const float y0 = (2 * c + 32 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sb[2 * c]), sl2, negm)) : 0.f;
        const float y1 =
            (2 * c + 33 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sb[2 * c + 1]), sl2, negm)) : 0.f;
        const float z0 = (2 * c + 64 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sc[2 * c]), sl2, negm)) : 0.f;
        const float z1 =
            (2 * c + 65 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sc[2 * c + 1]), sl2, negm)) : 0.f;
        const float w0 = (2 * c + 96 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sd[2 * c]), sl2, negm)) : 0.f;
        const float w1 =
            (2 * c + 97 < nvalid) ? ex2_approx(fmaf(__uint_as_float(sd[2 * c + 1]), sl2, negm)) : 0.f;
        rs += (x0 + x1) + (y0 + y1) + (z0 + z1) + (w0 + w1);
        pa[c] = pack_bf16x2(x0, x1);
        pa[c + 16] = pack_bf16x2(y0, y1);
        pb[c] = pack_bf16x2(z0, z1);
        pb[c + 16] = pack_bf16x2(w0, w1);
      }
      l += rs;
      if (r == 1) lref += rs;
      if (__any_sync(0xffffffffu, resc)) {
        ok = __all_sync(0xffffffffu, mbar_wait(o_done, (j - 1) & 1, ctl));
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t ov[32];
          tmem_ld32(tmem + lane_off + C::TM_O + c0, ov);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * alpha);
          tmem_st32(tmem + lane_off + C::TM_O + c0, ov);
        }
      }
      tmem_st32(s_t + 0, pa);
      tmem_st32(s_t + 32, pb);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(p_ready + (j & 1));
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_done, (nkv - 1) & 1, ctl));
    const int grow = qt * BM + row;
    const bool valid = grow < p.n[role];
    const float inv_l = 1.f / l;
    if (ok) {
      tc_fence_after();
      __nv_bfloat16* orow = p.o_ptr[role] + b * p.o_sb[role] + h * p.o_sh[role] + int64_t(grow) * p.o_sn[role];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t ov[32];
        tmem_ld32(tmem + lane_off + C::TM_O + c0, ov);
        tmem_ld_wait();
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 16; ++i)
          pk[i] = pack_bf16x2(__uint_as_float(ov[2 * i]) * inv_l, __uint_as_float(ov[2 * i + 1]) * inv_l);
        if (valid) {
          uint4* dst = reinterpret_cast<uint4*>(orow + c0);
          dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          dst[2] = make_uint4(pk[8], pk[9], pk[10], pk[11]);
          dst[3] = make_uint4(pk[12], pk[13], pk[14], pk[15]);
        }
      }
    }
    // Per-tile mass partial: sum over the tile's mass rows of l_ref / l, in a
    // fixed order (warp butterfly, then quarters 0..3).
    const bool in_mass = (role == 2) || (role == 0 && p.mass_rows == 1);
    float mv = (ok && valid && in_mass) ? lref * inv_l : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mv += __shfl_xor_sync(0xffffffffu, mv, o);
    if (lane == 0) red[quarter] = mv;
    named_bar_sync(1, 128);
    if (ok && role != 1 && quarter == 0 && lane == 0) {
      const int idx = (role == 0) ? qt : p.q_tiles[0] + qt;
      p.mass_partial[(int64_t(b) * p.H + h) * p.mpl + idx] = ((red[0] + red[1]) + red[2]) + red[3];
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 4-D map (d, n, head, sample) over one bf16 segment, box 64 x box_rows, 128-byte swizzle.
bool encode_seg(CUtensorMap* tm, const ra_seg& s, int B, int H, int d, int box_rows) {
  auto fn = encode_fn();
  if (!fn) {
    set_error("cuTensorMapEncodeTiled unavailable from the driver");
    return false;
  }
  const int64_t row_bytes = int64_t(s.stride_n) * 2;
  int64_t sh = int64_t(s.stride_h) * 2, sb = int64_t(s.stride_b) * 2;
  // A stride of a size-1 dimension is never used; give TMA a legal one.
  if (H == 1 && sh == 0) sh = row_bytes * (s.n > 0 ? s.n : 1);
  if (B == 1 && sb == 0) sb = sh * H;
  if (row_bytes == 0 && s.n > 1) {
    set_error("segment row stride is 0");
    return false;
  }
  cuuint64_t dims[4] = {cuuint64_t(d), cuuint64_t(s.n), cuuint64_t(H), cuuint64_t(B)};
  cuuint64_t strides[3] = {cuuint64_t(row_bytes > 0 ? row_bytes : 16 * ((d * 2 + 15) / 16)), cuuint64_t(sh),
                           cuuint64_t(sb)};
  cuuint32_t box[4] = {64u, cuuint32_t(box_rows), 1u, 1u};
  cuuint32_t es[4] = {1u, 1u, 1u, 1u};
  CUresult r = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, s.ptr, dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (%d)", int(r));
    return false;
  }
  return true;
}

template <int D>
ra_status launch(const Params& p, dim3 grid, cudaStream_t st) {
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(joint_attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    Cfg<D>::SMEM_ALLOC);
  });
  if (attr_err != cudaSuccess) {
    set_error("refadapt_joint_attn: cudaFuncSetAttribute: %s", cudaGetErrorString(attr_err));
    return RA_ECUDA;
  }
  joint_attn_kernel<D><<<grid, NUM_THREADS, Cfg<D>::SMEM_ALLOC, st>>>(p);
  return launch_status("refadapt_joint_attn");
}

}  // namespace attn
}  // namespace ra

extern "C" int32_t refadapt_mass_partial_len(int32_t n_text, int32_t n_tgt) {
  if (n_text < 0 || n_tgt < 0) return 0;
  return (n_text + RA_MASS_TILE_ROWS - 1) / RA_MASS_TILE_ROWS + (n_tgt + RA_MASS_TILE_ROWS - 1) / RA_MASS_TILE_ROWS;
}

extern "C" ra_status refadapt_joint_attn(const ra_attn_args* a, void* stream) {
  using namespace ra;
  using namespace ra::attn;
  clear_error();
  if (!a) {
    set_error("refadapt_joint_attn: args is NULL");
    return RA_EINVAL;
  }
  if (a->d != 64 && a->d != 128) {
    set_error("refadapt_joint_attn: d = %d (supported: 64, 128)", a->d);
    return RA_EINVAL;
  }
  if (a->B < 1 || a->H < 1 || a->B > 65535 || a->H > 65535) {
    set_error("refadapt_joint_attn: B = %d, H = %d out of range", a->B, a->H);
    return RA_EINVAL;
  }
  if (a->mass_rows != 0 && a->mass_rows != 1) {
    set_error("refadapt_joint_attn: mass_rows must be 0 or 1");
    return RA_EINVAL;
  }
  if (!(a->softmax_scale >= 0.f) || std::isinf(a->softmax_scale)) {
    set_error("refadapt_joint_attn: softmax_scale must be finite and >= 0");
    return RA_EINVAL;
  }
  if (!a->mass_partial) {
    set_error("refadapt_joint_attn: mass_partial is NULL");
    return RA_EINVAL;
  }
  static const char* names[3] = {"text", "ref", "tgt"};
  char what[64];
  Params p;
  std::memset(&p, 0, sizeof(p));
  const int n_ref = a->k[RA_REF].n;
  bool ref_rows = true;
  for (int r = 0; r < 3; ++r) {
    const int n = a->k[r].n;
    if (a->q[r].n != n || a->v[r].n != n || a->o[r].n != n) {
      set_error("refadapt_joint_attn: %s segments disagree on n", names[r]);
      return RA_EINVAL;
    }
    const ra_seg* segs[4] = {&a->q[r], &a->k[r], &a->v[r], &a->o[r]};
    const char* kinds[4] = {"q", "k", "v", "o"};
    for (int i = 0; i < 4; ++i) {
      snprintf(what, sizeof(what), "refadapt_joint_attn: %s[%s]", kinds[i], names[r]);
      const bool may_skip = (r == RA_REF) && (i == 0 || i == 3);
      if (may_skip && segs[i]->ptr == nullptr) {
        ref_rows = false;
        continue;
      }
      if (!check_seg(*segs[i], what)) return RA_EINVAL;
    }
  }
  if (a->k[RA_TGT].n < 1) {
    set_error("refadapt_joint_attn: n_tgt must be >= 1");
    return RA_EINVAL;
  }
  const int d = a->d;
  for (int r = 0; r < 3; ++r) {
    const int n = a->k[r].n;
    p.n[r] = n;
    p.kv_tiles[r] = (n + BN - 1) / BN;
    p.q_tiles[r] = (n + BM - 1) / BM;
    if (n == 0) continue;
    if (!encode_seg(&p.tm_k[r], a->k[r], a->B, a->H, d, BN) || !encode_seg(&p.tm_v[r], a->v[r], a->B, a->H, d, BN))
      return RA_EINVAL;
    if (r == RA_REF && !ref_rows) {
      p.q_tiles[r] = 0;
      continue;
    }
    if (!encode_seg(&p.tm_q[r], a->q[r], a->B, a->H, d, BM)) return RA_EINVAL;
    p.o_ptr[r] = static_cast<__nv_bfloat16*>(a->o[r].ptr);
    p.o_sb[r] = a->o[r].stride_b;
    p.o_sh[r] = a->o[r].stride_h;
    p.o_sn[r] = a->o[r].stride_n;
  }
  (void)n_ref;
  p.B = a->B;
  p.H = a->H;
  p.mass_rows = a->mass_rows;
  p.mpl = refadapt_mass_partial_len(a->k[RA_TEXT].n, a->k[RA_TGT].n);
  const float scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / std::sqrt(float(d));
  p.scale_log2 = scale * kLog2e;
  p.bias = a->ref_logit_bias;
  p.mode = a->mode;
  p.mass_partial = a->mass_partial;
  p.err_word = a->err_word;
  p.budget_ns = wait_budget_ns();
  const int tiles = p.q_tiles[0] + p.q_tiles[1] + p.q_tiles[2];
  dim3 grid(tiles, a->H, a->B);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return d == 128 ? launch<128>(p, grid, st) : launch<64>(p, grid, st);
}
