// refadapt_joint_attn: joint [text; reference; target] attention with the
// per-tile reference mass, on tcgen05 tensor cores (sm_103a).
//
// One CTA computes a pair of 128-row Q tiles (A, B) of one role for one
// (sample, head); both tiles share every K/V tile it streams:
//   warp 0      TMA producer: Q tiles A and B once, then K and V tiles of the
//               text, reference (cache slot) and target segments in that order
//               into a STAGES-deep ring of 128-byte-swizzled shared buffers.
//   warp 1      TMEM allocator and MMA issuer (one thread). TMEM columns:
//               S_A [0,128), S_B [128,256), O_A [256,..), O_B [384,..).
//               S_t = Q_t K_j^T (kind::f16, fp32 accumulate); P_t is written
//               back over the first 64 columns of S_t as packed bf16 and read
//               from TMEM as the A operand of O_t += P_t V_j. Issue order per
//               key tile: PV_A(j), QK_A(j+1), PV_B(j), QK_B(j+1), so the tensor
//               core works on one tile while the other tile's softmax runs.
//               Each product's K steps leave one asm block (one predicate,
//               descriptors advanced by immediates): the issuing warp shares
//               its SM sub-partition with two softmax warps, and the MMA rate
//               follows the issuing thread's instruction count.
//   warps 2, 3  idle (they complete warpgroup 0, which hands registers over:
//               setmaxnreg 56 there, 224 in the softmax warpgroups; 4 x 56 +
//               8 x 224 = 12 x 168, the launch allocation).
//   warps 4..7  softmax / epilogue of tile A, warps 8..11 of tile B: thread =
//               query row = TMEM lane (lane quarter = warp % 4). Online softmax
//               in log2 units with a lazy rescale (the running max only moves
//               when a tile's max exceeds it by more than 2^8), the row sum l
//               and the reference-only row sum l_ref (paper Eq. 4's inner sum
//               is l_ref / l); then O / l -> bf16 global and the tile's sum of
//               l_ref / l over its mass rows -> mass_partial.
// Fused reference-cache update (paper Eq. 11), when the caller passes this
// step's reference projections: samples in COMPUTE or FULL read reference
// Q/K/V from them, and the producer thread copies what it streams into the
// cache slot with TMA bulk-tensor stores from the swizzled stage buffers. The
// first CTA of each (sample, head) stores every reference K/V tile one tile
// after its load (the stage is refilled only once the store has read it);
// each reference-row CTA stores its two Q tiles. Each byte of the fresh
// reference rows is read from HBM once for both the MMAs and the copy.
// Segment tails: TMA zero-fills rows past a segment's end; tail key tiles mask
// the padded columns to -inf (probability 0) and the epilogue skips padded
// query rows; TMA stores clip rows past a segment's end. Every mbarrier wait is bounded (WaitCtl); on a timeout the CTA
// drains its own TMA and MMA work, frees TMEM, flags the caller's error word
// and returns.
#include <cuda.h>
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
constexpr int NUM_THREADS = 384;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleThresh = 8.0f;  // log2 units: p <= 2^8 between rescales

template <int D>
struct Cfg {
  static constexpr int CHUNKS = D / 64;           // 64-element (128-byte) swizzle chunks per row
  static constexpr int CHUNK_BYTES = BM * 128;    // one chunk of a 128-row tile
  static constexpr int TILE_BYTES = BM * D * 2;   // one Q, K or V tile (BN == BM)
  static constexpr int STAGES = (D == 128) ? 2 : 4;
  static constexpr int OFF_Q = 0;                 // Q tiles A and B
  static constexpr int OFF_K = OFF_Q + 2 * TILE_BYTES;
  static constexpr int OFF_V = OFF_K + STAGES * TILE_BYTES;
  static constexpr int OFF_BAR = OFF_V + STAGES * TILE_BYTES;
  // q_full, k_full[S], k_empty[S], v_full[S], v_empty[S], s_full[2], p_ready[2], o_done[2], drain
  static constexpr int NUM_BARS = 1 + 4 * STAGES + 2 + 2 + 2 + 1;
  static constexpr int OFF_MISC = OFF_BAR + NUM_BARS * 8;  // tmem slot, abort flag, 8 floats
  static constexpr int SMEM_BYTES = OFF_MISC + 64;
  static constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;  // slack for 1024-byte alignment
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr uint32_t TM_S = 0, TM_O = 256;       // + 128 * tile
  static_assert(SMEM_ALLOC <= 232448, "shared memory budget");
};

struct Params {
  CUtensorMap tm_q[3];
  CUtensorMap tm_k[3];
  CUtensorMap tm_v[3];
  CUtensorMap tm_qf, tm_kf, tm_vf;  // this step's reference rows (fused cache update)
  __nv_bfloat16* o_ptr[3];
  int64_t o_sb[3], o_sh[3], o_sn[3];
  int32_t nq[3];  // query rows per role
  int32_t nk[3];  // key rows per role
  int32_t q_tiles[3];
  int32_t q_blocks[3];  // pairs of Q tiles
  int32_t kv_tiles[3];
  int32_t B, H;
  int32_t mass_rows;
  int32_t mass_stride;  // count mass rows 0, k, 2k, ... (k <= 1: every row)
  int32_t mpl;
  float scale_log2;
  const float* bias;
  const int32_t* mode;
  float* mass_partial;
  int32_t* err_word;
  int32_t* a_b;
  int32_t step;
  int32_t fresh;     // refreshing samples read reference rows from tm_*f
  int32_t store_kv;  // ... and copy those K / V tiles into tm_k[1] / tm_v[1]
  int32_t store_q;   // ... and those Q tiles into tm_q[1]
  uint64_t budget_ns;
};

__device__ __forceinline__ bool refreshes(int m) { return m == RA_MODE_COMPUTE || m == RA_MODE_FULL; }

// Tile (c0 = column, c1 = row, c2 = head, c3 = sample) of a 4-D tensor map,
// shared -> global, bulk-group completion; rows past the tensor are clipped.
__device__ __forceinline__ void tma_store_4d(const void* tmap, const void* src, int32_t c0, int32_t c1,
                                             int32_t c2, int32_t c3) {
  asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%2, %3, %4, %5}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Shared memory written by TMA loads (async proxy) is next read by TMA stores.
__device__ __forceinline__ void fence_proxy_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

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

// Row maximum over the 64 logits in v[] (columns col0 .. col0+63 of the tile);
// TAIL ignores columns >= nvalid.
template <bool TAIL>
__device__ __forceinline__ float max64(const float (&v)[64], int col0, int nvalid, float m_in) {
  float m0 = m_in, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
#pragma unroll
  for (int c = 0; c < 64; c += 8) {
    if (TAIL) {
      const int e = col0 + c;
      m0 = fmax3f(m0, (e < nvalid) ? v[c] : -INFINITY, (e + 1 < nvalid) ? v[c + 1] : -INFINITY);
      m1 = fmax3f(m1, (e + 2 < nvalid) ? v[c + 2] : -INFINITY, (e + 3 < nvalid) ? v[c + 3] : -INFINITY);
      m2 = fmax3f(m2, (e + 4 < nvalid) ? v[c + 4] : -INFINITY, (e + 5 < nvalid) ? v[c + 5] : -INFINITY);
      m3 = fmax3f(m3, (e + 6 < nvalid) ? v[c + 6] : -INFINITY, (e + 7 < nvalid) ? v[c + 7] : -INFINITY);
    } else {
      m0 = fmax3f(m0, v[c], v[c + 1]);
      m1 = fmax3f(m1, v[c + 2], v[c + 3]);
      m2 = fmax3f(m2, v[c + 4], v[c + 5]);
      m3 = fmax3f(m3, v[c + 6], v[c + 7]);
    }
  }
  return fmaxf(fmaxf(m0, m1), fmaxf(m2, m3));
}

__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float (&v)[64]) {
  tmem_ld32(taddr, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
  tmem_ld32(taddr + 32, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
  tmem_ld_wait();
}

// Probabilities of 64 logits (columns col0 ..), p = 2^(v * sl2 + negm), packed
// to bf16 into 32 TMEM columns at p_taddr (16 at a time, so at most 16 packed
// words are live). Returns their fp32 sum. TAIL masks columns >= nvalid to
// probability 0.
template <bool TAIL>
__device__ __forceinline__ float exp64_store(const float (&v)[64], int col0, int nvalid, uint64_t scale2,
                                             uint64_t off2, uint32_t p_taddr) {
  uint64_t acc0 = f2_pack(0.f, 0.f), acc1 = acc0;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    uint32_t pk[16];
#pragma unroll
    for (int c = 0; c < 32; c += 4) {
      const int e = 32 * q + c;
      float a0, a1, b0, b1;
      f2_unpack(f2_fma(f2_pack(v[e], v[e + 1]), scale2, off2), a0, a1);
      f2_unpack(f2_fma(f2_pack(v[e + 2], v[e + 3]), scale2, off2), b0, b1);
      float p0 = ex2_approx(a0), p1 = ex2_approx(a1), p2 = ex2_approx(b0), p3 = ex2_approx(b1);
      if (TAIL) {
        const int g = col0 + e;
        p0 = (g < nvalid) ? p0 : 0.f;
        p1 = (g + 1 < nvalid) ? p1 : 0.f;
        p2 = (g + 2 < nvalid) ? p2 : 0.f;
        p3 = (g + 3 < nvalid) ? p3 : 0.f;
      }
      acc0 = f2_add(acc0, f2_pack(p0, p1));
      acc1 = f2_add(acc1, f2_pack(p2, p3));
      pk[c / 2] = pack_bf16x2(p0, p1);
      pk[c / 2 + 1] = pack_bf16x2(p2, p3);
    }
    tmem_st16(p_taddr + 16 * q, pk);
  }
  float s0, s1, s2, s3;
  f2_unpack(acc0, s0, s1);
  f2_unpack(acc1, s2, s3);
  return (s0 + s1) + (s2 + s3);
}

template <int D>
__global__ void __launch_bounds__(NUM_THREADS, 1) joint_attn_kernel(const __grid_constant__ Params p) {
  using C = Cfg<D>;
  constexpr int S = C::STAGES;
  const int b = blockIdx.z, h = blockIdx.y;
  int qb = blockIdx.x, role;
  if (qb < p.q_blocks[0]) {
    role = 0;
  } else if (qb - p.q_blocks[0] < p.q_blocks[1]) {
    qb -= p.q_blocks[0];
    role = 1;
  } else {
    qb -= p.q_blocks[0] + p.q_blocks[1];
    role = 2;
  }
  const int mode = p.mode ? __ldg(p.mode + b) : int(RA_MODE_FULL);
  if (role == 1 && mode == RA_MODE_REUSE) return;  // reference rows skipped (uniform exit)
  const int tileA = 2 * qb;
  const bool has_b = (tileA + 1) < p.q_tiles[role];

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;
  uint64_t* k_empty = bars + 1 + S;
  uint64_t* v_full = bars + 1 + 2 * S;
  uint64_t* v_empty = bars + 1 + 3 * S;
  uint64_t* s_full = bars + 1 + 4 * S;   // [tile]
  uint64_t* p_ready = bars + 3 + 4 * S;  // [tile]
  uint64_t* o_done = bars + 5 + 4 * S;   // [tile]
  uint64_t* drain = bars + 7 + 4 * S;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  float* red = reinterpret_cast<float*>(smem + C::OFF_MISC + 16);  // [tile][quarter]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < S; ++s) {
      mbar_init(k_full + s, 1);
      mbar_init(k_empty + s, 1);
      mbar_init(v_full + s, 1);
      mbar_init(v_empty + s, 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(s_full + t, 1);
      mbar_init(p_ready + t, 128);
      mbar_init(o_done + t, 1);
    }
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
  // Register split: warpgroup 0 (producer, MMA issuer, two idle warps) gives
  // up registers to the two softmax warpgroups: 4 x 56 + 8 x 224 = 12 x 168,
  // the launch allocation.
  if (warp < 4) {
    setmaxnreg_dec<56>();
    if (warp == 0) {
      if (lane == 0) {
        // ------------------------------------------------------------ TMA producer
        const bool fresh = p.fresh && refreshes(mode);
        const bool store_kv = fresh && p.store_kv && blockIdx.x == 0;
        const bool store_q = fresh && p.store_q && role == 1;
        const CUtensorMap* tq = (role == 1 && fresh) ? &p.tm_qf : &p.tm_q[role];
        if (fresh && blockIdx.x == 0 && h == 0 && p.a_b) p.a_b[b] = p.step;
        tma_prefetch_desc(tq);
        for (int r = 0; r < 3; ++r)
          if (p.kv_tiles[r] > 0) {
            tma_prefetch_desc((r == 1 && fresh) ? &p.tm_kf : &p.tm_k[r]);
            tma_prefetch_desc((r == 1 && fresh) ? &p.tm_vf : &p.tm_v[r]);
          }
        int k_issued = 0, v_issued = 0;  // K / V tiles whose loads were issued
        uint32_t stored_stages = 0;      // stages whose last tile has a store that may still read it
        bool q_stored = !store_q;
        // Copy tile jj (loaded by now or soon) into the cache slot if it is a
        // reference tile; the Q tiles go with the first call.
        auto store_tiles = [&](int jj) -> bool {
          if (!q_stored) {
            if (!mbar_wait(q_full, 0, ctl)) return false;
            fence_proxy_async_smem();
            for (int t = 0; t < (has_b ? 2 : 1); ++t)
              for (int c = 0; c < C::CHUNKS; ++c)
                tma_store_4d(&p.tm_q[1], smem + C::OFF_Q + t * C::TILE_BYTES + c * C::CHUNK_BYTES, c * 64,
                             (tileA + t) * BM, h, b);
            bulk_commit();
            q_stored = true;
          }
          int r, row0;
          kv_tile(p, jj, r, row0);
          if (!store_kv || r != 1) return true;
          const int s = jj % S;
          const uint32_t ph = (jj / S) & 1;
          if (!mbar_wait(k_full + s, ph, ctl) || !mbar_wait(v_full + s, ph, ctl)) return false;
          fence_proxy_async_smem();
          for (int c = 0; c < C::CHUNKS; ++c) {
            tma_store_4d(&p.tm_k[1], smem + C::OFF_K + s * C::TILE_BYTES + c * C::CHUNK_BYTES, c * 64, row0, h, b);
            tma_store_4d(&p.tm_v[1], smem + C::OFF_V + s * C::TILE_BYTES + c * C::CHUNK_BYTES, c * 64, row0, h, b);
          }
          bulk_commit();
          stored_stages |= 1u << s;
          return true;
        };
        mbar_arrive_expect_tx(q_full, C::TILE_BYTES * (has_b ? 2 : 1));
        for (int t = 0; t < (has_b ? 2 : 1); ++t)
          for (int c = 0; c < C::CHUNKS; ++c)
            tma_load_4d(smem + C::OFF_Q + t * C::TILE_BYTES + c * C::CHUNK_BYTES, tq, q_full, c * 64,
                        (tileA + t) * BM, h, b);
        for (int j = 0; j < nkv; ++j) {
          const int s = j % S;
          const uint32_t ph = (j / S) & 1;
          int r, row0;
          kv_tile(p, j, r, row0);
          if (j >= S && !mbar_wait(k_empty + s, ph ^ 1, ctl)) break;
          if (stored_stages & (1u << s)) {  // stage s still feeds a store of tile j - S
            bulk_wait_read_all();
            stored_stages = 0;
          }
          mbar_arrive_expect_tx(k_full + s, C::TILE_BYTES);
          for (int c = 0; c < C::CHUNKS; ++c)
            tma_load_4d(smem + C::OFF_K + s * C::TILE_BYTES + c * C::CHUNK_BYTES,
                        (r == 1 && fresh) ? &p.tm_kf : &p.tm_k[r], k_full + s, c * 64, row0, h, b);
          ++k_issued;
          if (j >= S && !mbar_wait(v_empty + s, ph ^ 1, ctl)) break;
          mbar_arrive_expect_tx(v_full + s, C::TILE_BYTES);
          for (int c = 0; c < C::CHUNKS; ++c)
            tma_load_4d(smem + C::OFF_V + s * C::TILE_BYTES + c * C::CHUNK_BYTES,
                        (r == 1 && fresh) ? &p.tm_vf : &p.tm_v[r], v_full + s, c * 64, row0, h, b);
          ++v_issued;
          if (j >= 1 && (store_kv || store_q) && !store_tiles(j - 1)) break;
        }
        if ((store_kv || store_q) && !*abort_flag && v_issued == nkv) store_tiles(nkv - 1);
        // Shared memory must outlive the reads of every store issued; the
        // cache slot is complete when the kernel is.
        if (store_kv || store_q) bulk_wait_all();
        if (*abort_flag) {
          // Let every load this thread issued land before the CTA exits: stage s
          // received loads for j = s, s + S, ...; wait for the last one's phase.
          mbar_wait_drain(q_full, 0, p.budget_ns);
          for (int s = 0; s < S; ++s) {
            const int nk = (k_issued > s) ? (k_issued - s + S - 1) / S : 0;
            const int nv = (v_issued > s) ? (v_issued - s + S - 1) / S : 0;
            if (nk > 0) mbar_wait_drain(k_full + s, (nk - 1) & 1, p.budget_ns);
            if (nv > 0) mbar_wait_drain(v_full + s, (nv - 1) & 1, p.budget_ns);
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
        const int ntile = has_b ? 2 : 1;
        bool issued_any = false;
        auto qk = [&](int j, int t) {
          const int s = j % S;
          umma_ss_ksteps<D / 16>(tmem + C::TM_S + 128 * t, sdesc_sw128(sq + t * C::TILE_BYTES, 16, 1024),
                                 sdesc_sw128(sk + s * C::TILE_BYTES, 16, 1024), IDESC_QK, 0u);
          umma_commit(s_full + t);
        };
        auto pv = [&](int j, int t) {
          const int s = j % S;
          umma_ts_ksteps8(tmem + C::TM_O + 128 * t, tmem + C::TM_S + 128 * t,
                          sdesc_sw128(sv + s * C::TILE_BYTES, C::CHUNK_BYTES, 1024), IDESC_PV, j > 0 ? 1u : 0u);
          // O_t is read only after the last P V (the epilogue); a rescale reads it
          // after s_full of the next tile, whose commit covers this P V too.
          if (j + 1 == nkv) umma_commit(o_done + t);
        };
        bool ok = mbar_wait(q_full, 0, ctl) && mbar_wait(k_full, 0, ctl);
        if (ok) {
          tc_fence_after();
          for (int t = 0; t < ntile; ++t) qk(0, t);
          umma_commit(k_empty);
          issued_any = true;
        }
        for (int j = 0; ok && j < nkv; ++j) {
          const int s = j % S;
          const bool next = j + 1 < nkv;
          if (!(ok = mbar_wait(v_full + s, (j / S) & 1, ctl))) break;
          if (next && !(ok = mbar_wait(k_full + (j + 1) % S, ((j + 1) / S) & 1, ctl))) break;
          for (int t = 0; t < ntile; ++t) {
            if (!(ok = mbar_wait(p_ready + t, j & 1, ctl))) break;
            tc_fence_after();
            pv(j, t);
            if (next) qk(j + 1, t);  // S_t is free: PV_t(j) was issued first
          }
          if (!ok) break;
          umma_commit(v_empty + s);
          if (next) umma_commit(k_empty + (j + 1) % S);
        }
        if (!ok && issued_any) {
          umma_commit(drain);
          mbar_wait_drain(drain, 0, p.budget_ns);
        }
      }
    }
  } else {
    setmaxnreg_inc<224>();
    // -------------------------------------------------------------- softmax
    const int t = (warp >= 8) ? 1 : 0;   // which Q tile this warpgroup owns
    const int quarter = warp & 3;        // TMEM lane quarter this warp may access
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    const uint32_t s_t = tmem + lane_off + C::TM_S + 128 * t;
    const uint32_t o_t = tmem + lane_off + C::TM_O + 128 * t;
    const int tile = tileA + t;
    const bool active = (t == 0) || has_b;
    const float sl2 = p.scale_log2;
    const float bias_l2 = (role == 2 && p.bias) ? __ldg(p.bias + h) * kLog2e : 0.f;
    float m = -INFINITY, l = 0.f, lref = 0.f;
    bool ok = active;
    for (int j = 0; ok && j < nkv; ++j) {
      int r, row0;
      kv_tile(p, j, r, row0);
      const int nvalid = min(BN, p.nk[r] - row0);
      const float badd = (r == 1) ? bias_l2 : 0.f;
      ok = __all_sync(0xffffffffu, mbar_wait(s_full + t, j & 1, ctl));
      if (!ok) break;
      tc_fence_after();
      // The previous P in S_t was consumed by PV_t(j-1), which completed before
      // QK_t(j) wrote S_t. The running max m only moves when the tile's max
      // exceeds it by more than 2^8 (then O, l, l_ref are rescaled by alpha).
      float alpha = 1.f;
      bool resc = false;
      const bool tail = nvalid < BN;
      float rs;
      if (!tail) {
        // Full key tile: one TMEM read of the row with the hardware row max
        // (tcgen05.ld.red), probabilities straight from registers.
        float va[64], vb[64];
        float m0, m1, m2, m3;
        tmem_ldred32_max(s_t + 0, *reinterpret_cast<uint32_t(*)[32]>(&va[0]), m0);
        tmem_ldred32_max(s_t + 32, *reinterpret_cast<uint32_t(*)[32]>(&va[32]), m1);
        tmem_ldred32_max(s_t + 64, *reinterpret_cast<uint32_t(*)[32]>(&vb[0]), m2);
        tmem_ldred32_max(s_t + 96, *reinterpret_cast<uint32_t(*)[32]>(&vb[32]), m3);
        tmem_ld_wait();
        const float mt = fmaf(fmaxf(fmaxf(m0, m1), fmaxf(m2, m3)), sl2, badd);  // tile max, log2 units
        if (mt > m + kRescaleThresh) {
          alpha = ex2_approx(m - mt);  // 0 when m = -inf
          resc = (j > 0);
          l *= alpha;
          lref *= alpha;
          m = mt;
        }
        // P_j over the first 64 columns of S_t: the logits are all in registers.
        const uint64_t scale2 = f2_pack(sl2, sl2);
        const uint64_t off2 = f2_pack(badd - m, badd - m);
        rs = exp64_store<false>(va, 0, BN, scale2, off2, s_t + 0);
        rs += exp64_store<false>(vb, 64, BN, scale2, off2, s_t + 32);
      } else {
        // Tail key tile: pass 1 takes the max over the valid columns only,
        // pass 2 re-reads the logits (half hf -> P columns [32 hf, 32 hf + 32),
        // never over logits still to be read).
        float mx = -INFINITY;
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          float v[64];
          tmem_ld64(s_t + 64 * hf, v);
          mx = max64<true>(v, 64 * hf, nvalid, mx);
        }
        const float mt = fmaf(mx, sl2, badd);
        if (mt > m + kRescaleThresh) {
          alpha = ex2_approx(m - mt);
          resc = (j > 0);
          l *= alpha;
          lref *= alpha;
          m = mt;
        }
        const uint64_t scale2 = f2_pack(sl2, sl2);
        const uint64_t off2 = f2_pack(badd - m, badd - m);
        rs = 0.f;
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          float v[64];
          tmem_ld64(s_t + 64 * hf, v);
          rs += exp64_store<true>(v, 64 * hf, nvalid, scale2, off2, s_t + 32 * hf);
        }
      }
      l += rs;
      if (r == 1) lref += rs;
      if (__any_sync(0xffffffffu, resc)) {
        // PV_t(j-1) is complete: the commit that signalled s_full for this
        // tile tracks every MMA issued before QK_t(j).
        tc_fence_after();
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t ov[32];
          tmem_ld32(o_t + c0, ov);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(__uint_as_float(ov[i]) * alpha);
          tmem_st32(o_t + c0, ov);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(p_ready + t);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_done + t, 0, ctl));
    const int grow = tile * BM + row;
    const bool valid = active && grow < p.nq[role];
    const float inv_l = 1.f / l;
    if (ok) {
      tc_fence_after();
      __nv_bfloat16* orow = p.o_ptr[role] + b * p.o_sb[role] + h * p.o_sh[role] + int64_t(grow) * p.o_sn[role];
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t ov[32];
        tmem_ld32(o_t + c0, ov);
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
    const bool in_mass = ((role == 2) || (role == 0 && p.mass_rows == 1)) &&
                         (p.mass_stride <= 1 || grow % p.mass_stride == 0);
    float mv = (ok && valid && in_mass) ? lref * inv_l : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mv += __shfl_xor_sync(0xffffffffu, mv, o);
    if (lane == 0) red[4 * t + quarter] = mv;
    named_bar_sync(1 + t, 128);
    if (ok && active && role != 1 && quarter == 0 && lane == 0) {
      const int idx = (role == 0) ? tile : p.q_tiles[0] + tile;
      p.mass_partial[(int64_t(b) * p.H + h) * p.mpl + idx] =
          ((red[4 * t] + red[4 * t + 1]) + red[4 * t + 2]) + red[4 * t + 3];
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
template <int D>
ra_status launch(const Params& p, dim3 grid, cudaStream_t st) {
  const ra_status as = ensure_dynamic_smem(reinterpret_cast<const void*>(joint_attn_kernel<D>), Cfg<D>::SMEM_ALLOC,
                                           "refadapt_joint_attn");
  if (as != RA_OK) return as;
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
  if (a->mass_row_stride < 0) {
    set_error("refadapt_joint_attn: mass_row_stride must be >= 0");
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
  bool ref_rows = true;
  for (int r = 0; r < 3; ++r) {
    if (a->v[r].n != a->k[r].n || a->o[r].n != a->q[r].n) {
      set_error("refadapt_joint_attn: %s: k and v (key rows) or q and o (query rows) disagree on n", names[r]);
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
    set_error("refadapt_joint_attn: the target segment needs at least one key row");
    return RA_EINVAL;
  }
  const int d = a->d;
  for (int r = 0; r < 3; ++r) {
    const int nk = a->k[r].n, nq = (r == RA_REF && !ref_rows) ? 0 : a->q[r].n;
    p.nk[r] = nk;
    p.nq[r] = nq;
    p.kv_tiles[r] = (nk + BN - 1) / BN;
    p.q_tiles[r] = (nq + BM - 1) / BM;
    p.q_blocks[r] = (p.q_tiles[r] + 1) / 2;
    if (nk > 0 && (!encode_seg(&p.tm_k[r], a->k[r], a->B, a->H, d, 64, BN, true) ||
                   !encode_seg(&p.tm_v[r], a->v[r], a->B, a->H, d, 64, BN, true)))
      return RA_EINVAL;
    if (nq == 0) continue;
    if (!encode_seg(&p.tm_q[r], a->q[r], a->B, a->H, d, 64, BM, true)) return RA_EINVAL;
    p.o_ptr[r] = static_cast<__nv_bfloat16*>(a->o[r].ptr);
    p.o_sb[r] = a->o[r].stride_b;
    p.o_sh[r] = a->o[r].stride_h;
    p.o_sn[r] = a->o[r].stride_n;
  }
  if (a->ref_fresh_q.ptr != nullptr || a->ref_fresh_k.ptr != nullptr || a->ref_fresh_v.ptr != nullptr ||
      a->a_b != nullptr) {
    // Fused cache update: this step's reference rows, read by refreshing
    // samples and copied into the segments k/v/q[RA_REF] point at.
    const ra_seg* fr[3] = {&a->ref_fresh_q, &a->ref_fresh_k, &a->ref_fresh_v};
    const ra_seg* ca[3] = {&a->q[RA_REF], &a->k[RA_REF], &a->v[RA_REF]};
    const char* kinds[3] = {"q", "k", "v"};
    bool copy[3] = {false, false, false};
    for (int i = 0; i < 3; ++i) {
      if (i == 0 && !ref_rows) {
        if (fr[0]->ptr != nullptr || fr[0]->n != 0) {
          set_error("refadapt_joint_attn: ref_fresh_q given without reference query rows (q[ref] is NULL)");
          return RA_EINVAL;
        }
        continue;
      }
      snprintf(what, sizeof(what), "refadapt_joint_attn: ref_fresh_%s", kinds[i]);
      if (!check_seg(*fr[i], what)) return RA_EINVAL;
      if (fr[i]->n != ca[i]->n) {
        set_error("refadapt_joint_attn: ref_fresh_%s has n = %d, %s[ref] has %d", kinds[i], fr[i]->n, kinds[i],
                  ca[i]->n);
        return RA_EINVAL;
      }
      if (fr[i]->ptr == ca[i]->ptr) {
        if (fr[i]->stride_b != ca[i]->stride_b || fr[i]->stride_h != ca[i]->stride_h ||
            fr[i]->stride_n != ca[i]->stride_n) {
          set_error("refadapt_joint_attn: ref_fresh_%s shares its pointer with %s[ref] but not its strides",
                    kinds[i], kinds[i]);
          return RA_EINVAL;
        }
        continue;  // read in place
      }
      copy[i] = true;
      if (fr[i]->n > 0) {
        CUtensorMap* tm = (i == 0) ? &p.tm_qf : (i == 1) ? &p.tm_kf : &p.tm_vf;
        if (!encode_seg(tm, *fr[i], a->B, a->H, d, 64, (i == 0) ? BM : BN, true)) return RA_EINVAL;
      }
    }
    if (copy[1] != copy[2]) {
      set_error("refadapt_joint_attn: ref_fresh_k and ref_fresh_v must both be in place or both be copied");
      return RA_EINVAL;
    }
    // Segments read in place keep their own maps as the fresh ones.
    if (!copy[0]) p.tm_qf = p.tm_q[RA_REF];
    if (!copy[1]) {
      p.tm_kf = p.tm_k[RA_REF];
      p.tm_vf = p.tm_v[RA_REF];
    }
    p.fresh = 1;
    p.store_kv = copy[1] ? 1 : 0;
    p.store_q = copy[0] ? 1 : 0;
    p.a_b = a->a_b;
    p.step = a->step;
  }
  p.B = a->B;
  p.H = a->H;
  p.mass_rows = a->mass_rows;
  p.mass_stride = a->mass_row_stride;
  p.mpl = refadapt_mass_partial_len(a->q[RA_TEXT].n, a->q[RA_TGT].n);
  const float scale = a->softmax_scale > 0.f ? a->softmax_scale : 1.0f / std::sqrt(float(d));
  p.scale_log2 = scale * kLog2e;
  p.bias = a->ref_logit_bias;
  p.mode = a->mode;
  p.mass_partial = a->mass_partial;
  p.err_word = a->err_word;
  p.budget_ns = wait_budget_ns();
  const int blocks = p.q_blocks[0] + p.q_blocks[1] + p.q_blocks[2];
  dim3 grid(blocks, a->H, a->B);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return d == 128 ? launch<128>(p, grid, st) : launch<64>(p, grid, st);
}
