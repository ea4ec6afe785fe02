// refadapt_q_delta: relative L2 change of the target query per (sample, head),
// D = ||q_t - q_{t-1}||_F / (||q_{t-1}||_F + eps)   (paper Eq. 1, Sec. 4).
//
// HBM-bound streaming reduction. Work is cut into units of one (sample,
// head) slab: 8 KB per tensor on the cluster path, 12 KB on the multi-block
// path (32 / 48 rows at d = 128, 64 / 96 at d = 64). When
// both tensors' rows are contiguous within a slab (stride_n == d) a unit is
// one 1-D bulk copy of its bytes (the slab's last unit is shorter); otherwise
// it is a 2-D TMA tensor load (any row strides; rows past the slab end arrive
// as zeros and add nothing). A producer thread streams both tensors' units
// through a shared-memory ring; unit i goes to stage i % S and is consumed by
// warp i % S, so every stage has one consumer that waits its phases in order.
//
// Arithmetic stays off the FP64 pipe, which is narrow on this GPU (a chain
// of dependent fp64 adds, square roots and a division cost microseconds at
// the end of a launch): packed fp32 sums of (q_t - q_{t-1})^2 and q_{t-1}^2
// per lane, an fp32 butterfly per unit, then compensated two-float sums
// (TwoSum: hi + lo carries the rounding error of every addition) across
// units, warps, CTAs and cluster ranks, and D formed in fp32 from hi + lo.
// Every sum has a fixed order, so D is deterministic.
//
// Cluster path (used when the slabs fit clusters that fill the GPU): one
// cluster of up to 8 CTAs per (sample, head) slab, each CTA streaming its
// contiguous share of the slab's units through a 12-stage ring (one CTA per
// SM) or a 6-stage ring (two per SM), whichever keeps more bytes in flight; every
// CTA stores its sums into the cluster leader's shared memory (distributed
// shared memory) and, after one cluster barrier, the leader adds them in rank
// order and writes D. No global atomics, fences or workspace: the reduction
// tail is one cluster barrier. On the bulk path each CTA asks L2 for its
// first S units before it waits for the previous kernel of the stream
// (programmatic dependent launch): L2 is the GPU's point of coherence, so the
// loads issued after that wait still see everything the previous kernel
// wrote, and the first units no longer pay the full trip from HBM after it.
//
// Multi-block path (slabs too long for one cluster, or too few slabs to fill
// the GPU): one CTA per SM, an 8-stage ring; CTA c takes the contiguous unit
// range [c U / G, (c+1) U / G) in slab-major order, adds its unit sums per
// slab in unit order into one slot per (slab, CTA) of the workspace; the
// slab's last contributor (ticket counter) adds the slots in CTA order,
// writes D and re-arms the counter.
//
// refadapt_q_delta_gate runs Algorithm 1's gate on the new D in the same
// launch (cluster path): each leader's first consumer warp reduces its
// slab's mass partials of the previous step into M right after the
// dependency wait (while the first units are in flight); after D, the leader
// stores its head's score term and takes a ticket, and the leader that takes
// the last one sums the B x H terms in head order and decides (gate_body.cuh;
// the same arithmetic and order as refadapt_gate). On the multi-block path
// the gate is a launch of its own.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <mutex>

#include "api_common.h"
#include "gate_body.cuh"
#include "tc_ptx.cuh"

namespace ra {
namespace qd {

constexpr int MAX_SPLITS = 128;       // slots per slab in the workspace
constexpr int CONSUMER_WARPS = 8;
constexpr int STAGES = CONSUMER_WARPS;  // stage s belongs to consumer warp s
constexpr int UNIT_BYTES = 12288;       // per tensor: 48 rows at d = 128, 96 at d = 64
constexpr int THREADS = 32 * (CONSUMER_WARPS + 1);
constexpr int MAX_UNITS_PER_CTA = 1024;
constexpr int OFF_BAR = STAGES * 2 * UNIT_BYTES;
constexpr int OFF_MISC = OFF_BAR + 2 * STAGES * 8;           // abort flag
constexpr int OFF_SUMS = OFF_MISC + 16;                       // float2 per unit
constexpr int SMEM_BYTES = OFF_SUMS + MAX_UNITS_PER_CTA * 8;
constexpr int SMEM_ALLOC = SMEM_BYTES + 1024;
static_assert(SMEM_ALLOC <= 232448, "shared memory budget");

struct Params {
  CUtensorMap tm_c, tm_p;  // (d, n, H, B), box (d, rows_per_unit), no swizzle
  const char* base_c;      // 1-D bulk path: slab (b, h) starts at base + b * sb + h * sh
  const char* base_p;
  int64_t c_sb, c_sh, p_sb, p_sh;  // bytes
  int64_t slab_bytes;      // n * d * 2
  int32_t bulk;            // 1: 1-D bulk copies, 0: 2-D tensor loads
  int32_t H, rows_per_unit;
  int32_t per_slab;        // units per slab
  int32_t units;           // all units
  int32_t grid;
  float eps;
  float* d_out;
  float4* partial;         // [B*H][MAX_SPLITS]: (hi, lo) of both sums
  uint32_t* counter;       // [B*H]
  uint64_t budget_ns;
};

// CTA that owns unit u under the balanced split of U units over G CTAs.
__device__ __forceinline__ int owner(int64_t u, int64_t U, int64_t G) {
  return int(((u + 1) * G + U - 1) / U - 1);
}

// Sums over one 16-byte vector pair: (c - p)^2 and p^2, two lanes of fp32 at a time.
__device__ __forceinline__ void acc16(const uint4& c, const uint4& p, uint64_t& sd, uint64_t& sp) {
  const uint32_t cw[4] = {c.x, c.y, c.z, c.w};
  const uint32_t pw[4] = {p.x, p.y, p.z, p.w};
  const uint64_t neg1 = f2_pack(-1.f, -1.f);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint64_t cc = f2_pack(__uint_as_float(cw[i] << 16), __uint_as_float(cw[i] & 0xFFFF0000u));
    const uint64_t pp = f2_pack(__uint_as_float(pw[i] << 16), __uint_as_float(pw[i] & 0xFFFF0000u));
    const uint64_t df = f2_fma(pp, neg1, cc);  // exact: both are bf16 values
    sd = f2_fma(df, df, sd);
    sp = f2_fma(pp, pp, sp);
  }
}

// L2 prefetch of `bytes` (a multiple of 16) at a 16-byte aligned global address.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(src)), "r"(bytes)
               : "memory");
}

// (hi, lo) += x with the rounding error of the addition kept in lo (TwoSum,
// six fp32 operations; the value is hi + lo).
__device__ __forceinline__ void ff_add(float& hi, float& lo, float x) {
  const float s = hi + x;
  const float v = s - hi;
  lo += (hi - (s - v)) + (x - v);
  hi = s;
}

// Sum of one lane value over the warp (fixed butterfly: every lane ends with
// the same value).
__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// (hi, lo) pairs of the 32 lanes added up in a fixed tree; lane 0 ends with
// the total (the other lanes' values are partial).
__device__ __forceinline__ void ff_tree(float& hi, float& lo) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float xh = __shfl_down_sync(0xffffffffu, hi, o);
    const float xl = __shfl_down_sync(0xffffffffu, lo, o);
    ff_add(hi, lo, xh);
    lo += xl;
  }
}

__global__ void __launch_bounds__(THREADS, 1) q_delta_kernel(const __grid_constant__ Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* empty = full + STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_MISC);
  float* sums = reinterpret_cast<float*>(smem + OFF_SUMS);
  const int c = blockIdx.x;
  const int u0 = int(int64_t(c) * p.units / p.grid);
  const int u1 = int(int64_t(c + 1) * p.units / p.grid);
  const int nu = u1 - u0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const WaitCtl ctl{abort_flag, nullptr, p.budget_ns};

  if (warp == CONSUMER_WARPS) {
    if (lane == 0) {
      // ---------------------------------------------------------- producer
      if (!p.bulk) {
        tma_prefetch_desc(&p.tm_c);
        tma_prefetch_desc(&p.tm_p);
      }
      int issued = 0;
      for (int i = 0; i < nu; ++i) {
        const int s = i % STAGES;
        if (i >= STAGES && !mbar_wait(empty + s, ((i / STAGES) - 1) & 1, ctl)) break;
        const int u = u0 + i;
        const int slab = u / p.per_slab, k = u % p.per_slab;
        const int b = slab / p.H, h = slab % p.H;
        if (p.bulk) {
          const int64_t off = int64_t(k) * UNIT_BYTES;
          const int64_t rem = p.slab_bytes - off;
          const uint32_t bytes = uint32_t(rem < UNIT_BYTES ? rem : UNIT_BYTES);
          mbar_arrive_expect_tx(full + s, 2 * bytes);
          bulk_load(smem + s * 2 * UNIT_BYTES, p.base_c + b * p.c_sb + h * p.c_sh + off, bytes, full + s);
          bulk_load(smem + s * 2 * UNIT_BYTES + UNIT_BYTES, p.base_p + b * p.p_sb + h * p.p_sh + off, bytes,
                    full + s);
        } else {
          mbar_arrive_expect_tx(full + s, 2 * UNIT_BYTES);
          tma_load_4d(smem + s * 2 * UNIT_BYTES, &p.tm_c, full + s, 0, k * p.rows_per_unit, h, b);
          tma_load_4d(smem + s * 2 * UNIT_BYTES + UNIT_BYTES, &p.tm_p, full + s, 0, k * p.rows_per_unit, h, b);
        }
        ++issued;
      }
      if (*abort_flag) {
        for (int s = 0; s < STAGES; ++s) {
          const int n_s = (issued > s) ? (issued - s + STAGES - 1) / STAGES : 0;
          if (n_s > 0) mbar_wait_drain(full + s, (n_s - 1) & 1, p.budget_ns);
        }
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    for (int i = warp; i < nu; i += CONSUMER_WARPS) {
      const int s = i % STAGES;
      if (!__all_sync(0xffffffffu, mbar_wait(full + s, (i / STAGES) & 1, ctl))) break;
      const uint4* vc = reinterpret_cast<const uint4*>(smem + s * 2 * UNIT_BYTES);
      const uint4* vp = reinterpret_cast<const uint4*>(smem + s * 2 * UNIT_BYTES + UNIT_BYTES);
      uint64_t sd = f2_pack(0.f, 0.f), sp = sd;
      int nvec = UNIT_BYTES / 16;  // a short last unit of the bulk path holds fewer bytes
      if (p.bulk) {
        const int64_t rem = p.slab_bytes - int64_t((u0 + i) % p.per_slab) * UNIT_BYTES;
        if (rem < UNIT_BYTES) nvec = int(rem / 16);
      }
      if (nvec == UNIT_BYTES / 16) {
#pragma unroll 8
        for (int m = 0; m < UNIT_BYTES / 16 / 32; ++m) acc16(vc[lane + 32 * m], vp[lane + 32 * m], sd, sp);
      } else {
        for (int v = lane; v < nvec; v += 32) acc16(vc[v], vp[v], sd, sp);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty + s);
      float a0, a1, b0, b1;
      f2_unpack(sd, a0, a1);
      f2_unpack(sp, b0, b1);
      const float ud = warp_sum(a0 + a1), up = warp_sum(b0 + b1);
      if (lane == 0) {
        sums[2 * i] = ud;
        sums[2 * i + 1] = up;
      }
    }
    named_bar_sync(1, 32 * CONSUMER_WARPS);
    if (warp == 0) {
      // Per slab touched by this CTA: add its unit sums in unit order, store the
      // slot, take a ticket; the slab's last contributor finishes D.
      const bool aborted = *abort_flag != 0;
      int i = 0;
      while (i < nu) {
        const int slab = (u0 + i) / p.per_slab;
        float dh = 0.f, dl = 0.f, ph = 0.f, pl = 0.f;
        int j = i;
        for (; j < nu && (u0 + j) / p.per_slab == slab; ++j) {
          ff_add(dh, dl, sums[2 * j]);
          ff_add(ph, pl, sums[2 * j + 1]);
        }
        const int64_t first_u = int64_t(slab) * p.per_slab;
        const int64_t last_u = first_u + p.per_slab - 1;
        const int c_lo = owner(first_u, p.units, p.grid);
        const int count = owner(last_u, p.units, p.grid) - c_lo + 1;
        float4* slots = p.partial + int64_t(slab) * MAX_SPLITS;
        uint32_t last = 0;
        if (lane == 0) {
          __stcg(slots + (c - c_lo), make_float4(aborted ? NAN : dh, dl, ph, pl));
          __threadfence();
          last = (atomicAdd(p.counter + slab, 1u) == uint32_t(count - 1)) ? 1u : 0u;
        }
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          __threadfence();
          // lane q adds the slots q, q + 32, ... in order; then a fixed tree
          // over the lanes' (hi, lo) pairs ends in lane 0
          float sdh = 0.f, sdl = 0.f, sph = 0.f, spl = 0.f;
          for (int q = lane; q < count; q += 32) {
            const float4 v = __ldcg(slots + q);
            ff_add(sdh, sdl, v.x);
            sdl += v.y;
            ff_add(sph, spl, v.z);
            spl += v.w;
          }
          ff_tree(sdh, sdl);
          ff_tree(sph, spl);
          if (lane == 0) {
            p.d_out[slab] = sqrtf(sdh + sdl) / (sqrtf(sph + spl) + p.eps);
            p.counter[slab] = 0u;  // re-arm for the next call
          }
        }
        i = j;
      }
    }
  }
}

// ---------------------------------------------------------------- cluster path
constexpr int CL_MAX_CS = 8;       // CTAs per cluster (portable limit)
constexpr int CL_MAX_UNITS = 384;  // units per CTA (longer slabs take the multi-block path)

// Units of the cluster path: 8 KB per tensor (32 rows at d = 128, 64 at d = 64).
// What sets a short read's time is how many units each SM has in flight and
// how many warps drain them: 12 stages of 8 KB (192 KB, 12 consumer warps)
// read the image-edit target query (24 slabs of 1 MB) in 9.8 us and the video
// one (24 slabs of 4.2 MB) in 31.4 us, against 10.7 and 31.9 us for 8 stages
// of 12 KB over the same 192 KB, and 13.2 us for 6 stages of 8 KB.
constexpr int CL_UNIT_BYTES = 8192;

// Shared-memory layout of a cluster CTA with S stages of UB-byte units per
// tensor (stage s belongs to consumer warp s; warp S is the producer).
template <int S, int UB>
struct ClLayout {
  static constexpr int THREADS = 32 * (S + 1);
  static constexpr int OFF_BAR = S * 2 * UB;
  static constexpr int OFF_MISC = OFF_BAR + 2 * S * 8;          // abort flag
  static constexpr int OFF_WSUM = OFF_MISC + 16;                 // float4 (hi, lo of both sums) per consumer warp
  static constexpr int OFF_SLOTS = OFF_WSUM + S * 16;            // leader: float4 per rank
  static constexpr int BYTES = OFF_SLOTS + CL_MAX_CS * 16;
  static constexpr int ALLOC = BYTES + 1024;
};
static_assert(ClLayout<12, CL_UNIT_BYTES>::ALLOC <= 232448, "shared memory budget");
static_assert(2 * ClLayout<6, CL_UNIT_BYTES>::ALLOC <= 232448, "two 6-stage CTAs per SM");

struct ClusterParams {
  CUtensorMap tm_c, tm_p;
  const char* base_c;
  const char* base_p;
  int64_t c_sb, c_sh, p_sb, p_sh;
  int64_t slab_bytes;
  int32_t bulk;
  int32_t H, rows_per_unit, per_slab, cs;
  int32_t k_begin[CL_MAX_CS + 1];  // rank r streams units [k_begin[r], k_begin[r + 1]) of its slab
  float eps;
  float* d_out;
  uint64_t budget_ns;
  // refadapt_q_delta_gate: each leader stores its head's score term and takes
  // a ticket; the leader that takes the last one decides for the block
  int32_t fuse_gate;
  uint32_t* gate_ticket;  // workspace counter (zero between launches)
  float2* gate_terms;     // workspace [B * H]: each head's score term (g, e)
  gate::Params gp;        // gp.qd == d_out
};

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Arrival that only says "this CTA has started": no release (nothing is
// published by it; the final cluster_sync_all orders the remote stores).
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <int S, int UB>
__global__ void __launch_bounds__(ClLayout<S, UB>::THREADS)
    q_delta_cluster_kernel(const __grid_constant__ ClusterParams p) {
  using L = ClLayout<S, UB>;
  constexpr int CL_STAGES = S, CL_CONSUMERS = S;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* empty = full + CL_STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC);
  float4* wsum = reinterpret_cast<float4*>(smem + L::OFF_WSUM);
  float4* slots = reinterpret_cast<float4*>(smem + L::OFF_SLOTS);
  uint32_t rank;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const int h = blockIdx.y, b = blockIdx.z;
  const int k0 = p.k_begin[rank];
  const int nu = p.k_begin[rank + 1] - k0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float m_exp = 0.f;  // fused gate: M_{t-1,b,h} of this slab (leader, thread 0)
  float d_val = 0.f;  // the slab's D (leader, thread 0)
  // This CTA has started (its shared memory exists): the remote stores at the
  // end wait for every CTA's arrival, the loads below need no one else.
  cluster_arrive();
  const WaitCtl ctl{abort_flag, nullptr, p.budget_ns};
  // Programmatic dependent launch: this grid may start while the previous
  // kernel of the stream finishes. Each role waits for that kernel (complete,
  // its writes visible) before it touches global memory; the next kernel of
  // the stream may start its own set-up as soon as every CTA got here.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == CL_CONSUMERS) {
    // The producer warp sets up the ring itself and releases the consumers
    // (named barrier 2) without waiting for them, so its first loads leave at
    // once.
    if (lane == 0) {
      for (int s = 0; s < CL_STAGES; ++s) {
        mbar_init(full + s, 1);
        mbar_init(empty + s, 1);
      }
      *abort_flag = 0;
      fence_mbar_init();
    }
    __syncwarp();
    named_bar_arrive(2, L::THREADS);
    if (p.bulk && lane < CL_STAGES && lane < nu) {
      // Ask L2 for this CTA's first units while the previous kernel of the
      // stream may still run. Only L2 is filled: the copies into shared
      // memory start after griddepcontrol.wait, and L2 is coherent, so they
      // see whatever that kernel writes meanwhile.
      const int64_t off = int64_t(k0 + lane) * UB;
      const int64_t rem = p.slab_bytes - off;
      const uint32_t bytes = uint32_t(rem < UB ? rem : UB);
      bulk_prefetch_l2(p.base_c + b * p.c_sb + h * p.c_sh + off, bytes);
      bulk_prefetch_l2(p.base_p + b * p.p_sb + h * p.p_sh + off, bytes);
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (lane == 0) {
      // ---------------------------------------------------------- producer
      if (!p.bulk) {
        tma_prefetch_desc(&p.tm_c);
        tma_prefetch_desc(&p.tm_p);
      }
      int issued = 0;
      for (int i = 0; i < nu; ++i) {
        const int s = i % CL_STAGES;
        if (i >= CL_STAGES && !mbar_wait(empty + s, ((i / CL_STAGES) - 1) & 1, ctl)) break;
        const int k = k0 + i;
        if (p.bulk) {
          const int64_t off = int64_t(k) * UB;
          const int64_t rem = p.slab_bytes - off;
          const uint32_t bytes = uint32_t(rem < UB ? rem : UB);
          mbar_arrive_expect_tx(full + s, 2 * bytes);
          bulk_load(smem + s * 2 * UB, p.base_c + b * p.c_sb + h * p.c_sh + off, bytes, full + s);
          bulk_load(smem + s * 2 * UB + UB, p.base_p + b * p.p_sb + h * p.p_sh + off, bytes,
                    full + s);
        } else {
          mbar_arrive_expect_tx(full + s, 2 * UB);
          tma_load_4d(smem + s * 2 * UB, &p.tm_c, full + s, 0, k * p.rows_per_unit, h, b);
          tma_load_4d(smem + s * 2 * UB + UB, &p.tm_p, full + s, 0, k * p.rows_per_unit, h, b);
        }
        ++issued;
      }
      if (*abort_flag) {
        for (int s = 0; s < CL_STAGES; ++s) {
          const int n_s = (issued > s) ? (issued - s + CL_STAGES - 1) / CL_STAGES : 0;
          if (n_s > 0) mbar_wait_drain(full + s, (n_s - 1) & 1, p.budget_ns);
        }
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    named_bar_sync(2, L::THREADS);  // the ring's barriers are initialised
    asm volatile("griddepcontrol.wait;" ::: "memory");  // orders the final store of D
    // Fused gate: the leader's first warp reduces this slab's mass partials of
    // the previous step (they need nothing of this launch) while the first
    // units are still on their way.
    if (p.fuse_gate && rank == 0 && warp == 0) m_exp = gate::head_exposure(p.gp, b * p.H + h);
    float dh = 0.f, dl = 0.f, ph = 0.f, pl = 0.f;  // this warp's units, in order (lane 0)
    for (int i = warp; i < nu; i += CL_CONSUMERS) {
      const int s = i % CL_STAGES;
      if (!__all_sync(0xffffffffu, mbar_wait(full + s, (i / CL_STAGES) & 1, ctl))) break;
      const uint4* vc = reinterpret_cast<const uint4*>(smem + s * 2 * UB);
      const uint4* vp = reinterpret_cast<const uint4*>(smem + s * 2 * UB + UB);
      uint64_t sd = f2_pack(0.f, 0.f), sp = sd;
      int nvec = UB / 16;
      if (p.bulk) {
        const int64_t rem = p.slab_bytes - int64_t(k0 + i) * UB;
        if (rem < UB) nvec = int(rem / 16);
      }
      if (nvec == UB / 16) {
#pragma unroll 8
        for (int m = 0; m < UB / 16 / 32; ++m) acc16(vc[lane + 32 * m], vp[lane + 32 * m], sd, sp);
      } else {
        for (int v = lane; v < nvec; v += 32) acc16(vc[v], vp[v], sd, sp);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(empty + s);
      float a0, a1, b0, b1;
      f2_unpack(sd, a0, a1);
      f2_unpack(sp, b0, b1);
      const float ud = warp_sum(a0 + a1), up = warp_sum(b0 + b1);
      if (lane == 0) {
        ff_add(dh, dl, ud);
        ff_add(ph, pl, up);
      }
    }
    if (lane == 0) wsum[warp] = make_float4(dh, dl, ph, pl);
    named_bar_sync(1, 32 * CL_CONSUMERS);
  }
  // Every CTA of the cluster has arrived (started), so the leader's shared
  // memory exists; then this CTA's share, in unit order, goes into the
  // leader's slot `rank`.
  cluster_wait();
  if (threadIdx.x == 0) {
    float dh = 0.f, dl = 0.f, ph = 0.f, pl = 0.f;
    for (int w = 0; w < CL_CONSUMERS; ++w) {
      const float4 v = wsum[w];
      ff_add(dh, dl, v.x);
      dl += v.y;
      ff_add(ph, pl, v.z);
      pl += v.w;
    }
    if (*abort_flag) dh = NAN;
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(slots)), "r"(0));
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote + 16 * rank), "f"(dh), "f"(dl),
                 "f"(ph), "f"(pl)
                 : "memory");
  }
  // All remote stores are done and visible to the leader; no CTA exits while
  // another may still write into its shared memory.
  cluster_sync_all();
  if (rank == 0 && threadIdx.x == 0) {
    float dh = 0.f, dl = 0.f, ph = 0.f, pl = 0.f;
    for (int r = 0; r < p.cs; ++r) {
      const float4 v = slots[r];
      ff_add(dh, dl, v.x);
      dl += v.y;
      ff_add(ph, pl, v.z);
      pl += v.w;
    }
    d_val = sqrtf(dh + dl) / (sqrtf(ph + pl) + p.eps);
    p.d_out[b * p.H + h] = d_val;
  }
  if (p.fuse_gate && rank == 0) {
    // Every leader publishes its head's score term (and M for the log), then
    // a ticket after a fence; the leader that takes the last ticket re-arms
    // the counter and its CTA sums the terms in head order and decides (the
    // arithmetic of refadapt_gate, in its order). No CTA waits for another.
    volatile int32_t* last = reinterpret_cast<volatile int32_t*>(smem + L::OFF_MISC + 4);
    volatile int32_t* full_step = last + 1;
    if (threadIdx.x == 0) {
      const int sh = b * p.H + h;
      float g, e;
      gate::score_term(p.gp.cue, d_val, m_exp, g, e);
      p.gate_terms[sh] = make_float2(g, e);
      if (p.gp.m_out) p.gp.m_out[sh] = m_exp;
      __threadfence();
      const uint32_t total = gridDim.y * gridDim.z;
      const bool is_last = atomicAdd(p.gate_ticket, 1u) == total - 1;
      if (is_last) {
        *p.gate_ticket = 0u;  // re-armed for the next launch (visible when this one completes)
        *full_step = gate::open_step(p.gp);
      }
      *last = is_last ? 1 : 0;
    }
    __syncthreads();
    if (*last) {
      const float2* terms = p.gate_terms;
      for (int s = threadIdx.x; s < p.gp.B; s += blockDim.x)
        gate::decide_sample(p.gp, s, *full_step, true, [&](int hh, float& g, float& e) {
          const float2 v = __ldcg(terms + s * p.gp.H + hh);
          g = v.x;
          e = v.y;
        });
    }
  }
}

// The cluster kernels: 12 stages (one CTA per SM) or 6 stages (two per SM).
constexpr int CL_VARIANTS = 2;
struct ClVariant {
  int S, threads, smem;
  void (*fn)(ClusterParams);
};
inline const ClVariant& cl_variant(int i) {
  static const ClVariant v[CL_VARIANTS] = {
      {12, ClLayout<12, CL_UNIT_BYTES>::THREADS, ClLayout<12, CL_UNIT_BYTES>::ALLOC,
       q_delta_cluster_kernel<12, CL_UNIT_BYTES>},
      {6, ClLayout<6, CL_UNIT_BYTES>::THREADS, ClLayout<6, CL_UNIT_BYTES>::ALLOC,
       q_delta_cluster_kernel<6, CL_UNIT_BYTES>},
  };
  return v[i];
}

// Clusters of cs CTAs of cluster variant vi that can be resident at once on
// the current device (cached per device); -1 with the error set on failure.
// Also raises the kernels' dynamic shared-memory limit once per device.
int max_active_clusters(int vi, int cs) {
  static std::mutex mu;
  static int cache[64][CL_VARIANTS][CL_MAX_CS + 1];
  static bool ready[64] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    set_error("refadapt_q_delta: no usable current device");
    return -1;
  }
  std::lock_guard<std::mutex> lk(mu);
  if (!ready[dev]) {
    cudaError_t e = cudaSuccess;
    for (int i = 0; i < CL_VARIANTS && e == cudaSuccess; ++i)
      e = cudaFuncSetAttribute(cl_variant(i).fn, cudaFuncAttributeMaxDynamicSharedMemorySize, cl_variant(i).smem);
    for (int i = 0; i < CL_VARIANTS && e == cudaSuccess; ++i) {
      for (int c = 1; c <= CL_MAX_CS && e == cudaSuccess; ++c) {
        cudaLaunchConfig_t cfg;
        std::memset(&cfg, 0, sizeof(cfg));
        cfg.gridDim = dim3(c, 1, 1);
        cfg.blockDim = dim3(cl_variant(i).threads, 1, 1);
        cfg.dynamicSmemBytes = cl_variant(i).smem;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = c;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        e = cudaOccupancyMaxActiveClusters(&n, cl_variant(i).fn, &cfg);
        cache[dev][i][c] = n;
      }
    }
    if (e != cudaSuccess) {
      set_error("refadapt_q_delta: cluster occupancy query: %s", cudaGetErrorString(e));
      cudaGetLastError();
      return -1;
    }
    ready[dev] = true;
  }
  return cache[dev][vi][cs];
}

}  // namespace qd
}  // namespace ra

extern "C" size_t refadapt_q_delta_workspace_size(int32_t B, int32_t H) {
  if (B < 1 || H < 1) return 0;
  const size_t bh = size_t(B) * size_t(H);
  const size_t counters = ((bh * sizeof(uint32_t)) + 255) / 256 * 256;
  // refadapt_q_delta_gate: the heads' score terms and a ticket counter
  return counters + bh * ra::qd::MAX_SPLITS * sizeof(float4) + (bh * sizeof(float2) + 255) / 256 * 256 + 256;
}

namespace ra {
namespace qd {

// Argument checks shared by both entry points (everything but the workspace).
ra_status validate(const char* who, const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                   float eps, const float* d_out) {
  if (!q_cur || !q_prev || !d_out) {
    set_error("%s: NULL argument", who);
    return RA_EINVAL;
  }
  if (d != 64 && d != 128) {
    set_error("%s: d = %d (supported: 64, 128)", who, d);
    return RA_EINVAL;
  }
  if (B < 1 || H < 1 || B > 65535 || H > 65535) {
    set_error("%s: B = %d, H = %d out of range", who, B, H);
    return RA_EINVAL;
  }
  if (!check_seg(*q_cur, who, false) || !check_seg(*q_prev, who, false)) return RA_EINVAL;
  if (q_cur->n != q_prev->n || q_cur->n < 1) {
    set_error("%s: q_cur.n = %d and q_prev.n = %d must be equal and >= 1", who, q_cur->n, q_prev->n);
    return RA_EINVAL;
  }
  if (!(eps >= 0.f)) {
    set_error("%s: eps must be >= 0", who);
    return RA_EINVAL;
  }
  const int rows_per_unit = UNIT_BYTES / (2 * d);
  const int64_t units = int64_t(B) * H * ((q_cur->n + rows_per_unit - 1) / rows_per_unit);
  if (units > (int64_t(1) << 30)) {
    set_error("%s: problem too large", who);
    return RA_EINVAL;
  }
  return RA_OK;
}

// Picks the cluster path or the multi-block path and launches it, after
// validate(). The workspace is touched only by the multi-block path; with
// clear_counters its ticket counters are zeroed on the stream right before
// that kernel (for a workspace whose earlier contents are unknown).
// With `fuse` (refadapt_q_delta_gate) the gate runs on the new D: inside the
// cluster kernel, or as its own launch behind the multi-block kernel.
ra_status launch(const char* who, const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                 float eps, float* d_out, void* workspace, bool clear_counters, void* stream,
                 const gate::Params* fuse = nullptr) {
  const int n = q_cur->n;
  const int bh = B * H;
  {
    // Cluster path. Stages S = 12 (one CTA per SM, 192 KB in flight) or
    // S = 6 (two CTAs per SM); cluster size cs <= 8. Clusters live inside one GPC,
    // so how many fit at once depends on the GPU's floorplan: the runtime's
    // occupancy query says, and only configurations whose B * H clusters all
    // run in one wave are candidates. Among those the one with the most bytes
    // in flight (CTAs x stages) wins. Taken when it occupies at least 60 % of
    // the CTAs the multi-block path would run (min(SMs, units)).
    const int rows_per_unit = CL_UNIT_BYTES / (2 * d);
    const int per_slab = (n + rows_per_unit - 1) / rows_per_unit;
    const int64_t sms = num_sms();
    int best_v = -1, best_cs = 0;
    int64_t best_score = 0;
    for (int vi = 0; vi < CL_VARIANTS; ++vi) {
      const int S = cl_variant(vi).S;
      for (int cs = 1; cs <= CL_MAX_CS && cs <= per_slab; ++cs) {
        if ((per_slab + cs - 1) / cs > CL_MAX_UNITS) continue;
        const int fit = max_active_clusters(vi, cs);
        if (fit < 0) return RA_ECUDA;
        if (bh > fit) continue;
        const int64_t score = int64_t(bh) * cs * S;
        if (score > best_score) {
          best_score = score;
          best_v = vi;
          best_cs = cs;
        }
      }
    }
    // The multi-block path's units are 12 KB.
    const int64_t units_all = int64_t(bh) * ((int64_t(n) * d * 2 + UNIT_BYTES - 1) / UNIT_BYTES);
    const int64_t ticket_ctas = units_all < sms ? units_all : sms;
    if (best_v >= 0 && double(bh) * best_cs >= 0.6 * double(ticket_ctas)) {
      const ClVariant& cv = cl_variant(best_v);
      ClusterParams c;
      std::memset(&c, 0, sizeof(c));
      c.bulk = (q_cur->stride_n == d && q_prev->stride_n == d) ? 1 : 0;
      c.base_c = static_cast<const char*>(q_cur->ptr);
      c.base_p = static_cast<const char*>(q_prev->ptr);
      c.c_sb = q_cur->stride_b * 2;
      c.c_sh = q_cur->stride_h * 2;
      c.p_sb = q_prev->stride_b * 2;
      c.p_sh = q_prev->stride_h * 2;
      c.slab_bytes = int64_t(n) * d * 2;
      c.H = H;
      c.rows_per_unit = rows_per_unit;
      c.per_slab = per_slab;
      c.cs = best_cs;
      for (int r = 0; r <= best_cs; ++r) c.k_begin[r] = int(int64_t(r) * per_slab / best_cs);
      c.eps = eps;
      c.d_out = d_out;
      c.budget_ns = wait_budget_ns();
      if (fuse) {
        const size_t counters = ((size_t(bh) * sizeof(uint32_t)) + 255) / 256 * 256;
        char* tail = static_cast<char*>(workspace) + counters + size_t(bh) * MAX_SPLITS * sizeof(float4);
        c.fuse_gate = 1;
        c.gate_terms = reinterpret_cast<float2*>(tail);
        c.gate_ticket = reinterpret_cast<uint32_t*>(tail + (size_t(bh) * sizeof(float2) + 255) / 256 * 256);
        c.gp = *fuse;
      }
      if (!c.bulk && (!encode_seg(&c.tm_c, *q_cur, B, H, d, d, rows_per_unit, false) ||
                      !encode_seg(&c.tm_p, *q_prev, B, H, d, d, rows_per_unit, false)))
        return RA_EINVAL;
      cudaLaunchConfig_t cfg;
      std::memset(&cfg, 0, sizeof(cfg));
      cfg.gridDim = dim3(best_cs, H, B);
      cfg.blockDim = dim3(cv.threads, 1, 1);
      cfg.dynamicSmemBytes = cv.smem;
      cfg.stream = static_cast<cudaStream_t>(stream);
      cudaLaunchAttribute attr[2];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = best_cs;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      // may overlap the previous kernel's tail (the kernel waits for it with
      // griddepcontrol.wait before touching global memory)
      attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[1].val.programmaticStreamSerializationAllowed = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 2;
      const cudaError_t e = cudaLaunchKernelEx(&cfg, cv.fn, c);
      if (e != cudaSuccess) {
        set_error("%s: cluster launch failed: %s", who, cudaGetErrorString(e));
        cudaGetLastError();
        return RA_ECUDA;
      }
      return launch_status(who);
    }
  }
  Params p;
  p.H = H;
  p.rows_per_unit = UNIT_BYTES / (2 * d);
  p.per_slab = (n + p.rows_per_unit - 1) / p.rows_per_unit;
  const int64_t units = int64_t(bh) * p.per_slab;
  p.units = int(units);
  // One CTA per SM; at most MAX_SPLITS - 1 CTAs may share a slab (slots) and
  // at most MAX_UNITS_PER_CTA units may fall to one CTA.
  int64_t G = num_sms();
  if (G > units) G = units;
  if (G > int64_t(MAX_SPLITS - 1) * bh) G = int64_t(MAX_SPLITS - 1) * bh;
  while ((units + G - 1) / G > MAX_UNITS_PER_CTA) G *= 2;
  if (G > units) G = units;
  if (G > int64_t(MAX_SPLITS - 1) * bh || G > 2147483647) {
    set_error("%s: n = %d rows per slab is too large", who, n);
    return RA_EINVAL;
  }
  p.grid = int(G);
  p.eps = eps;
  p.d_out = d_out;
  const size_t counters = ((size_t(bh) * sizeof(uint32_t)) + 255) / 256 * 256;
  p.counter = static_cast<uint32_t*>(workspace);
  p.partial = reinterpret_cast<float4*>(static_cast<char*>(workspace) + counters);
  p.budget_ns = wait_budget_ns();
  p.bulk = (q_cur->stride_n == d && q_prev->stride_n == d) ? 1 : 0;
  p.base_c = static_cast<const char*>(q_cur->ptr);
  p.base_p = static_cast<const char*>(q_prev->ptr);
  p.c_sb = q_cur->stride_b * 2;
  p.c_sh = q_cur->stride_h * 2;
  p.p_sb = q_prev->stride_b * 2;
  p.p_sh = q_prev->stride_h * 2;
  p.slab_bytes = int64_t(n) * d * 2;
  if (p.bulk) {
    // Units are byte ranges of a slab; rows_per_unit * d * 2 == UNIT_BYTES either way.
    std::memset(&p.tm_c, 0, sizeof(p.tm_c));
    std::memset(&p.tm_p, 0, sizeof(p.tm_p));
  } else if (!encode_seg(&p.tm_c, *q_cur, B, H, d, d, p.rows_per_unit, false) ||
             !encode_seg(&p.tm_p, *q_prev, B, H, d, d, p.rows_per_unit, false)) {
    return RA_EINVAL;
  }
  const ra_status as = ensure_dynamic_smem(reinterpret_cast<const void*>(q_delta_kernel), SMEM_ALLOC, who);
  if (as != RA_OK) return as;
  if (clear_counters) {
    const cudaError_t e = cudaMemsetAsync(workspace, 0, counters, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
      set_error("%s: cudaMemsetAsync: %s", who, cudaGetErrorString(e));
      cudaGetLastError();
      return RA_ECUDA;
    }
  }
  q_delta_kernel<<<p.grid, THREADS, SMEM_ALLOC, static_cast<cudaStream_t>(stream)>>>(p);
  const ra_status ls = launch_status(who);
  if (ls != RA_OK || !fuse) return ls;
  return gate::launch(*fuse, static_cast<cudaStream_t>(stream), who);
}

}  // namespace qd
}  // namespace ra

extern "C" ra_status refadapt_q_delta(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                                      float eps, float* d_out, void* workspace, size_t workspace_bytes,
                                      void* stream) {
  using namespace ra;
  clear_error();
  const char* who = "refadapt_q_delta";
  const ra_status v = qd::validate(who, q_cur, q_prev, B, H, d, eps, d_out);
  if (v != RA_OK) return v;
  if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 16 != 0 ||
      workspace_bytes < refadapt_q_delta_workspace_size(B, H)) {
    set_error("%s: workspace must be non-NULL, 16-byte aligned and >= %zu bytes", who,
              refadapt_q_delta_workspace_size(B, H));
    return RA_EINVAL;
  }
  return qd::launch(who, q_cur, q_prev, B, H, d, eps, d_out, workspace, false, stream);
}

extern "C" ra_status refadapt_q_delta_gate(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H,
                                           int32_t d, float eps, float* d_out, void* workspace,
                                           size_t workspace_bytes, const ra_gate_args* gate, void* stream) {
  using namespace ra;
  clear_error();
  const char* who = "refadapt_q_delta_gate";
  const ra_status v = qd::validate(who, q_cur, q_prev, B, H, d, eps, d_out);
  if (v != RA_OK) return v;
  if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 16 != 0 ||
      workspace_bytes < refadapt_q_delta_workspace_size(B, H)) {
    set_error("%s: workspace must be non-NULL, 16-byte aligned and >= %zu bytes", who,
              refadapt_q_delta_workspace_size(B, H));
    return RA_EINVAL;
  }
  if (!gate) {
    set_error("%s: gate args are NULL", who);
    return RA_EINVAL;
  }
  if (gate->B != B || gate->H != H || gate->t < 1 || (gate->q_delta && gate->q_delta != d_out)) {
    set_error("%s: the gate's B, H must match, t must be >= 1 and q_delta must be NULL or d_out", who);
    return RA_EINVAL;
  }
  ra_gate_args ga = *gate;
  ga.q_delta = d_out;
  gate::Params gp;
  const ra_status gv = gate::make_params(&ga, who, &gp);
  if (gv != RA_OK) return gv;
  return qd::launch(who, q_cur, q_prev, B, H, d, eps, d_out, workspace, false, stream, &gp);
}

// ---------------------------------------------------------------------------
// No-allocation variant: the workspace is a file-scope static device array.
// Host code must not hand the array's name to a kernel (it is a host-side
// stand-in); the device address comes from cudaGetSymbolAddress with the
// device current, looked up once per CUDA context (a context torn down by
// cudaDeviceReset and created again gets the address looked up anew).
namespace ra {
namespace qd {

constexpr int kNoAllocMaxBH = RA_Q_DELTA_NOALLOC_MAX_BH;
constexpr size_t kNoAllocCounterBytes = ((size_t(kNoAllocMaxBH) * sizeof(uint32_t)) + 255) / 256 * 256;
constexpr size_t kNoAllocBytes = kNoAllocCounterBytes + size_t(kNoAllocMaxBH) * MAX_SPLITS * sizeof(float4);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {
struct NoAllocSlot {
  uint64_t ctx_id;  // context the address belongs to; 0 = none looked up yet
  void* ptr;
};
std::mutex g_noalloc_mu;
NoAllocSlot g_noalloc[64] = {};
}  // namespace

// Device address of g_noalloc_scratch in the current context (nullptr + error on failure).
void* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    set_error("refadapt_q_delta_noalloc: no usable current device");
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  NoAllocSlot& slot = g_noalloc[dev];
  const uint64_t ctx = current_context_id();  // 0: no context yet, or unknown
  if (ctx != 0 && slot.ctx_id == ctx && slot.ptr != nullptr) return slot.ptr;
  // The lookup makes the device's primary context current when no context is.
  void* ptr = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
  if (e != cudaSuccess || ptr == nullptr) {
    cudaGetLastError();
    set_error("refadapt_q_delta_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
    return nullptr;
  }
  slot.ctx_id = current_context_id();  // 0 (unknown): looked up again on the next call
  slot.ptr = ptr;
  return ptr;
}

}  // namespace qd
}  // namespace ra

extern "C" ra_status refadapt_q_delta_noalloc(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H,
                                              int32_t d, float eps, float* d_out, void* stream) {
  using namespace ra;
  clear_error();
  const char* who = "refadapt_q_delta_noalloc";
  const ra_status v = qd::validate(who, q_cur, q_prev, B, H, d, eps, d_out);
  if (v != RA_OK) return v;
  if (int64_t(B) * H > qd::kNoAllocMaxBH) {
    set_error("%s: B * H = %lld exceeds %d, the size of the static scratch; use refadapt_q_delta with a "
              "workspace",
              who, (long long)B * H, qd::kNoAllocMaxBH);
    return RA_EINVAL;
  }
  void* scratch = qd::noalloc_scratch();
  if (scratch == nullptr) return RA_ECUDA;
  // The array keeps the last call's contents: the multi-block path clears its
  // ticket counters before its kernel (the cluster path does not touch it).
  return qd::launch(who, q_cur, q_prev, B, H, d, eps, d_out, scratch, true, stream);
}
