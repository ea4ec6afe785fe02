// refadapt_ref_cache_update: materialise a block's reference K/V (and an
// optional hidden-state tensor) into its cache slot for every sample whose mode
// is COMPUTE or FULL, and record a_b = t (paper Eq. 11; Algorithm 1).
//
// HBM-bound copy; the mode is read on the device, so no host sync is needed.
// When every (sample, head) slab of a tensor is contiguous (rows of exactly
// `width` elements, in source and cache alike) the copy is a stream of 32 KB
// bulk copies through shared memory: one thread per CTA keeps a 6-stage ring
// (loads run three chunks ahead of the bulk stores), so about 64 CTAs keep
// HBM busy. The copy runs beside the previous block's attention, whose CTAs
// fill an SM's registers, so each copy CTA holds an SM the attention cannot
// use: few CTAs with many bytes in flight take the fewest SM-microseconds.
// Other layouts take a grid-stride loop of 16-byte vectors per (tensor, sample).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "api_common.h"
#include "tc_ptx.cuh"

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

constexpr int BULK_STAGES = 6;
constexpr int BULK_LAG = 3;            // stores trail the loads by this many chunks
constexpr int CHUNK_BYTES = 32768;
constexpr int BULK_SMEM = BULK_STAGES * CHUNK_BYTES + BULK_STAGES * 8 + 1024;
constexpr int BULK_CTAS = 64;          // in all, over the (tensor, sample) pairs

// Bulk path: grid.y = tensor * B + sample; CTA x copies chunks [x C / G, (x+1) C / G)
// of that pair, C = heads * chunks per slab. One thread does everything.
__global__ void __launch_bounds__(32) copy_bulk_kernel(const Params p, int B, uint64_t budget_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + BULK_STAGES * CHUNK_BYTES);
  const int ti = blockIdx.y / B;
  const int s = blockIdx.y % B;
  if (threadIdx.x != 0) return;
  const int32_t m = __ldg(p.mode + s);
  if (!refreshes(m)) return;
  if (ti == 0 && blockIdx.x == 0 && p.a_b) p.a_b[s] = p.step;
  const Tensor& T = p.t[ti];
  if (T.src == T.dst) return;
  const int64_t slab = int64_t(p.n) * T.vec_per_row * 16;  // bytes
  const int64_t per_slab = (slab + CHUNK_BYTES - 1) / CHUNK_BYTES;
  const int64_t total = per_slab * T.heads;
  const int64_t c0 = int64_t(blockIdx.x) * total / gridDim.x;
  const int64_t c1 = int64_t(blockIdx.x + 1) * total / gridDim.x;
  const int n = int(c1 - c0);
  if (n <= 0) return;
  for (int i = 0; i < BULK_STAGES; ++i) mbar_init(full + i, 1);
  fence_mbar_init();
  const char* src = reinterpret_cast<const char*>(T.src + s * T.s_sb);
  char* dst = reinterpret_cast<char*>(T.dst + s * T.d_sb);
  auto where = [&](int64_t c, int64_t& soff, int64_t& doff, uint32_t& bytes) {
    const int64_t h = c / per_slab, k = c - h * per_slab;
    const int64_t off = k * CHUNK_BYTES;
    const int64_t rem = slab - off;
    bytes = uint32_t(rem < CHUNK_BYTES ? rem : CHUNK_BYTES);
    soff = h * T.s_sh * 2 + off;
    doff = h * T.d_sh * 2 + off;
  };
  bool ok = true;
  int issued = 0;  // chunks whose load was issued
  for (int i = 0; i < n + BULK_LAG; ++i) {
    if (i < n) {
      // The stage of chunk i last held chunk i - S, whose store was issued
      // S - 1 - LAG stores ago: at most that many may still be reading.
      if (i >= BULK_STAGES) asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(BULK_STAGES - 1 - BULK_LAG) : "memory");
      int64_t so, dof;
      uint32_t bytes;
      where(c0 + i, so, dof, bytes);
      uint64_t* bar = full + (i % BULK_STAGES);
      mbar_arrive_expect_tx(bar, bytes);
      bulk_load(smem + (i % BULK_STAGES) * CHUNK_BYTES, src + so, bytes, bar);
      ++issued;
    }
    const int j = i - BULK_LAG;
    if (j >= 0) {
      uint64_t* bar = full + (j % BULK_STAGES);
      if (!mbar_wait_drain(bar, uint32_t((j / BULK_STAGES) & 1), budget_ns)) {
        ok = false;
        break;
      }
      int64_t so, dof;
      uint32_t bytes;
      where(c0 + j, so, dof, bytes);
      asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst + dof),
                   "r"(smem_u32(smem + (j % BULK_STAGES) * CHUNK_BYTES)), "r"(bytes)
                   : "memory");
      asm volatile("cp.async.bulk.commit_group;" ::: "memory");
    }
  }
  // Every store complete (and its writes performed) before the CTA exits; after
  // a timeout, the loads still in flight land before the shared memory goes away.
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
  if (!ok) {
    for (int i = 0; i < BULK_STAGES && i < issued; ++i) {
      const int last = ((issued - 1 - i) / BULK_STAGES) * BULK_STAGES + i;  // last chunk loaded into stage i
      mbar_wait_drain(full + i, uint32_t((last / BULK_STAGES) & 1), budget_ns);
    }
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
  const int pairs = p.n_tensors * B;
  // Bulk path: every tensor's rows contiguous in source and cache.
  bool bulk = true;
  for (int i = 0; i < p.n_tensors; ++i) {
    const cu::Tensor& T = p.t[i];
    const int64_t w = int64_t(T.vec_per_row) * 8;
    if (T.s_sn != w || T.d_sn != w) bulk = false;
  }
  if (bulk) {
    const ra_status as =
        ensure_dynamic_smem(reinterpret_cast<const void*>(cu::copy_bulk_kernel), cu::BULK_SMEM, "refadapt_ref_cache_update");
    if (as != RA_OK) return as;
    const int per = (cu::BULK_CTAS + pairs - 1) / pairs;
    cu::copy_bulk_kernel<<<dim3(per, pairs), 32, cu::BULK_SMEM, st>>>(p, B, wait_budget_ns());
    return launch_status("refadapt_ref_cache_update");
  }
  // About four CTAs per SM over all (tensor, sample) pairs.
  int per = (4 * num_sms() + pairs - 1) / pairs;
  const int64_t vecs = int64_t(n) * H * (d / 8);
  const int64_t max_useful = (vecs + cu::THREADS - 1) / cu::THREADS;
  if (per > max_useful) per = int(max_useful);
  if (per < 1) per = 1;
  dim3 grid(per, pairs);
  cu::copy_kernel<<<grid, cu::THREADS, 0, st>>>(p, B);
  return launch_status("refadapt_ref_cache_update");
}
