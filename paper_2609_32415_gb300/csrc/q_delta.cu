// refadapt_q_delta: relative L2 change of the target query per (sample, head),
// D = ||q_t - q_{t-1}||_F / (||q_{t-1}||_F + eps)   (paper Eq. 1, Sec. 4).
//
// HBM-bound: each (sample, head) slab of n rows x d columns is split into
// `splits` row ranges, one CTA each, sized so the grid covers every SM several
// times. A CTA streams both tensors with 16-byte loads (several in flight per
// thread), accumulates sum (q_t - q_{t-1})^2 and sum q_{t-1}^2 in fp32 per
// thread, reduces them in fp64 across the CTA in a fixed order and stores the
// pair in the workspace. The last CTA of a slab to finish (ticket counter in
// the workspace) adds the pairs in split order and writes D, then re-arms the
// counter, so results are deterministic and the workspace is ready for the
// next call.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

#include "api_common.h"

namespace ra {
namespace qd {

constexpr int THREADS = 256;
constexpr int MAX_SPLITS = 128;
constexpr int UNROLL = 8;

struct Params {
  const __nv_bfloat16* qc;
  const __nv_bfloat16* qp;
  int64_t c_sb, c_sh, c_sn;
  int64_t p_sb, p_sh, p_sn;
  int32_t H, n, vec_per_row;  // vec = 8 bf16 = 16 bytes
  int32_t splits, rows_per_split;
  float eps;
  float* d_out;
  double* partial;     // [B*H][MAX_SPLITS][2]
  uint32_t* counter;   // [B*H]
};

__device__ __forceinline__ void acc16(const uint4& a, const uint4& b, float& sd, float& sp) {
  const __nv_bfloat162* x = reinterpret_cast<const __nv_bfloat162*>(&a);
  const __nv_bfloat162* y = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 fx = __bfloat1622float2(x[i]);
    const float2 fy = __bfloat1622float2(y[i]);
    const float d0 = fx.x - fy.x, d1 = fx.y - fy.y;
    sd = fmaf(d0, d0, sd);
    sd = fmaf(d1, d1, sd);
    sp = fmaf(fy.x, fy.x, sp);
    sp = fmaf(fy.y, fy.y, sp);
  }
}

// Thread t always reads the same 16-byte column v = t % vec_per_row of rows
// r0 + t / vec_per_row, stepping THREADS / vec_per_row rows at a time, so the
// loop needs no division and a warp reads whole contiguous rows.
__global__ void __launch_bounds__(THREADS) q_delta_kernel(const Params p) {
  const int split = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int bh = b * p.H + h;
  const int r0 = split * p.rows_per_split;
  const int r1 = min(p.n, r0 + p.rows_per_split);
  const int vpr = p.vec_per_row;
  const int rstep = THREADS / vpr;
  const int v = threadIdx.x % vpr;
  const __nv_bfloat16* qc = p.qc + b * p.c_sb + h * p.c_sh + v * 8;
  const __nv_bfloat16* qp = p.qp + b * p.p_sb + h * p.p_sh + v * 8;
  float sd = 0.f, sp = 0.f;
  int row = r0 + threadIdx.x / vpr;
  for (; row + (UNROLL - 1) * rstep < r1; row += UNROLL * rstep) {
    uint4 a[UNROLL], c[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int64_t rr = row + u * rstep;
      a[u] = __ldg(reinterpret_cast<const uint4*>(qc + rr * p.c_sn));
      c[u] = __ldg(reinterpret_cast<const uint4*>(qp + rr * p.p_sn));
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) acc16(a[u], c[u], sd, sp);
  }
  for (; row < r1; row += rstep) {
    const uint4 a = __ldg(reinterpret_cast<const uint4*>(qc + int64_t(row) * p.c_sn));
    const uint4 c = __ldg(reinterpret_cast<const uint4*>(qp + int64_t(row) * p.p_sn));
    acc16(a, c, sd, sp);
  }
  // CTA reduction in fp64, fixed order.
  double dd = sd, dp = sp;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    dd += __shfl_xor_sync(0xffffffffu, dd, o);
    dp += __shfl_xor_sync(0xffffffffu, dp, o);
  }
  __shared__ double red[2][THREADS / 32];
  __shared__ bool last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red[0][warp] = dd;
    red[1][warp] = dp;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double td = 0.0, tp = 0.0;
    for (int w = 0; w < THREADS / 32; ++w) {
      td += red[0][w];
      tp += red[1][w];
    }
    double* slot = p.partial + (int64_t(bh) * MAX_SPLITS + split) * 2;
    slot[0] = td;
    slot[1] = tp;
    __threadfence();
    const uint32_t ticket = atomicAdd(p.counter + bh, 1u);
    last = (ticket == uint32_t(p.splits - 1));
  }
  __syncthreads();
  if (last && warp == 0) {
    // The slab's last CTA: lane i adds splits i, i + 32, ... (L2 reads), then
    // a butterfly finishes the sum; the order is fixed, so D is deterministic.
    __threadfence();
    const double* base = p.partial + int64_t(bh) * MAX_SPLITS * 2;
    double td = 0.0, tp = 0.0;
    for (int s = lane; s < p.splits; s += 32) {
      td += __ldcg(base + 2 * s);
      tp += __ldcg(base + 2 * s + 1);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      td += __shfl_xor_sync(0xffffffffu, td, o);
      tp += __shfl_xor_sync(0xffffffffu, tp, o);
    }
    if (lane == 0) {
      p.d_out[bh] = float(sqrt(td) / (sqrt(tp) + double(p.eps)));
      p.counter[bh] = 0u;  // re-arm for the next call
    }
  }
}

}  // namespace qd
}  // namespace ra

extern "C" size_t refadapt_q_delta_workspace_size(int32_t B, int32_t H) {
  if (B < 1 || H < 1) return 0;
  const size_t bh = size_t(B) * size_t(H);
  const size_t counters = ((bh * sizeof(uint32_t)) + 255) / 256 * 256;
  return counters + bh * ra::qd::MAX_SPLITS * 2 * sizeof(double);
}

extern "C" ra_status refadapt_q_delta(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H, int32_t d,
                                      float eps, float* d_out, void* workspace, size_t workspace_bytes,
                                      void* stream) {
  using namespace ra;
  clear_error();
  if (!q_cur || !q_prev || !d_out || !workspace) {
    set_error("refadapt_q_delta: NULL argument");
    return RA_EINVAL;
  }
  if (d != 64 && d != 128) {
    set_error("refadapt_q_delta: d = %d (supported: 64, 128)", d);
    return RA_EINVAL;
  }
  if (B < 1 || H < 1 || B > 65535 || H > 65535) {
    set_error("refadapt_q_delta: B = %d, H = %d out of range", B, H);
    return RA_EINVAL;
  }
  if (!check_seg(*q_cur, "refadapt_q_delta: q_cur", false) || !check_seg(*q_prev, "refadapt_q_delta: q_prev", false))
    return RA_EINVAL;
  if (q_cur->n != q_prev->n || q_cur->n < 1) {
    set_error("refadapt_q_delta: q_cur.n = %d and q_prev.n = %d must be equal and >= 1", q_cur->n, q_prev->n);
    return RA_EINVAL;
  }
  if (!(eps >= 0.f)) {
    set_error("refadapt_q_delta: eps must be >= 0");
    return RA_EINVAL;
  }
  if (reinterpret_cast<uintptr_t>(workspace) % 16 != 0 || workspace_bytes < refadapt_q_delta_workspace_size(B, H)) {
    set_error("refadapt_q_delta: workspace must be 16-byte aligned and >= %zu bytes",
              refadapt_q_delta_workspace_size(B, H));
    return RA_EINVAL;
  }
  const int n = q_cur->n;
  const int bh = B * H;
  // Enough CTAs to cover every SM about four times, at least 8 rows each.
  const int want = (4 * num_sms() + bh - 1) / bh;
  int splits = want < 1 ? 1 : want;
  if (splits > qd::MAX_SPLITS) splits = qd::MAX_SPLITS;
  const int max_by_rows = (n + 7) / 8;
  if (splits > max_by_rows) splits = max_by_rows;
  const int rps = (n + splits - 1) / splits;
  splits = (n + rps - 1) / rps;

  qd::Params p;
  p.qc = static_cast<const __nv_bfloat16*>(q_cur->ptr);
  p.qp = static_cast<const __nv_bfloat16*>(q_prev->ptr);
  p.c_sb = q_cur->stride_b;
  p.c_sh = q_cur->stride_h;
  p.c_sn = q_cur->stride_n;
  p.p_sb = q_prev->stride_b;
  p.p_sh = q_prev->stride_h;
  p.p_sn = q_prev->stride_n;
  p.H = H;
  p.n = n;
  p.vec_per_row = d / 8;
  p.splits = splits;
  p.rows_per_split = rps;
  p.eps = eps;
  p.d_out = d_out;
  const size_t counters = ((size_t(bh) * sizeof(uint32_t)) + 255) / 256 * 256;
  p.counter = static_cast<uint32_t*>(workspace);
  p.partial = reinterpret_cast<double*>(static_cast<char*>(workspace) + counters);
  dim3 grid(splits, H, B);
  qd::q_delta_kernel<<<grid, qd::THREADS, 0, static_cast<cudaStream_t>(stream)>>>(p);
  return launch_status("refadapt_q_delta");
}

// ---------------------------------------------------------------------------
// No-allocation variant: the workspace is a file-scope static device array.
// Host code must not hand the array's name to a kernel (it is a host-side
// stand-in); the device address comes from cudaGetSymbolAddress, looked up
// once per device with that device current.
namespace ra {
namespace qd {

constexpr int kNoAllocMaxBH = RA_Q_DELTA_NOALLOC_MAX_BH;
constexpr size_t kNoAllocCounterBytes = ((size_t(kNoAllocMaxBH) * sizeof(uint32_t)) + 255) / 256 * 256;
constexpr size_t kNoAllocBytes = kNoAllocCounterBytes + size_t(kNoAllocMaxBH) * MAX_SPLITS * 2 * sizeof(double);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[64] = {nullptr};
}  // namespace

// Device address of g_noalloc_scratch on the current device (nullptr + error on failure).
void* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    set_error("refadapt_q_delta_noalloc: no usable current device");
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (g_noalloc_ptr[dev] == nullptr) {
    void* ptr = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr) {
      set_error("refadapt_q_delta_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
      return nullptr;
    }
    g_noalloc_ptr[dev] = ptr;
  }
  return g_noalloc_ptr[dev];
}

}  // namespace qd
}  // namespace ra

extern "C" ra_status refadapt_q_delta_noalloc(const ra_seg* q_cur, const ra_seg* q_prev, int32_t B, int32_t H,
                                              int32_t d, float eps, float* d_out, void* stream) {
  using namespace ra;
  clear_error();
  if (B < 1 || H < 1 || int64_t(B) * H > qd::kNoAllocMaxBH) {
    set_error("refadapt_q_delta_noalloc: B * H = %lld outside [1, %d], the size of the static scratch; "
              "use refadapt_q_delta with a workspace",
              (long long)B * H, qd::kNoAllocMaxBH);
    return RA_EINVAL;
  }
  void* scratch = qd::noalloc_scratch();
  if (scratch == nullptr) return RA_ECUDA;
  // The ticket counters must start at zero; the array keeps the last call's contents.
  const size_t counters = ((size_t(B) * H * sizeof(uint32_t)) + 255) / 256 * 256;
  const cudaError_t e = cudaMemsetAsync(scratch, 0, counters, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    set_error("refadapt_q_delta_noalloc: cudaMemsetAsync: %s", cudaGetErrorString(e));
    return RA_ECUDA;
  }
  return refadapt_q_delta(q_cur, q_prev, B, H, d, eps, d_out, scratch, qd::kNoAllocBytes, stream);
}
