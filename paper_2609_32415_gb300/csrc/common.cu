// Status strings, error message, wait budget and the error-word check.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "api_common.h"
#include "tc_ptx.cuh"

namespace ra {

namespace {
thread_local char g_err[512] = {0};
std::atomic<uint64_t> g_budget_ns{2000000000ull};
std::mutex g_sm_mu;
int g_sm_count[64] = {0};
}  // namespace

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}
void clear_error() { g_err[0] = 0; }

uint64_t wait_budget_ns() { return g_budget_ns.load(std::memory_order_relaxed); }

namespace {
struct SmemAttrKey {
  const void* func;
  int dev;
};
// Fixed-size record (no allocation, nothing that can throw across the ABI);
// past its capacity the attribute is simply set again on every call.
constexpr int kSmemAttrSlots = 256;
std::mutex g_smem_attr_mu;
SmemAttrKey g_smem_attr_done[kSmemAttrSlots];
int g_smem_attr_count = 0;
}  // namespace

ra_status ensure_dynamic_smem(const void* func, int bytes, const char* who) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    set_error("%s: cudaGetDevice: %s", who, cudaGetErrorString(e));
    return RA_ECUDA;
  }
  std::lock_guard<std::mutex> lk(g_smem_attr_mu);
  for (int i = 0; i < g_smem_attr_count; ++i)
    if (g_smem_attr_done[i].func == func && g_smem_attr_done[i].dev == dev) return RA_OK;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) {
    set_error("%s: cudaFuncSetAttribute: %s", who, cudaGetErrorString(e));
    return RA_ECUDA;
  }
  if (g_smem_attr_count < kSmemAttrSlots) g_smem_attr_done[g_smem_attr_count++] = {func, dev};
  return RA_OK;
}

int num_sms() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev < 0 || dev >= 64) dev = 0;
  std::lock_guard<std::mutex> lk(g_sm_mu);
  if (g_sm_count[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    g_sm_count[dev] = n;
  }
  return g_sm_count[dev];
}

uint64_t current_context_id() {
  using GetCurrentFn = CUresult (*)(CUcontext*);
  using GetIdFn = CUresult (*)(CUcontext, unsigned long long*);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(ptr);
    ptr = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &ptr, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(ptr);
  });
  if (!get_current || !get_id) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return uint64_t(id);
}

bool check_seg(const ra_seg& s, const char* what, bool allow_null_if_empty) {
  if (s.n < 0) {
    set_error("%s: n = %d is negative", what, s.n);
    return false;
  }
  if (s.ptr == nullptr) {
    if (s.n == 0 && allow_null_if_empty) return true;
    set_error("%s: ptr is NULL", what);
    return false;
  }
  if (reinterpret_cast<uintptr_t>(s.ptr) % 16 != 0) {
    set_error("%s: ptr is not 16-byte aligned", what);
    return false;
  }
  if (s.stride_b < 0 || s.stride_h < 0 || s.stride_n < 0) {
    set_error("%s: negative stride", what);
    return false;
  }
  if (s.stride_b % 8 || s.stride_h % 8 || s.stride_n % 8) {
    set_error("%s: strides must be multiples of 8 elements (16 bytes)", what);
    return false;
  }
  return true;
}

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

bool encode_seg(CUtensorMap* tm, const ra_seg& s, int B, int H, int d, int box_cols, int box_rows,
                bool swizzle128) {
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
  cuuint32_t box[4] = {cuuint32_t(box_cols), cuuint32_t(box_rows), 1u, 1u};
  cuuint32_t es[4] = {1u, 1u, 1u, 1u};
  CUresult r = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, s.ptr, dims, strides, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    set_error("cuTensorMapEncodeTiled failed (%d)", int(r));
    return false;
  }
  return true;
}

}  // namespace ra

extern "C" const char* refadapt_status_string(ra_status s) {
  switch (s) {
    case RA_OK: return "RA_OK";
    case RA_EINVAL: return "RA_EINVAL: invalid argument";
    case RA_EUNSUPPORTED: return "RA_EUNSUPPORTED: unsupported configuration";
    case RA_ECUDA: return "RA_ECUDA: CUDA error";
    case RA_ETIMEOUT: return "RA_ETIMEOUT: device wait ran out of its budget";
  }
  return "unknown ra_status";
}

extern "C" const char* refadapt_last_error(void) { return ra::g_err; }

extern "C" void refadapt_set_wait_budget_ns(uint64_t ns) {
  ra::g_budget_ns.store(ns == 0 ? 1 : ns, std::memory_order_relaxed);
}

extern "C" ra_status refadapt_check_error(int32_t* err_word, void* stream) {
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) {
    ra::set_error("refadapt_check_error: %s", cudaGetErrorString(cudaGetLastError()));
    return RA_ECUDA;
  }
  if (err_word == nullptr) return RA_OK;
  int32_t host = 0;
  if (cudaMemcpy(&host, err_word, sizeof(host), cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemset(err_word, 0, sizeof(int32_t)) != cudaSuccess) {
    ra::set_error("refadapt_check_error: %s", cudaGetErrorString(cudaGetLastError()));
    return RA_ECUDA;
  }
  if (host & 1) {
    ra::set_error("a device-side wait exceeded its budget");
    return RA_ETIMEOUT;
  }
  return RA_OK;
}

extern "C" int32_t refadapt_version(void) { return 1; }

namespace ra {
namespace {
__global__ void selftest_wait_kernel(int32_t* err, uint64_t budget_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const WaitCtl ctl{&abort_flag, err, budget_ns};
    (void)mbar_wait(&bar, 0, ctl);  // nothing arrives: returns false after budget_ns
  }
}
}  // namespace
}  // namespace ra

extern "C" ra_status refadapt_selftest_wait_timeout(int32_t* err_word, uint64_t budget_ns, void* stream) {
  ra::clear_error();
  if (!err_word) {
    ra::set_error("refadapt_selftest_wait_timeout: err_word is NULL");
    return RA_EINVAL;
  }
  if (budget_ns > 1000000000ull) budget_ns = 1000000000ull;
  ra::selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(err_word, budget_ns);
  return ra::launch_status("refadapt_selftest_wait_timeout");
}
