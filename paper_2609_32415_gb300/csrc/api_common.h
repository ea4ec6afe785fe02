// Host-side helpers shared by the C-ABI entry points: argument checks, the
// thread-local error message, device properties and the wait budget.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "refadapt.h"

namespace ra {

// Records a one-line reason for the last RA_EINVAL / RA_ECUDA of this thread.
void set_error(const char* fmt, ...);
void clear_error();

uint64_t wait_budget_ns();
int num_sms();  // of the current device (cached per device)

// Unique id of the CUDA context current in the calling thread; 0 when none is
// current yet or the driver cannot say. Changes nothing (no context is made
// current or created). A context torn down (cudaDeviceReset) and created
// again gets a new id, so state that belongs to a context (device addresses
// of module symbols) is keyed by it.
uint64_t current_context_id();

// Raises `func`'s dynamic shared-memory limit to `bytes` on the current
// device, once per (function, device): the attribute belongs to the device's
// context, so a process that drives several GPUs sets it on each. Returns
// RA_ECUDA with the reason recorded (prefixed by `who`) on failure.
ra_status ensure_dynamic_smem(const void* func, int bytes, const char* who);

// A bf16 segment usable by 16-byte vector access and by TMA: 16-byte aligned
// pointer and strides, n >= 0, non-negative strides. `what` names it in errors.
bool check_seg(const ra_seg& s, const char* what, bool allow_null_if_empty = true);

// 4-D TMA tensor map (c, n, head, sample) over one bf16 segment of head dim d,
// box box_cols x box_rows, 128-byte swizzle or none, zero fill out of bounds.
bool encode_seg(CUtensorMap* tm, const ra_seg& s, int B, int H, int d, int box_cols, int box_rows,
                bool swizzle128);

inline ra_status launch_status(const char* what) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_error("%s: launch failed: %s", what, cudaGetErrorString(e));
    return RA_ECUDA;
  }
  return RA_OK;
}

}  // namespace ra
