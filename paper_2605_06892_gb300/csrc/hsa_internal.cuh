// Internal helpers shared by the libhsa translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "hsa.h"

namespace hsa {

// Device-side error word bits.  Kernels never trap: they skip the offending
// access, set a bit here with atomicOr, and hsa_get_device_error() maps the
// lowest set bit back to a status code.
enum : unsigned {
  kErrIndex = 1u << 0,
  kErrNonfinite = 1u << 1,
  kErrTimeout = 1u << 2,
};

// Device address of this device's error word (resolved once per device).
unsigned *device_error_word();

// Number of SMs of the current device (cached per device).
int sm_count();

// Adds n to the process-wide count of kernels this library has launched
// (read through hsa_launch_count); called next to every launch.
void count_launches(int n);

inline int launch_status() {
  return cudaGetLastError() == cudaSuccess ? HSA_OK : HSA_ERR_CUDA;
}

inline bool aligned16(const void *p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

// Programmatic dependent launch, for the kernels of one HSA iteration: a
// kernel launched with launch_pdl may be launched while the kernel before it
// in the stream is still running.  It calls pdl_wait() before it touches
// global memory: the wait returns once that kernel has completed and its
// writes are visible (and, since that kernel waited the same way, every
// earlier one).  pdl_trigger() lets the next kernel be launched; a kernel
// that never calls it does so when its blocks exit.  Outside such a launch
// both are no-ops.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline void launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

__device__ __forceinline__ void set_error(unsigned *err, unsigned bit) {
  atomicOr(err, bit);
}

// Number of lanes that cooperate on one row of `vecs` 16-byte vectors:
// a power of two, at most 32.
inline int lanes_per_row(long long vecs) {
  int l = 1;
  while (l < 32 && l < vecs) l <<= 1;
  return l;
}

}  // namespace hsa
