// Host-side helpers shared by the library's translation units.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "hdl.h"

#ifndef HDL_NO_NVTX
#include <nvtx3/nvToolsExt.h>
#endif

namespace hdl {

// Names the enclosing entry point on profiler timelines (an NVTX range, seen
// by nsys and by ncu's NVTX filters); without a tool attached it costs a few
// nanoseconds.  Build with -DHDL_NO_NVTX to drop it.
struct HostRange {
#ifndef HDL_NO_NVTX
  explicit HostRange(const char* name) { nvtxRangePushA(name); }
  ~HostRange() { nvtxRangePop(); }
#else
  explicit HostRange(const char*) {}
#endif
  HostRange(const HostRange&) = delete;
  HostRange& operator=(const HostRange&) = delete;
};

inline bool aligned_to(const void* p, uintptr_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

// Number of SMs of the current device (queried per call; cheap).
inline int current_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

inline hdl_status launch_status() {
  return cudaGetLastError() == cudaSuccess ? HDL_OK : HDL_ERR_CUDA;
}

constexpr int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
constexpr size_t align_up(size_t a, size_t b) { return (a + b - 1) / b * b; }

}  // namespace hdl
