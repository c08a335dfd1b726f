// Host-side helpers shared by the libfvrag translation units (not exported).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "fvrag.h"

namespace fvrag {

// Current limit of the kernels' bounded waits, in nanoseconds.
uint64_t wait_limit_ns();

// Whether the public calls mark themselves with NVTX ranges: FVRAG_NVTX set in the
// environment (and not "0"), read once.
bool nvtx_enabled();

// An NVTX range (nvtxRangePushA / nvtxRangePop) around one public call, so that a profiler
// attached to the process (Nsight Systems, or ncu's NVTX filters) can group the kernels the
// call enqueues under the call's name.  Off unless nvtx_enabled(); with no tool attached the
// NVTX calls do nothing.
struct NvtxRange {
  bool on;
  explicit NvtxRange(const char* name);
  ~NvtxRange();
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Number of SMs of the current device (cached per device); 0 if it cannot be read.
int sm_count();

// SMs a call plans for: the device's count when `budget` is 0, else `budget`
// (callers have checked 0 <= budget <= sm_count()).
inline int sm_plan(int budget) {
  const int s = sm_count();
  return budget > 0 && (s <= 0 || budget <= s) ? budget : s;
}

// Records one kernel launch that the runtime accepted (fvrag_launch_count).
void count_launch();

// Passes a launch's result through, counting it when the runtime accepted it.
inline cudaError_t counted(cudaError_t e) {
  if (e == cudaSuccess) count_launch();
  return e;
}

// Tiled TMA descriptor over a row-major tensor of 16-bit elements.
//   dims[0] = innermost extent (elements), dims[i] = extent of dimension i,
//   strides_bytes[i-1] = byte stride of dimension i (multiple of 16),
//   box[i] = box extent in dimension i (box[0] * 2 bytes <= 128 with the 128-byte swizzle).
// Returns false when the driver rejects the description.
bool encode_tmap_bf16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                      const uint64_t* strides_bytes, const uint32_t* box, bool swizzle128);

// The same over fp16 elements.
bool encode_tmap_f16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                     const uint64_t* strides_bytes, const uint32_t* box, bool swizzle128);

// The CUDA context current on this thread (driver entry point fetched through the
// runtime), or null when none is current or the driver call is unavailable.
CUcontext current_cu_context();

// Status a workspace status word reports: OK when 0, TIMEOUT when both of its bits are set
// (codes are OR-ed in, and TIMEOUT's bits contain UNSUPPORTED's), else the recorded code.
inline fvrag_status status_of_word(uint32_t v) {
  if (v == 0) return FVRAG_OK;
  if ((v & FVRAG_ERR_TIMEOUT) == FVRAG_ERR_TIMEOUT) return FVRAG_ERR_TIMEOUT;
  return (fvrag_status)v;
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Launches `kernel` with programmatic stream serialization: its launch and
// prologue may overlap the tail of the previous kernel on the stream; the kernel
// itself calls griddep_wait() before touching global memory.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
  if (e == cudaSuccess) count_launch();
  return e;
}

inline fvrag_status launch_status() {
  return cudaGetLastError() == cudaSuccess ? FVRAG_OK : FVRAG_ERR_CUDA;
}

}  // namespace fvrag
