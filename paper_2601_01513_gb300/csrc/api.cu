// libfvrag: version, status strings, device status word, wait-limit control,
// the bounded-wait self-test, and the TMA descriptor encoder (driver entry
// point fetched through the runtime, so the library links without libcuda).
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

#include <cstdlib>
#include <cstring>
#include <nvtx3/nvToolsExt.h>

namespace fvrag {

static std::atomic<uint64_t> g_wait_limit_ns{1000000000ull};

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

bool nvtx_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("FVRAG_NVTX");
    return v != nullptr && v[0] != '\0' && std::strcmp(v, "0") != 0;
  }();
  return on;
}

NvtxRange::NvtxRange(const char* name) : on(nvtx_enabled()) {
  if (on) nvtxRangePushA(name);
}

NvtxRange::~NvtxRange() {
  if (on) nvtxRangePop();
}

static std::atomic<uint64_t> g_launches{0};

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int sm_count() {
  static std::mutex mu;
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    cache[dev] = n;
  }
  return cache[dev];
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

CUcontext current_cu_context() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
  });
  CUcontext c = nullptr;
  if (!fn || fn(&c) != CUDA_SUCCESS) return nullptr;
  return c;
}

static bool encode_tmap_16bit(CUtensorMap* map, CUtensorMapDataType dtype, const void* base,
                              int rank, const uint64_t* dims, const uint64_t* strides_bytes,
                              const uint32_t* box, bool swizzle128) {
  auto fn = encode_fn();
  if (!fn || rank < 1 || rank > 5) return false;
  cuuint64_t gdim[5], gstride[4];
  cuuint32_t bdim[5], estride[5];
  for (int i = 0; i < rank; ++i) {
    gdim[i] = dims[i];
    bdim[i] = box[i];
    estride[i] = 1;
    if (i > 0) gstride[i - 1] = strides_bytes[i - 1];
  }
  CUresult r = fn(map, dtype, (cuuint32_t)rank, const_cast<void*>(base), gdim, gstride, bdim,
                  estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_tmap_bf16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                      const uint64_t* strides_bytes, const uint32_t* box, bool swizzle128) {
  return encode_tmap_16bit(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base, rank, dims, strides_bytes,
                           box, swizzle128);
}

bool encode_tmap_f16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                     const uint64_t* strides_bytes, const uint32_t* box, bool swizzle128) {
  return encode_tmap_16bit(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base, rank, dims, strides_bytes,
                           box, swizzle128);
}

// One CTA, one thread: waits on a barrier whose phase never completes (its
// expected arrival count is 2 and only one arrival is ever made).
__global__ void selftest_wait_kernel(uint32_t* status, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 2);
    fence_barrier_init();
    mbar_arrive(b);
    if (!mbar_wait(b, 0, limit_ns)) record_error(status, FVRAG_ERR_TIMEOUT, 0xD1A6u);
  }
}

}  // namespace fvrag

using namespace fvrag;

extern "C" {

int fvrag_abi_version(void) { return FVRAG_ABI_VERSION; }

const char* fvrag_status_string(int s) {
  switch (s) {
    case FVRAG_OK: return "ok";
    case FVRAG_ERR_INVALID_ARG: return "invalid argument";
    case FVRAG_ERR_UNSUPPORTED: return "unsupported shape";
    case FVRAG_ERR_MISALIGNED: return "misaligned pointer or row pitch";
    case FVRAG_ERR_WORKSPACE: return "workspace missing or too small";
    case FVRAG_ERR_CUDA: return "CUDA error";
    case FVRAG_ERR_TIMEOUT: return "device wait timed out";
    default: return "unknown status";
  }
}

fvrag_status fvrag_read_status(const void* ws, fvrag_stream_t stream) {
  if (!ws) return FVRAG_ERR_INVALID_ARG;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return FVRAG_ERR_CUDA;
  uint32_t v = 0;
  if (cudaMemcpy(&v, ws, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return FVRAG_ERR_CUDA;
  return status_of_word(v);
}

fvrag_status fvrag_clear_status(void* ws, fvrag_stream_t stream) {
  if (!ws) return FVRAG_ERR_INVALID_ARG;
  if (cudaMemsetAsync(ws, 0, sizeof(WsHeader), reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  return FVRAG_OK;
}

void fvrag_set_wait_limit_ns(uint64_t ns) {
  g_wait_limit_ns.store(ns < 1000 ? 1000 : ns, std::memory_order_relaxed);
}

uint64_t fvrag_get_wait_limit_ns(void) { return wait_limit_ns(); }

fvrag_status fvrag_selftest_wait_timeout(void* ws, fvrag_stream_t stream) {
  if (!ws) return FVRAG_ERR_INVALID_ARG;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;
  selftest_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      reinterpret_cast<uint32_t*>(ws), wait_limit_ns());
  const fvrag_status st = launch_status();
  if (st == FVRAG_OK) count_launch();
  return st;
}

uint64_t fvrag_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"
