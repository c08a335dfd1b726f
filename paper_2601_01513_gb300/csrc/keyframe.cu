// Keyframe extraction (Eq. 1, the first loop of Algorithm 1): the colour
// histogram of every frame, the histogram-intersection similarity with the
// previous frame of the same video, the keyframe decision sim < theta and the
// compacted keyframe list.
//
// The histogram pass streams every pixel byte once and is HBM-bound
// (1280 x 720 RGB = 2.76 MB per frame).  Persistent grid, one CTA per SM, each
// CTA walks whole frames (frame blockIdx.x, then + gridDim.x, ...).  One warp
// streams each frame through a 4-deep shared-memory ring of 24 KB chunks with
// untiled bulk copies (cp.async.bulk, mbarrier completion); 16 consumer warps
// take 48 bytes (16 pixels) per thread per chunk, form the 9-bit joint bin of
// each pixel with byte-wise shifts and dot-product instructions, and count it in
// one of 32 private shared-memory histograms (one per lane index, rows padded
// to 513 words so equal bins of different lanes fall in different banks).  At
// the end of a frame the 32 copies are summed into the frame's histogram
// (plain stores, no global atomics) and cleared.
//
// A second kernel (one warp per frame) intersects consecutive histograms and
// takes the decision in fp64; a third (one CTA) compacts the keyframe ids.
#include <algorithm>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {
namespace kf {

constexpr int kBins = 512;
constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kThreads = kConsumers + 32;          // + one producer warp
constexpr int kGroupBytes = 48;                    // 16 RGB pixels per consumer thread
constexpr int kChunk = kConsumers * kGroupBytes;   // 24576 bytes per ring stage
constexpr int kStages = 4;
constexpr int kCopies = 32;
constexpr int kCopyStride = kBins + 1;
constexpr int kSmemBytes = kStages * kChunk + kCopies * kCopyStride * 4 + 128;

enum : uint32_t { kSiteProd = 0x401, kSiteCons = 0x402, kSiteDrain = 0x403 };

// Named barrier over the 16 consumer warps only (the producer warp never joins).
__device__ __forceinline__ void consumers_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kConsumers) : "memory");
}

// Bins of the four pixels packed in three words of top-3-bit values
// q = (bytes >> 5) & 7: pixel p starts at byte 3p.  __dp4a weights the bytes
// r, g, b by 64, 8, 1.
__device__ __forceinline__ void bins4(uint32_t q0, uint32_t q1, uint32_t q2, uint32_t (&b)[4]) {
  b[0] = __dp4a(q0, 0x00010840u, 0u);                              // bytes 0,1,2 of q0
  b[1] = __dp4a(q0, 0x40000000u, __dp4a(q1, 0x00000108u, 0u));     // byte 3 of q0, bytes 0,1 of q1
  b[2] = __dp4a(q1, 0x08400000u, __dp4a(q2, 0x00000001u, 0u));     // bytes 2,3 of q1, byte 0 of q2
  b[3] = __dp4a(q2, 0x01084000u, 0u);                              // bytes 1,2,3 of q2
}

__global__ void __launch_bounds__(kThreads, 1)
    hist_kernel(const uint8_t* __restrict__ pixels, int T, long long frame_bytes,
                int32_t* __restrict__ hist, uint32_t* status, uint64_t limit_ns) {
  extern __shared__ __align__(128) uint8_t smem[];
  uint8_t* ring = smem;
  uint32_t* copies = reinterpret_cast<uint32_t*>(smem + kStages * kChunk);
  uint64_t* full = reinterpret_cast<uint64_t*>(copies + kCopies * kCopyStride);
  uint64_t* empty = full + kStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(empty + kStages);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), kConsumerWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  for (int i = tid; i < kCopies * kCopyStride; i += kThreads) copies[i] = 0u;
  __syncthreads();
  griddep_wait();

  const int nchunks = (int)((frame_bytes + kChunk - 1) / kChunk);
  if (warp == kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t seq = 0;
      for (int f = blockIdx.x; f < T && !*abort_flag; f += gridDim.x) {
        const uint8_t* src = pixels + (long long)f * frame_bytes;
        for (int c = 0; c < nchunks; ++c, ++seq) {
          const int stage = seq % kStages;
          const uint32_t phase = (seq / kStages) & 1u;
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1u, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteProd);
            *abort_flag = 1;
            break;
          }
          const long long off = (long long)c * kChunk;
          const uint32_t bytes = (uint32_t)min((long long)kChunk, frame_bytes - off);
          mbar_arrive_expect_tx(smem_u32(&full[stage]), bytes);
          bulk_load(smem_u32(ring + stage * kChunk), src + off, bytes, smem_u32(&full[stage]), pol);
        }
      }
      // leave no copy in flight: the last (up to kStages) loads must have landed
      const uint32_t pend = seq < kStages ? seq : kStages;
      for (uint32_t i = 0; i < pend; ++i) {
        const uint32_t s = seq - 1 - i;
        if (!mbar_wait(smem_u32(&full[s % kStages]), (s / kStages) & 1u, limit_ns))
          record_error(status, FVRAG_ERR_TIMEOUT, kSiteDrain);
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    uint32_t* mine = copies + lane * kCopyStride;
    uint32_t seq = 0;
    for (int f = blockIdx.x; f < T; f += gridDim.x) {
      for (int c = 0; c < nchunks; ++c, ++seq) {
        const int stage = seq % kStages;
        const uint32_t phase = (seq / kStages) & 1u;
        bool ok = !*abort_flag;
        if (ok && !mbar_wait(smem_u32(&full[stage]), phase, limit_ns)) {
          record_error(status, FVRAG_ERR_TIMEOUT, kSiteCons);
          *abort_flag = 1;
          ok = false;
        }
        const long long off = (long long)c * kChunk;
        const int bytes = (int)min((long long)kChunk, frame_bytes - off);
        if (ok && tid * kGroupBytes < bytes) {
          const uint4* g = reinterpret_cast<const uint4*>(ring + stage * kChunk + tid * kGroupBytes);
          const uint4 a = g[0], b = g[1], d = g[2];
          const uint32_t w[12] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w, d.x, d.y, d.z, d.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            uint32_t bn[4];
            bins4((w[3 * k] >> 5) & 0x07070707u, (w[3 * k + 1] >> 5) & 0x07070707u,
                  (w[3 * k + 2] >> 5) & 0x07070707u, bn);
#pragma unroll
            for (int p = 0; p < 4; ++p) atomicAdd(&mine[bn[p]], 1u);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty[stage]));
      }
      // frame done: fold the 32 copies into its histogram and clear them
      consumers_sync();
      for (int bin = tid; bin < kBins; bin += kConsumers) {
        uint32_t s = 0;
#pragma unroll 8
        for (int k = 0; k < kCopies; ++k) {
          s += copies[k * kCopyStride + bin];
          copies[k * kCopyStride + bin] = 0u;
        }
        hist[(long long)f * kBins + bin] = (int32_t)s;
      }
      consumers_sync();
    }
  }
  griddep_launch_dependents();
  __syncthreads();
}

// sim[i] = sum_b min(h_i[b], h_{i-1}[b]) / npix (0 for the first frame of a video),
// is_key[i] = sim < theta with the quotient and the comparison in fp64.
__global__ void sim_kernel(const int32_t* __restrict__ hist, const int32_t* __restrict__ video_offsets,
                           int Nv, int T, long long npix, double theta, float* __restrict__ sim,
                           uint8_t* __restrict__ is_key) {
  griddep_wait();
  griddep_launch_dependents();
  const int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (i >= T) return;
  // the video holding frame i: the last v with video_offsets[v] <= i
  int lo = 0, hi = Nv - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (__ldg(&video_offsets[mid]) <= i) lo = mid;
    else hi = mid - 1;
  }
  const bool first = i == 0 || __ldg(&video_offsets[lo]) == i;
  long long inter = 0;
  if (!first) {
    const int4* a = reinterpret_cast<const int4*>(hist + (long long)i * kBins) + lane * 4;
    const int4* b = reinterpret_cast<const int4*>(hist + (long long)(i - 1) * kBins) + lane * 4;
    int s = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int4 x = a[k], y = b[k];
      s += min(x.x, y.x) + min(x.y, y.y) + min(x.z, y.z) + min(x.w, y.w);
    }
    inter = s;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) inter += __shfl_xor_sync(0xffffffffu, inter, o);
  }
  if (lane == 0) {
    const double q = (double)inter / (double)npix;
    sim[i] = (float)q;
    is_key[i] = q < theta ? 1 : 0;
  }
}

// key_index = ids of the frames with is_key set, in order; key_offsets[v] = the
// number of keyframes before video v's first frame.  One CTA of 1024 threads.
__global__ void __launch_bounds__(1024) compact_kernel(const uint8_t* __restrict__ is_key,
                                                       const int32_t* __restrict__ video_offsets,
                                                       int Nv, int T, int32_t* __restrict__ key_index,
                                                       int32_t* __restrict__ key_offsets) {
  __shared__ int warp_tot[32];
  griddep_wait();
  griddep_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (T + 1023) / 1024;
  const int i0 = min(T, tid * per), i1 = min(T, i0 + per);
  int cnt = 0;
  for (int i = i0; i < i1; ++i) cnt += is_key[i] ? 1 : 0;
  // exclusive scan of cnt over the block
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int t = warp_tot[lane];
    int ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += y;
    }
    warp_tot[lane] = ti - t;
  }
  __syncthreads();
  int pos = warp_tot[warp] + incl - cnt;
  for (int i = i0; i < i1; ++i)
    if (is_key[i]) key_index[pos++] = i;
  __shared__ int s_total;
  if (tid == 1023) s_total = warp_tot[31] + incl;   // exclusive prefix of warp 31 + its total
  __syncthreads();
  // key_offsets[v] = number of keyframes with id < video_offsets[v] (lower bound)
  for (int v = tid; v <= Nv; v += 1024) {
    const int target = video_offsets[v];
    int lo = 0, hi = s_total;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (key_index[mid] < target) lo = mid + 1;
      else hi = mid;
    }
    key_offsets[v] = lo;
  }
}

static size_t ws_bytes(const fvrag_keyframe_desc* d) {
  return kWsHeaderBytes + (size_t)d->total_frames * kBins * sizeof(int32_t);
}

}  // namespace kf
}  // namespace fvrag

using namespace fvrag;

extern "C" size_t fvrag_keyframes_workspace(const fvrag_keyframe_desc* d) {
  if (!d || d->num_videos < 1 || d->total_frames < 0) return 0;
  return kf::ws_bytes(d);
}

extern "C" fvrag_status fvrag_keyframes(const fvrag_keyframe_desc* d, const uint8_t* pixels,
                                        const int32_t* video_offsets, int32_t* hist, float* sim,
                                        uint8_t* is_key, int32_t* key_index, int32_t* key_offsets,
                                        void* ws, size_t ws_size, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_keyframes");
  using namespace kf;
  if (!d || !video_offsets || !sim || !is_key || !key_index || !key_offsets)
    return FVRAG_ERR_INVALID_ARG;
  if (d->num_videos < 1 || d->total_frames < 0 || d->height < 1 || d->width < 1 || d->flags != 0 ||
      !(d->theta > 0.0) || !(d->theta < 1e300))
    return FVRAG_ERR_INVALID_ARG;
  if (d->total_frames > 0 && !pixels) return FVRAG_ERR_INVALID_ARG;
  const long long npix = (long long)d->height * d->width;
  if (npix % 16 != 0) return FVRAG_ERR_MISALIGNED;  // frames must start on 16-byte boundaries
  if ((pixels && !aligned16(pixels)) || (hist && !aligned16(hist))) return FVRAG_ERR_MISALIGNED;
  if (!ws || ws_size < ws_bytes(d)) return FVRAG_ERR_WORKSPACE;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;

  uint8_t* base = reinterpret_cast<uint8_t*>(ws);
  uint32_t* status = reinterpret_cast<uint32_t*>(base);
  int32_t* h = hist ? hist : reinterpret_cast<int32_t*>(base + kWsHeaderBytes);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int T = d->total_frames;
  if (T > 0) {
    const int sms = sm_count() > 0 ? sm_count() : 148;
    const int ctas = std::max(1, std::min(T, sms));
    if (cudaFuncSetAttribute(hist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
        cudaSuccess)
      return FVRAG_ERR_CUDA;
    if (launch_pdl(hist_kernel, dim3(ctas), dim3(kThreads), (size_t)kSmemBytes, s, pixels, T,
                   npix * 3, h, status, wait_limit_ns()) != cudaSuccess)
      return FVRAG_ERR_CUDA;
    if (launch_pdl(sim_kernel, dim3((T + 7) / 8), dim3(256), 0, s, (const int32_t*)h, video_offsets,
                   d->num_videos, T, npix, d->theta, sim, is_key) != cudaSuccess)
      return FVRAG_ERR_CUDA;
  }
  if (launch_pdl(compact_kernel, dim3(1), dim3(1024), 0, s, (const uint8_t*)is_key, video_offsets,
                 d->num_videos, T, key_index, key_offsets) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}
