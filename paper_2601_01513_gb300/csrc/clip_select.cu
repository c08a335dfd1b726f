// K3: CLIP entity alignment (Eq. 14-15) with the keep threshold, and
// K4: candidate selection (masked mean log-prob; Algorithm 1's two stages,
// Eq. 12-13 and the final argmax over alignment).
//
// Both steps move kilobytes to a few megabytes, so they are latency-bound:
// K3 uses one CTA per (query, candidate), 16 warps with four frames' 16-byte
// loads in flight per warp; K4 uses one CTA per query.
#include <cuda_fp16.h>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {

constexpr int kClipThreads = 512;
constexpr int kClipUnroll = 4;   // frames in flight per warp
constexpr int kClipMaxDim = 4096;

// One CTA per (query q, candidate k).  The candidate embedding is widened to
// fp32 in shared memory; warp w handles frames w, w + 16, w + 32, w + 48 together
// (then the next 64): the 32 lanes split the E dimension in 16-byte (8 x fp16)
// chunks with the four frames' loads in flight at once, reduce <e, f> and |f|^2
// with shuffles, and lane 0 keeps the warp's best (cos, frame).  The 16 warp
// results are then reduced by one warp: larger cos wins, equal cos goes to the
// lower frame index.
__global__ void __launch_bounds__(kClipThreads) clip_align_kernel(
    const __half* __restrict__ cand, const __half* __restrict__ frames, int K, int F, int E,
    float tau, float* __restrict__ cos_out, float* __restrict__ max_cos, int32_t* __restrict__ argmax,
    uint8_t* __restrict__ keep) {
  __shared__ __align__(16) float e_s[kClipMaxDim];
  __shared__ float red[kClipThreads / 32];
  __shared__ float best_v[kClipThreads / 32];
  __shared__ int best_i[kClipThreads / 32];
  griddep_wait();
  griddep_launch_dependents();
  const int qk = blockIdx.x;
  const int q = qk / K;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nchunk = E >> 3;

  const __half* e = cand + (size_t)qk * E;
  float ee_part = 0.f;
  for (int c = threadIdx.x; c < nchunk; c += kClipThreads) {
    const uint4 raw = __ldg(reinterpret_cast<const uint4*>(e) + c);
    const __half2* h2 = reinterpret_cast<const __half2*>(&raw);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __half22float2(h2[j]);
      e_s[8 * c + 2 * j] = f.x;
      e_s[8 * c + 2 * j + 1] = f.y;
      ee_part = fmaf(f.x, f.x, fmaf(f.y, f.y, ee_part));
    }
  }
  ee_part = warp_sum(ee_part);
  if (lane == 0) red[warp] = ee_part;
  __syncthreads();
  float ee = 0.f;
#pragma unroll
  for (int w = 0; w < kClipThreads / 32; ++w) ee += red[w];
  const float inv_e = ee > 0.f ? rsqrtf(ee) : 0.f;

  constexpr int NW = kClipThreads / 32;
  float wbest = -INFINITY;
  int wbest_i = 0x7fffffff;
  const __half* fq = frames + (size_t)q * F * E;
  for (int f0 = warp; f0 < F; f0 += NW * kClipUnroll) {
    float dot[kClipUnroll], ff[kClipUnroll];
#pragma unroll
    for (int u = 0; u < kClipUnroll; ++u) dot[u] = ff[u] = 0.f;
    for (int c = lane; c < nchunk; c += 32) {
      const float4 ea = *reinterpret_cast<const float4*>(&e_s[8 * c]);
      const float4 eb = *reinterpret_cast<const float4*>(&e_s[8 * c + 4]);
      uint4 raw[kClipUnroll];
#pragma unroll
      for (int u = 0; u < kClipUnroll; ++u) {
        const int f = f0 + u * NW;
        raw[u] = f < F ? __ldg(reinterpret_cast<const uint4*>(fq + (size_t)f * E) + c)
                       : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < kClipUnroll; ++u) {
        const __half2* h2 = reinterpret_cast<const __half2*>(&raw[u]);
        const float2 f0v = __half22float2(h2[0]), f1v = __half22float2(h2[1]);
        const float2 f2v = __half22float2(h2[2]), f3v = __half22float2(h2[3]);
        float d = dot[u], n = ff[u];
        d = fmaf(ea.x, f0v.x, d); d = fmaf(ea.y, f0v.y, d);
        d = fmaf(ea.z, f1v.x, d); d = fmaf(ea.w, f1v.y, d);
        d = fmaf(eb.x, f2v.x, d); d = fmaf(eb.y, f2v.y, d);
        d = fmaf(eb.z, f3v.x, d); d = fmaf(eb.w, f3v.y, d);
        n = fmaf(f0v.x, f0v.x, n); n = fmaf(f0v.y, f0v.y, n);
        n = fmaf(f1v.x, f1v.x, n); n = fmaf(f1v.y, f1v.y, n);
        n = fmaf(f2v.x, f2v.x, n); n = fmaf(f2v.y, f2v.y, n);
        n = fmaf(f3v.x, f3v.x, n); n = fmaf(f3v.y, f3v.y, n);
        dot[u] = d;
        ff[u] = n;
      }
    }
#pragma unroll
    for (int u = 0; u < kClipUnroll; ++u) {
      const int f = f0 + u * NW;
      const float dsum = warp_sum(dot[u]);
      const float nsum = warp_sum(ff[u]);
      if (f < F && lane == 0) {
        const float c = (nsum > 0.f && inv_e > 0.f) ? dsum * inv_e * rsqrtf(nsum) : 0.f;
        if (cos_out) cos_out[(size_t)qk * F + f] = c;
        if (c > wbest) {  // a warp sees its frames in increasing order: strict > keeps the lowest
          wbest = c;
          wbest_i = f;
        }
      }
    }
  }
  if (lane == 0) {
    best_v[warp] = wbest;
    best_i[warp] = wbest_i;
  }
  __syncthreads();
  if (warp == 0) {
    float v = lane < NW ? best_v[lane] : -INFINITY;
    int i = lane < NW ? best_i[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, v, o);
      const int oi = __shfl_xor_sync(0xffffffffu, i, o);
      if (ov > v || (ov == v && oi < i)) {
        v = ov;
        i = oi;
      }
    }
    if (lane == 0) {
      max_cos[qk] = v;
      argmax[qk] = i;
      keep[qk] = v >= tau ? 1 : 0;
    }
  }
}

// SplitMix64 (Steele, Lea & Flood 2014): output n of the generator seeded with s.
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t s, uint64_t n) {
  uint64_t z = s + (n + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// One CTA per query; thread k scores candidate k in fp64 (fixed summation
// order l = 0 .. n_k-1), then thread 0 runs the selection rule serially
// (K <= 1024 candidates).
__global__ void select_kernel(const float* __restrict__ logprob, const int32_t* __restrict__ lengths,
                              const uint8_t* __restrict__ keep, const float* __restrict__ max_cos,
                              int K, int L, int G, int mode, double delta, uint64_t seed,
                              float* __restrict__ score, int32_t* __restrict__ selected) {
  extern __shared__ double sc[];
  griddep_wait();
  griddep_launch_dependents();
  const int q = blockIdx.x;
  const double nan = __longlong_as_double(0x7ff8000000000000ll);
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const size_t qk = (size_t)q * K + k;
    const int n = lengths ? lengths[qk] : L;
    double s = nan;
    if (mode == FVRAG_SEL_RANDOM) {
      s = 0.0;
    } else if (n >= 1 && n <= L) {
      const float* lp = logprob + qk * L * G;
      if (mode == FVRAG_SEL_MASKED_MEAN_LOGPROB) {
        double acc = 0.0;
#pragma unroll 8
        for (int l = 0; l < n; ++l) acc += (double)lp[(size_t)l * G];
        s = acc / (double)n;
      } else if (mode == FVRAG_SEL_ALIGNMENT_ONLY) {
        s = (double)max_cos[qk];
      } else {
        const double lpY = lp[(size_t)(n - 1) * G + 0];
        const double lpN = lp[(size_t)(n - 1) * G + 1];
        s = 1.0 / (1.0 + exp(lpN - lpY));   // Eq. 12
        if (mode == FVRAG_SEL_ADDITION) s += (double)max_cos[qk];
      }
    }
    sc[k] = s;
    score[qk] = (float)s;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int sel = -1;
    if (mode == FVRAG_SEL_RANDOM) {
      const uint64_t x = splitmix64_at(seed, (uint64_t)q);
      sel = (int)(((x >> 32) * (uint64_t)K) >> 32);
    } else if (mode == FVRAG_SEL_TWO_STAGE) {
      double top = -INFINITY;
      for (int k = 0; k < K; ++k)
        if (!isnan(sc[k]) && sc[k] > top) top = sc[k];
      float best = -INFINITY;
      for (int k = 0; k < K; ++k) {
        const double s = sc[k];
        if (isnan(s) || !(s >= top - delta)) continue;   // Eq. 13
        const float a = max_cos[(size_t)q * K + k];
        if (sel < 0 || a > best) {
          best = a;
          sel = k;
        }
      }
    } else {
      const bool masked = mode == FVRAG_SEL_MASKED_MEAN_LOGPROB || mode == FVRAG_SEL_INVERT;
      double best = -INFINITY;
      for (int k = 0; k < K; ++k) {
        const double s = sc[k];
        if (isnan(s) || (masked && !keep[(size_t)q * K + k])) continue;
        if (sel < 0 || s > best) {
          best = s;
          sel = k;
        }
      }
    }
    selected[q] = sel;
  }
}

}  // namespace fvrag

using namespace fvrag;

extern "C" fvrag_status fvrag_clip_align(const fvrag_clip_desc* d, const void* cand_emb,
                                         const void* frame_emb, float* cos, float* max_cos,
                                         int32_t* argmax, uint8_t* keep, fvrag_stream_t stream) {
  if (!d || !cand_emb || !frame_emb || !max_cos || !argmax || !keep) return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_cand < 1 || d->num_frames < 1 || d->dim < 1 || d->flags != 0)
    return FVRAG_ERR_INVALID_ARG;
  if (d->dim % 8 != 0 || d->dim > kClipMaxDim) return FVRAG_ERR_UNSUPPORTED;
  if ((int64_t)d->num_queries * d->num_cand > 0x7fffffff) return FVRAG_ERR_UNSUPPORTED;
  if (!aligned16(cand_emb) || !aligned16(frame_emb)) return FVRAG_ERR_MISALIGNED;
  const int blocks = d->num_queries * d->num_cand;
  if (launch_pdl(clip_align_kernel, dim3(blocks), dim3(kClipThreads), 0,
                 reinterpret_cast<cudaStream_t>(stream), reinterpret_cast<const __half*>(cand_emb),
                 reinterpret_cast<const __half*>(frame_emb), d->num_cand, d->num_frames, d->dim,
                 d->threshold, cos, max_cos, argmax, keep) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

extern "C" fvrag_status fvrag_select_candidate(const fvrag_select_desc* d, const float* logprob,
                                               const int32_t* lengths, const uint8_t* keep,
                                               const float* max_cos, float* score,
                                               int32_t* selected, fvrag_stream_t stream) {
  if (!d || !logprob || !score || !selected) return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_cand < 1 || d->cand_len < 1 || d->gathers < 1 || d->flags != 0)
    return FVRAG_ERR_INVALID_ARG;
  const int m = d->mode;
  if (m < FVRAG_SEL_MASKED_MEAN_LOGPROB || m > FVRAG_SEL_RANDOM) return FVRAG_ERR_INVALID_ARG;
  const bool needs_keep = m == FVRAG_SEL_MASKED_MEAN_LOGPROB || m == FVRAG_SEL_INVERT;
  const bool needs_cos = m == FVRAG_SEL_TWO_STAGE || m == FVRAG_SEL_ADDITION ||
                         m == FVRAG_SEL_ALIGNMENT_ONLY;
  const bool needs_rel = m == FVRAG_SEL_TWO_STAGE || m == FVRAG_SEL_ADDITION ||
                         m == FVRAG_SEL_INVERT || m == FVRAG_SEL_RELIABILITY_ONLY;
  if ((needs_keep && !keep) || (needs_cos && !max_cos) || (needs_rel && d->gathers < 2))
    return FVRAG_ERR_INVALID_ARG;
  if (d->num_cand > 1024) return FVRAG_ERR_UNSUPPORTED;
  const int threads = ((d->num_cand + 31) / 32) * 32;
  if (launch_pdl(select_kernel, dim3(d->num_queries), dim3(threads), sizeof(double) * d->num_cand,
                 reinterpret_cast<cudaStream_t>(stream), logprob, lengths, keep, max_cos,
                 d->num_cand, d->cand_len, d->gathers, d->mode, (double)d->delta, d->seed, score,
                 selected) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}
