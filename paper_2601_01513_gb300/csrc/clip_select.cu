// K3: CLIP entity alignment (Eq. 14-15) with the keep threshold, and
// K4: candidate selection (masked mean log-prob; Algorithm 1's two stages,
// Eq. 12-13 and the final argmax over alignment).
//
// At the paper's sizes both steps move kilobytes to a few megabytes and are
// latency-bound.  K3 reads every frame embedding once per group of 16 candidates:
// a warp scores 16 frames against all of them with mma.sync tensor-core tiles (the
// contraction is [16 frames x E] x [E x 16 candidates], too small in M for tcgen05
// tiles), so with many frames it streams at HBM rates; a query's frames are split
// over a cluster of up to 8 CTAs whose per-candidate bests are merged in distributed
// shared memory (the cluster size is picked from how many clusters fit the GPU at once).
// K4 uses one CTA per query.
#include <cuda_fp16.h>

#include <algorithm>
#include <mutex>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {

constexpr int kClipThreads = 512;
constexpr int kClipWarps = kClipThreads / 32;
constexpr int kClipKG = 16;      // candidates a CTA scores against each frame (two MMA n-tiles)
constexpr int kClipTile = 16;    // frames per warp tile (MMA m)
constexpr int kClipUnroll = 4;   // 32-element chunks of E in flight per thread
constexpr int kClipMaxDim = 4096;
constexpr int kClipMaxSplit = 8; // CTAs (one cluster) sharing one query's frames
constexpr int kClipPad = 8;      // fp16 elements of padding per candidate row in shared memory

__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_s32(uint32_t addr, int v) {
  asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

// (v, i) beats (bv, bi): larger cosine, or equal cosine and lower frame index.
__device__ __forceinline__ bool clip_better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// D = A * B + D for one m16n8k16 tile: A 16 x 16 fp16 (row), B 16 x 8 fp16 (col), fp32 D.
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Grid: Qn x G x S CTAs, blockIdx.x = (q * G + g) * S + s, in clusters of S along x.
// CTA (q, g, s) scores frames [s F / S, (s + 1) F / S) of query q against candidates
// k0 .. k0 + kg - 1 (k0 = 16 g): every frame is read once per group of 16 candidates.
//
// The dot products are tensor-core tiles: a warp takes 16 frames as the A operand (rows)
// and the 16 candidates as B (two n-tiles of 8), accumulating fp32 over E.  The order in
// which E enters the contraction does not change the sums, so lane (r, t) (r = lane / 4,
// t = lane % 4) loads elements [32 c + 8 t, 32 c + 8 t + 8) of frames r and r + 8 and of
// candidates r and r + 8 with 16-byte loads and uses them as its fragment pairs of two
// consecutive k16 steps; A and B pair up the same elements.  The frames' squared norms
// come from two more MMAs of the frame tile against itself (B = the tile's own rows), of
// which the diagonal is kept.  Each lane then holds the cosines of frames r, r + 8 with
// candidates 2t, 2t + 1, 2t + 8, 2t + 9; the per-candidate best (cos, frame) is reduced over
// the warp, the CTA and, through rank 0's shared memory, the cluster, which writes max_cos,
// argmax and keep.
__global__ void __launch_bounds__(kClipThreads) clip_align_kernel(
    const __half* __restrict__ cand, const __half* __restrict__ frames, int K, int F, int E,
    float tau, float* __restrict__ cos_out, float* __restrict__ max_cos, int32_t* __restrict__ argmax,
    uint8_t* __restrict__ keep, int G, int S) {
  extern __shared__ __align__(16) __half c_s[];     // [kClipKG][E + kClipPad], then the
                                                    // accumulator exchange [warps][32][16] fp32
  __shared__ float inv_e_s[kClipKG];
  __shared__ float red_v[kClipWarps][kClipKG];
  __shared__ int red_i[kClipWarps][kClipKG];
  __shared__ float part_v[kClipMaxSplit][kClipKG];  // rank 0: one row per CTA of the cluster
  __shared__ int part_i[kClipMaxSplit][kClipKG];
  griddep_wait();
  griddep_launch_dependents();
  const int s = blockIdx.x % S;
  const int qg = blockIdx.x / S;
  const int g = qg % G, q = qg / G;
  const int k0 = g * kClipKG, kg = min(kClipKG, K - k0);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int r = lane >> 2, t = lane & 3;
  const int nchunk = E >> 3;                          // 16-byte chunks per row
  const int ldc = E + kClipPad;

  // candidates k0 .. k0 + kg - 1 (rows past kg are zero) and their inverse norms
  for (int idx = tid; idx < kClipKG * nchunk; idx += kClipThreads) {
    const int k = idx / nchunk, c = idx - k * nchunk;
    const uint4 raw = k < kg ? __ldg(reinterpret_cast<const uint4*>(cand + ((size_t)q * K + k0 + k) * E) + c)
                             : make_uint4(0u, 0u, 0u, 0u);
    *reinterpret_cast<uint4*>(&c_s[(size_t)k * ldc + 8 * c]) = raw;
  }
  __syncthreads();
  for (int k = warp; k < kClipKG; k += kClipWarps) {
    float ee = 0.f;
    for (int i = lane; i < E; i += 32) {
      const float v = __half2float(c_s[(size_t)k * ldc + i]);
      ee = fmaf(v, v, ee);
    }
    ee = warp_sum(ee);
    if (lane == 0) inv_e_s[k] = ee > 0.f ? rsqrtf(ee) : 0.f;
  }
  __syncthreads();
  const float ie0 = inv_e_s[2 * t], ie1 = inv_e_s[2 * t + 1];
  const float ie8 = inv_e_s[2 * t + 8], ie9 = inv_e_s[2 * t + 9];

  const int fa = (int)(((long long)s * F) / S), fb = (int)(((long long)(s + 1) * F) / S);
  const __half* fq = frames + (size_t)q * F * E;
  const __half* c_lo = c_s + (size_t)r * ldc + 8 * t;          // candidate r
  const __half* c_hi = c_s + (size_t)(r + 8) * ldc + 8 * t;    // candidate r + 8
  const int nc32 = (E + 31) >> 5;                              // 32-element chunks
  // With few frame tiles, ne warps share a tile, each over a slice of E, and add their
  // accumulators through shared memory before the epilogue (warp part 0).
  const int ntile = (fb - fa + kClipTile - 1) / kClipTile;
  int ne = 1;
  while (ne < 8 && 2 * ne * ntile <= kClipWarps && 2 * ne <= nc32) ne *= 2;
  const int part = warp % ne, tpi = kClipWarps / ne;
  const int c_beg = (part * nc32) / ne, c_end = ((part + 1) * nc32) / ne;
  const int iters = (ntile + tpi - 1) / tpi;
  float* xch = reinterpret_cast<float*>(c_s + (size_t)kClipKG * ldc);   // [warps][16][32]
  // running best of candidates 2t, 2t+1, 2t+8, 2t+9 over this warp's frames
  float bv[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
  int bi[4] = {0x7fffffff, 0x7fffffff, 0x7fffffff, 0x7fffffff};
  for (int it = 0; it < iters; ++it) {
    const int tile = warp / ne + it * tpi;
    const int f0 = fa + tile * kClipTile;
    const int fr0 = f0 + r, fr1 = f0 + r + 8;
    const bool v0 = tile < ntile && fr0 < fb, v1 = tile < ntile && fr1 < fb;
    const uint4* p0 = reinterpret_cast<const uint4*>(fq + (size_t)(v0 ? fr0 : fa) * E + 8 * t);
    const uint4* p1 = reinterpret_cast<const uint4*>(fq + (size_t)(v1 ? fr1 : fa) * E + 8 * t);
    float acc[16];              // candidates 0-7 | 8-15 | frames x frames 0-7 | 8-15
#pragma unroll
    for (int i = 0; i < 16; ++i) acc[i] = 0.f;
    float(&dc0)[4] = *reinterpret_cast<float(*)[4]>(&acc[0]);
    float(&dc1)[4] = *reinterpret_cast<float(*)[4]>(&acc[4]);
    float(&nn0)[4] = *reinterpret_cast<float(*)[4]>(&acc[8]);
    float(&nn1)[4] = *reinterpret_cast<float(*)[4]>(&acc[12]);
    for (int cb = c_beg; cb < c_end; cb += kClipUnroll) {
      uint4 a_lo[kClipUnroll], a_hi[kClipUnroll];
#pragma unroll
      for (int u = 0; u < kClipUnroll; ++u) {
        const int c = cb + u;
        const bool in = c < c_end && 32 * c + 8 * t < E;
        a_lo[u] = (in && v0) ? __ldg(p0 + 4 * c) : make_uint4(0u, 0u, 0u, 0u);
        a_hi[u] = (in && v1) ? __ldg(p1 + 4 * c) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kClipUnroll; ++u) {
        const int c = cb + u;
        const bool in = c < c_end && 32 * c + 8 * t < E;
        const uint4 b_lo = in ? *reinterpret_cast<const uint4*>(c_lo + 32 * c) : make_uint4(0u, 0u, 0u, 0u);
        const uint4 b_hi = in ? *reinterpret_cast<const uint4*>(c_hi + 32 * c) : make_uint4(0u, 0u, 0u, 0u);
        // k16 step 1: elements 8t .. 8t+3 of the chunk; step 2: 8t+4 .. 8t+7
        mma_f16_16816(dc0, a_lo[u].x, a_hi[u].x, a_lo[u].y, a_hi[u].y, b_lo.x, b_lo.y);
        mma_f16_16816(dc0, a_lo[u].z, a_hi[u].z, a_lo[u].w, a_hi[u].w, b_lo.z, b_lo.w);
        mma_f16_16816(dc1, a_lo[u].x, a_hi[u].x, a_lo[u].y, a_hi[u].y, b_hi.x, b_hi.y);
        mma_f16_16816(dc1, a_lo[u].z, a_hi[u].z, a_lo[u].w, a_hi[u].w, b_hi.z, b_hi.w);
        mma_f16_16816(nn0, a_lo[u].x, a_hi[u].x, a_lo[u].y, a_hi[u].y, a_lo[u].x, a_lo[u].y);
        mma_f16_16816(nn0, a_lo[u].z, a_hi[u].z, a_lo[u].w, a_hi[u].w, a_lo[u].z, a_lo[u].w);
        mma_f16_16816(nn1, a_lo[u].x, a_hi[u].x, a_lo[u].y, a_hi[u].y, a_hi[u].x, a_hi[u].y);
        mma_f16_16816(nn1, a_lo[u].z, a_hi[u].z, a_lo[u].w, a_hi[u].w, a_hi[u].z, a_hi[u].w);
      }
    }
    if (ne > 1) {                 // part 0 adds the other parts' accumulators
#pragma unroll
      for (int i = 0; i < 16; ++i) xch[((size_t)warp * 16 + i) * 32 + lane] = acc[i];
      __syncthreads();
      if (part == 0)
        for (int pp = 1; pp < ne; ++pp)
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[i] += xch[((size_t)(warp + pp) * 16 + i) * 32 + lane];
      __syncthreads();
    }
    if (part != 0 || tile >= ntile) continue;
    // |f_r|^2 sits in lane (r, r / 2) as nn0[r & 1]; |f_{r+8}|^2 there as nn1[2 + (r & 1)]
    const float d_lo = (r & 1) ? nn0[1] : nn0[0];
    const float d_hi = (r & 1) ? nn1[3] : nn1[2];
    const int src = 4 * r + (r >> 1);
    const float n_lo = __shfl_sync(0xffffffffu, d_lo, src);
    const float n_hi = __shfl_sync(0xffffffffu, d_hi, src);
    const float if0 = n_lo > 0.f ? rsqrtf(n_lo) : 0.f;
    const float if1 = n_hi > 0.f ? rsqrtf(n_hi) : 0.f;
    // dc0 = {C[r][2t], C[r][2t+1], C[r+8][2t], C[r+8][2t+1]}, dc1 the same for candidates + 8
    const float iek[4] = {ie0, ie1, ie8, ie9};
    const int kk[4] = {2 * t, 2 * t + 1, 2 * t + 8, 2 * t + 9};
    const float dlo[4] = {dc0[0], dc0[1], dc1[0], dc1[1]};   // frame r
    const float dhi[4] = {dc0[2], dc0[3], dc1[2], dc1[3]};   // frame r + 8
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const bool kv = kk[j] < kg;
      const float c_a = (if0 > 0.f && iek[j] > 0.f) ? dlo[j] * iek[j] * if0 : 0.f;
      const float c_b = (if1 > 0.f && iek[j] > 0.f) ? dhi[j] * iek[j] * if1 : 0.f;
      if (kv && v0) {
        if (cos_out) cos_out[((size_t)q * K + k0 + kk[j]) * F + fr0] = c_a;
        if (clip_better(c_a, fr0, bv[j], bi[j])) { bv[j] = c_a; bi[j] = fr0; }
      }
      if (kv && v1) {
        if (cos_out) cos_out[((size_t)q * K + k0 + kk[j]) * F + fr1] = c_b;
        if (clip_better(c_b, fr1, bv[j], bi[j])) { bv[j] = c_b; bi[j] = fr1; }
      }
    }
  }
  // over the 8 lanes that share t (the tile's rows)
#pragma unroll
  for (int j = 0; j < 4; ++j) {
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv[j], o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi[j], o);
      if (clip_better(ov, oi, bv[j], bi[j])) { bv[j] = ov; bi[j] = oi; }
    }
  }
  if (r == 0) {
    red_v[warp][2 * t] = bv[0];     red_i[warp][2 * t] = bi[0];
    red_v[warp][2 * t + 1] = bv[1]; red_i[warp][2 * t + 1] = bi[1];
    red_v[warp][2 * t + 8] = bv[2]; red_i[warp][2 * t + 8] = bi[2];
    red_v[warp][2 * t + 9] = bv[3]; red_i[warp][2 * t + 9] = bi[3];
  }
  __syncthreads();
  float v = -INFINITY;
  int vi = 0x7fffffff;
  if (tid < kClipKG) {
#pragma unroll
    for (int w = 0; w < kClipWarps; ++w)
      if (clip_better(red_v[w][tid], red_i[w][tid], v, vi)) {
        v = red_v[w][tid];
        vi = red_i[w][tid];
      }
  }
  if (S > 1) {
    if (tid < kClipKG) {
      st_cluster_f32(mapa_shared(smem_u32(&part_v[s][tid]), 0), v);
      st_cluster_s32(mapa_shared(smem_u32(&part_i[s][tid]), 0), vi);
    }
    cluster_sync();
    if (s != 0) return;
    if (tid < kClipKG) {
      v = part_v[0][tid];
      vi = part_i[0][tid];
      for (int rr = 1; rr < S; ++rr)
        if (clip_better(part_v[rr][tid], part_i[rr][tid], v, vi)) {
          v = part_v[rr][tid];
          vi = part_i[rr][tid];
        }
    }
  }
  if (tid < kg) {
    const size_t qk = (size_t)q * K + k0 + tid;
    max_cos[qk] = v;
    argmax[qk] = vi;
    keep[qk] = v >= tau ? 1 : 0;
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
        const float m = max_cos[(size_t)q * K + k];
        const float a = isnan(m) ? -INFINITY : m;       // NaN ranks below every number
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

// Clusters of S CTAs of clip_align_kernel that can be resident at once (S <= 8), cached
// per device and shared-memory size.
static int clip_max_clusters(int S, int smem) {
  static std::mutex mu;
  static int cache_dev[64] = {0}, cache_smem[64] = {0}, cache_n[64][kClipMaxSplit + 1] = {{0}};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cache_dev[dev] == 0 || cache_smem[dev] != smem) {
    for (int k = 0; k <= kClipMaxSplit; ++k) cache_n[dev][k] = -1;
    cache_dev[dev] = 1;
    cache_smem[dev] = smem;
  }
  if (cache_n[dev][S] < 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S);
    cfg.blockDim = dim3(kClipThreads);
    cfg.dynamicSmemBytes = (size_t)smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, clip_align_kernel, &cfg) != cudaSuccess) n = 0;
    cudaGetLastError();
    cache_n[dev][S] = n;
  }
  return cache_n[dev][S];
}

// CTAs per (query, candidate group): about 256 frames each, at most 8 (one cluster), and
// among those the split that finishes soonest when `groups` clusters share the GPU: each
// CTA's work scales as 1 / S and the clusters run in ceil(groups / resident(S)) waves (on a
// GB300, 15 clusters of 8 fit at once but 36 of 4: 16 queries x 8 CTAs took two waves).
static int clip_split(int F, long long groups, int smem) {
  int smax = 1;
  while (smax < kClipMaxSplit && (long long)smax * 256 < F && 2 * smax <= F) smax *= 2;
  int best = 1;
  double best_cost = 0.0;
  for (int S = 1; S <= smax; ++S) {
    const int n = S == 1 ? 0 : clip_max_clusters(S, smem);
    const long long per_wave = S == 1 ? std::max(1, sm_count()) : n;
    if (per_wave <= 0) continue;
    const double cost = (double)((groups + per_wave - 1) / per_wave) / S;
    if (S == 1 || cost < best_cost) {
      best = S;
      best_cost = cost;
    }
  }
  return best;
}

extern "C" fvrag_status fvrag_clip_align(const fvrag_clip_desc* d, const void* cand_emb,
                                         const void* frame_emb, float* cos, float* max_cos,
                                         int32_t* argmax, uint8_t* keep, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_clip_align");
  if (!d || !cand_emb || !frame_emb || !max_cos || !argmax || !keep) return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_cand < 1 || d->num_frames < 1 || d->dim < 1 || d->flags != 0)
    return FVRAG_ERR_INVALID_ARG;
  if (d->dim % 8 != 0 || d->dim > kClipMaxDim) return FVRAG_ERR_UNSUPPORTED;
  if ((int64_t)d->num_queries * d->num_cand > 0x7fffffff) return FVRAG_ERR_UNSUPPORTED;
  if (!aligned16(cand_emb) || !aligned16(frame_emb)) return FVRAG_ERR_MISALIGNED;
  const int G = (d->num_cand + kClipKG - 1) / kClipKG;
  const size_t smem = (size_t)kClipKG * (d->dim + kClipPad) * sizeof(__half) +
                      (size_t)kClipWarps * 16 * 32 * sizeof(float);
  if (cudaFuncSetAttribute(clip_align_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  const int S = clip_split(d->num_frames, (long long)d->num_queries * G, (int)smem);
  const long long blocks = (long long)d->num_queries * G * S;
  if (blocks > 0x7fffffffLL) return FVRAG_ERR_UNSUPPORTED;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(kClipThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = reinterpret_cast<cudaStream_t>(stream);
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (counted(cudaLaunchKernelEx(&cfg, clip_align_kernel,
                                 reinterpret_cast<const __half*>(cand_emb),
                                 reinterpret_cast<const __half*>(frame_emb), d->num_cand,
                                 d->num_frames, d->dim, d->threshold, cos, max_cos, argmax, keep,
                                 G, S)) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

extern "C" fvrag_status fvrag_select_candidate(const fvrag_select_desc* d, const float* logprob,
                                               const int32_t* lengths, const uint8_t* keep,
                                               const float* max_cos, float* score,
                                               int32_t* selected, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_select_candidate");
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
