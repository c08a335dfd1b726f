// Video-to-text retrieval (Eq. 2-3, the retrieval loop of Algorithm 1): every
// keyframe's k_frame most similar corpus texts by CLIP cosine, then per query the
// k_query best texts of the union of its keyframes' lists.
//
// Shape of the work: sim = frames[Fr x E] * texts[Nt x E]^T with Fr (keyframes of
// a batch of queries) small (1 .. 2048) and the corpus large (1,048,576 x 768
// fp16 = 1.6 GB).  It is the LM head's shape with a different epilogue, so the
// kernels have the same structure: a persistent grid, each CTA (or CTA pair)
// owning a contiguous range of texts (16-row units) and walking it in tiles of 256
// texts; per tile a tcgen05 GEMM accumulates frames_tile * texts_tile^T in tensor
// memory (fp16 inputs, fp32 accumulate), K-loop over E in 64-element blocks (one
// 128-byte swizzled row per operand row).
//
// Warp roles (192 threads):
//   warp 0     TMA producer (frame tiles 64 x 128, text tiles 64 x 64 / 64 x 16)
//              into a shared-memory ring;
//   warp 1     tensor-memory allocation and the single MMA-issuing lane;
//   warps 2-5  epilogue: tcgen05.ld of 32 columns (one keyframe per thread),
//              scale by the text's inverse norm, keep a running top-k_frame list
//              per keyframe (in shared memory between tiles).  Columns arrive in
//              increasing text id, so a strict > keeps the smaller id on ties.
// Two accumulator sets in tensor memory let the epilogue of one tile overlap the
// MMAs of the next.  Up to 128 keyframes: one CTA per SM (retrieve_kernel<256, 1>).
// More: clusters of two CTAs with tcgen05 cta_group::2 MMAs of M = 256 keyframes
// (retrieve_pair_kernel), each SM loading half of every text tile and its own 128
// keyframes of every 256-row pair-tile.
//
// Two small kernels follow: one merges the per-CTA lists of each keyframe and
// applies the keyframe's inverse norm (cos = <f, t> / |f| / |t|); one forms each
// query's union (a text scored by its best retrieving keyframe) and its top
// k_query.  A fourth, optional kernel computes the corpus inverse norms when the
// caller does not pass them (fvrag_embed_inv_norms is the same kernel on its own).
#include <cuda_fp16.h>

#include <algorithm>
#include <mutex>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {
namespace rt {

constexpr int kThreads = 192;
constexpr int kBK = 64;            // fp16 elements per 128-byte swizzled row
constexpr int kBM = 128;           // keyframes per M-tile (MMA M)
constexpr int kStages = 4;
constexpr int kMaxCtas = 256;
constexpr int kMaxMTiles = 16;     // keyframes <= 2048
constexpr int kMaxKf = 8;          // k_frame <= 8
constexpr int kMaxState = 4096;    // ceil(keyframes / 128) * 128 * k_frame <= 4096 (32 KB of lists)
constexpr int kMaxKq = 64;

enum : uint32_t { kSiteProdEmpty = 0x601, kSiteMmaTmem = 0x602, kSiteMmaFull = 0x603,
                  kSiteEpiFull = 0x604, kSiteDrain = 0x605 };

template <int BN, int MG>
struct Cfg {
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = MG * kABytes + kBBytes;
  static constexpr int kSlots = 2;
  static constexpr int kTmemCols = kSlots * MG * BN;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 256 + kMaxState * 8;
  static_assert(kTmemCols == 512, "tensor memory plan uses all 512 columns");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

// (s, i) ranks before (t, j): larger similarity first, smaller id first on ties.
__device__ __forceinline__ bool better(float s, int i, float t, int j) {
  return s > t || (s == t && (unsigned)i < (unsigned)j);  // id -1 ranks last among equals
}

// One keyframe row's pass over the ncols similarities of a text tile held in tensor
// memory at tbase (this thread's lane): scale by the texts' inverse norms (lane i of
// chunk c holds column 32 c + i in invr[c]) and insert those that beat the row's list
// (ss / si, best first; columns are text ids v0 + column).  The accumulator is read
// kLdGroup chunks of 32 columns per tensor-memory wait: a load waits behind the MMAs
// already queued on the SM's tensor core, so fewer, larger waits keep the epilogue off
// the critical path.
constexpr int kLdGroup = 1;

template <int BN>
__device__ __forceinline__ void row_chunk(const uint32_t (&r0)[32], int c, int ncols, int v0,
                                          bool live, int kf, const float (&invr)[BN / 32],
                                          float& thr, float* ss, int32_t* si) {
  uint32_t r[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) r[i] = r0[i];
  float invc = invr[0];
#pragma unroll
  for (int cc = 1; cc < BN / 32; ++cc)
    if (cc == c) invc = invr[cc];
  const int nvalid = min(32, ncols - c * 32);
  // fast filter: scaled similarities in place, bit i set when column i beats the list
  uint32_t hits = 0;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const float v = __uint_as_float(r[i]) * __shfl_sync(0xffffffffu, invc, i);
    r[i] = __float_as_uint(v);
    hits |= (v > thr ? 1u : 0u) << i;
  }
  if (!live) hits = 0;
  if (nvalid < 32) hits &= (1u << nvalid) - 1u;
  // more hits than the list holds (the lists fill on a CTA's first tiles): only the
  // chunk's kf best can enter it, so keep those (larger value, then lower column)
  if (__popc(hits) > kf) {
    uint32_t keepm = 0;
#pragma unroll 1
    for (int p = 0; p < kf; ++p) {
      float bv = -INFINITY;
      int bi = -1;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float v = __uint_as_float(r[i]);
        const bool cand = ((hits & ~keepm) >> i) & 1u;
        if (cand && (bi < 0 || v > bv)) {
          bv = v;
          bi = i;
        }
      }
      keepm |= 1u << bi;
    }
    hits = keepm;
  }
  // rare path: insert the hits in column order (ids ascend, so a strict >
  // against the list keeps the smaller id first among equal similarities)
  while (hits) {
    const int i = __ffs(hits) - 1;
    hits &= hits - 1u;
    float v = 0.f;
#pragma unroll
    for (int k = 0; k < 32; ++k)
      if (k == i) v = __uint_as_float(r[k]);
    if (!(v > thr)) continue;
    const int id = v0 + c * 32 + i;
    int p = kf - 1;
    while (p > 0 && better(v, id, ss[p - 1], si[p - 1])) {
      ss[p] = ss[p - 1];
      si[p] = si[p - 1];
      --p;
    }
    ss[p] = v;
    si[p] = id;
    thr = ss[kf - 1];
  }
}

template <int BN>
__device__ __forceinline__ void row_tile(uint32_t tbase, int ncols, int v0, bool live, int kf,
                                         const float (&invr)[BN / 32], float* ss, int32_t* si) {
  float thr = ss[kf - 1];
  const int nch = (ncols + 31) / 32;
#pragma unroll 1
  for (int c0 = 0; c0 < nch; c0 += kLdGroup) {
    uint32_t r[kLdGroup][32];
#pragma unroll
    for (int g = 0; g < kLdGroup; ++g)
      if (c0 + g < nch) tmem_ld_32x32b_x32(tbase + (c0 + g) * 32, r[g]);
    tmem_wait_ld();
#pragma unroll
    for (int g = 0; g < kLdGroup; ++g)
      if (c0 + g < nch) row_chunk<BN>(r[g], c0 + g, ncols, v0, live, kf, invr, thr, ss, si);
  }
}

template <int BN, int MG>
__global__ void __launch_bounds__(kThreads, 1)
    retrieve_kernel(const __grid_constant__ CUtensorMap tm_frames,
                    const __grid_constant__ CUtensorMap tm_t64,
                    const __grid_constant__ CUtensorMap tm_t16,
                    const float* __restrict__ text_inv_norm, int M, int E, int Nt, int kf,
                    int hrows, float* __restrict__ part_sim, int32_t* __restrict__ part_idx,
                    uint32_t* status, uint64_t limit_ns) {
  using C = Cfg<BN, MG>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + kStages * C::kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* tfull = bars + 2 * kStages;
  uint64_t* tempty = tfull + C::kSlots;
  uint64_t* drain = tempty + C::kSlots;
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* st_sim = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);
  int32_t* st_idx = reinterpret_cast<int32_t*>(st_sim + kMaxState);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int nunits = (Nt + 15) >> 4;
  const int u_lo = (int)(((long long)blockIdx.x * nunits) / gridDim.x);
  const int u_hi = (int)(((long long)(blockIdx.x + 1) * nunits) / gridDim.x);
  const int v_lo = u_lo * 16;
  const int v_hi = min(u_hi * 16, Nt);
  const int ntiles = (v_hi - v_lo + BN - 1) / BN;
  const int mtiles = (M + kBM - 1) / kBM;
  const int ngroups = (mtiles + MG - 1) / MG;
  const int nitems = ntiles * ngroups;
  const int kblocks = (E + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int s = 0; s < C::kSlots; ++s) {
      mbar_init(smem_u32(&tfull[s]), 1);
      mbar_init(smem_u32(&tempty[s]), 4);
    }
    mbar_init(smem_u32(drain), 1);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_frames);
    tma_prefetch_desc(&tm_t64);
    tma_prefetch_desc(&tm_t16);
  }
  for (int i = threadIdx.x; i < mtiles * kBM * kf; i += kThreads) {
    st_sim[i] = -INFINITY;
    st_idx[i] = -1;
  }
  if (hrows < kBM) {
    for (int i = threadIdx.x; i < kStages * MG * (kBM - hrows) * 8; i += kThreads) {
      const int chunk = i & 7, rr = (i >> 3) % (kBM - hrows) + hrows, tile = (i >> 3) / (kBM - hrows);
      uint4* dst = reinterpret_cast<uint4*>(ring + (tile / MG) * C::kStageBytes +
                                            (tile % MG) * C::kABytes + rr * 128 + chunk * 16);
      *dst = make_uint4(0u, 0u, 0u, 0u);
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  griddep_wait();

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_t = policy_evict_first();
      const uint64_t pol_f = policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int it = 0; it < nitems && ok; ++it) {
        const int t = it / ngroups, grp = it % ngroups;
        const int v0 = v_lo + t * BN;
        const int rows16 = (min(BN, v_hi - v0) + 15) & ~15;
        const int mcount = min(MG, mtiles - grp * MG);
        const uint32_t bytes = mcount * hrows * kBK * 2 + rows16 * kBK * 2;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteProdEmpty);
            ok = false;
            break;
          }
          const uint32_t fb = smem_u32(&full[stage]);
          mbar_arrive_expect_tx(fb, bytes);
          uint8_t* st = ring + stage * C::kStageBytes;
          for (int j = 0; j < mcount; ++j)
            tma_load_2d(smem_u32(st + j * C::kABytes), &tm_frames, fb, kb * kBK,
                        (grp * MG + j) * kBM, pol_f);
          uint8_t* bsm = st + MG * C::kABytes;
          int r = 0;
          for (; r + 64 <= rows16; r += 64)
            tma_load_2d(smem_u32(bsm + r * 128), &tm_t64, fb, kb * kBK, v0 + r, pol_t);
          for (; r < rows16; r += 16)
            tma_load_2d(smem_u32(bsm + r * 128), &tm_t16, fb, kb * kBK, v0 + r, pol_t);
          ++issued;
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      const int pend = issued < kStages ? (int)issued : kStages;
      for (int i = 0; i < pend; ++i) {
        if (--stage < 0) {
          stage = kStages - 1;
          phase ^= 1;
        }
        mbar_wait(smem_u32(&full[stage]), phase, limit_ns);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int it = 0; it < nitems && ok; ++it) {
        const int slot = it % C::kSlots;
        const uint32_t use = it / C::kSlots;
        const int t = it / ngroups, grp = it % ngroups;
        const int v0 = v_lo + t * BN;
        const int rows16 = (min(BN, v_hi - v0) + 15) & ~15;
        const int mcount = min(MG, mtiles - grp * MG);
        const uint32_t idesc = idesc_f16_f32(kBM, rows16);
        if (!mbar_wait(smem_u32(&tempty[slot]), (use & 1) ^ 1, limit_ns)) {
          record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaTmem);
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait(smem_u32(&full[stage]), phase, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaFull);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(ring + stage * C::kStageBytes);
          const uint32_t bsm = st + MG * C::kABytes;
          for (int j = 0; j < mcount; ++j) {
            const uint32_t d = tmem_base + (uint32_t)((slot * MG + j) * BN);
#pragma unroll
            for (int k16 = 0; k16 < kBK / 16; ++k16) {
              const uint64_t a = desc_kmajor_sw128(st + j * C::kABytes + k16 * 32);
              const uint64_t b = desc_kmajor_sw128(bsm + k16 * 32);
              tc_mma_bf16(d, a, b, idesc, (kb | k16) != 0);
            }
          }
          tc_commit(smem_u32(&empty[stage]));
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(&tfull[slot]));
      }
      tc_commit(smem_u32(drain));
      if (!mbar_wait(smem_u32(drain), 0, limit_ns))
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    for (int it = 0; it < nitems; ++it) {
      const int slot = it % C::kSlots;
      const uint32_t use = it / C::kSlots;
      const int t = it / ngroups, grp = it % ngroups;
      const int v0 = v_lo + t * BN;
      const int ncols = min(BN, v_hi - v0);
      const int mcount = min(MG, mtiles - grp * MG);
      // the tile's inverse text norms, lane i holding column 32 c + i of chunk c; loaded
      // before the accumulator wait so their latency hides behind the MMAs
      float invr[BN / 32];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        const int col = c * 32 + lane;
        invr[c] = col < ncols ? __ldg(text_inv_norm + v0 + col) : 0.f;
      }
      if (!mbar_wait(smem_u32(&tfull[slot]), use & 1, limit_ns)) {
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteEpiFull);
        break;
      }
      tc_fence_after();
      for (int j = 0; j < mcount; ++j) {
        const int mt = grp * MG + j;
        const bool live = mt * kBM + row < M;
        // this keyframe's running list, best first, in shared memory (row-private)
        const uint32_t tbase =
            tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((slot * MG + j) * BN);
        row_tile<BN>(tbase, ncols, v0, live, kf, invr, st_sim + (mt * kBM + row) * kf,
                     st_idx + (mt * kBM + row) * kf);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[slot]));
    }
    for (int mt = 0; mt < mtiles; ++mt) {
      const int m = mt * kBM + row;
      if (m < M)
        for (int p = 0; p < kf; ++p) {
          part_sim[((size_t)blockIdx.x * M + m) * kf + p] = st_sim[(mt * kBM + row) * kf + p];
          part_idx[((size_t)blockIdx.x * M + m) * kf + p] = st_idx[(mt * kBM + row) * kf + p];
        }
    }
  }
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, C::kTmemCols);
}

// ---------------------------------------------------------------------------
// Pair form for more than 128 keyframes: a cluster of two CTAs on two SMs runs
// tcgen05 cta_group::2 MMAs of M = 256 keyframes x N = 256 texts.  CTA r of the pair
// holds keyframes [128 r, 128 r + 128) of every 256-row pair-tile and texts
// [v0 + N/2 r, v0 + N/2 (r + 1)) of every text tile, keeps the top-k lists of its own
// keyframes, and receives their similarities against all N texts (rank 0's texts
// first, so column c is text v0 + c).  Each SM so loads half of every text tile and
// half of every pair-tile, per 256 texts; two accumulator sets of 256 columns per
// CTA let the epilogue of one item overlap the MMAs of the next.  Rank 0 issues the
// MMAs; both CTAs' copies complete on rank 0's barriers.
//
// A last pair-tile of at most 128 keyframes (320 keyframes = 256 + 64, say) runs as
// M = 128 MMAs instead, which take half the time of M = 256 ones: CTA r holds
// keyframes [64 r, 64 r + 64) of it, and its accumulator (N/2 columns) holds them
// twice over the 128 lanes: lane l < 64 keyframe l against rank 0's texts
// (v0 + [0, N/2)), lane 64 + l the same keyframe against rank 1's (v0 + N/2 + [0, N/2)).
// Each lane keeps its own list; the two lists of a keyframe are merged at the end.
struct PairCfg {
  static constexpr int BN = 256;
  static constexpr int kABytes = kBM * kBK * 2;             // this CTA's 128 keyframes
  static constexpr int kBBytes = (BN / 2) * kBK * 2;        // this CTA's 128 texts
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kStagesP = 6;
  static constexpr int kSlots = 2;
  static constexpr int kTmemCols = 512;
  static constexpr int kSmemBytes = kStagesP * kStageBytes + 1024 + 256 + kMaxState * 8;
  static_assert(kSlots * BN <= kTmemCols, "accumulators fit tensor memory");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

__global__ void __launch_bounds__(kThreads, 1)
    retrieve_pair_kernel(const __grid_constant__ CUtensorMap tm_frames,
                         const __grid_constant__ CUtensorMap tm_frames64,
                         const __grid_constant__ CUtensorMap tm_t64,
                         const __grid_constant__ CUtensorMap tm_t16,
                         const float* __restrict__ text_inv_norm, int M, int E, int Nt, int kf,
                         float* __restrict__ part_sim, int32_t* __restrict__ part_idx,
                         uint32_t* status, uint64_t limit_ns) {
  using C = PairCfg;
  constexpr int BN = C::BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStagesP * C::kStageBytes);
  uint64_t* full = bars;                        // rank 0: both CTAs' copies
  uint64_t* empty = bars + C::kStagesP;         // each CTA: its stage is free
  uint64_t* tfull = bars + 2 * C::kStagesP;     // each CTA: accumulators ready
  uint64_t* tempty = tfull + C::kSlots;         // rank 0: both epilogues done
  uint64_t* drain = tempty + C::kSlots;         // rank 0: every MMA done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* st_sim = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);
  int32_t* st_idx = reinterpret_cast<int32_t*>(st_sim + kMaxState);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

  // ---- this pair's text range, in units of 16 rows
  const int nunits = (Nt + 15) >> 4;
  const int u_lo = (int)(((long long)pair * nunits) / npairs);
  const int u_hi = (int)(((long long)(pair + 1) * nunits) / npairs);
  const int v_lo = u_lo * 16;
  const int v_hi = min(u_hi * 16, Nt);
  const int ntiles = (v_hi - v_lo + BN - 1) / BN;
  const int ptiles = (M + 2 * kBM - 1) / (2 * kBM);
  const bool tail = M - (ptiles - 1) * 2 * kBM <= kBM;   // last pair-tile: M = 128 MMAs
  const int nitems = ntiles * ptiles;
  const int kblocks = (E + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStagesP; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int s = 0; s < C::kSlots; ++s) {
      mbar_init(smem_u32(&tfull[s]), 1);
      mbar_init(smem_u32(&tempty[s]), 8);  // one arrival per epilogue warp of both CTAs
    }
    mbar_init(smem_u32(drain), 1);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_frames);
    tma_prefetch_desc(&tm_frames64);
    tma_prefetch_desc(&tm_t64);
    tma_prefetch_desc(&tm_t16);
  }
  for (int i = threadIdx.x; i < ptiles * kBM * kf; i += kThreads) {
    st_sim[i] = -INFINITY;
    st_idx[i] = -1;
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_holder), C::kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // the peer's barriers are initialised before any remote use
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const uint32_t full0 = mapa_shared(smem_u32(&full[0]), 0);      // rank 0's barriers
  const uint32_t tempty0 = mapa_shared(smem_u32(&tempty[0]), 0);
  griddep_wait();                 // inputs may come from the previous kernel

  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      const uint64_t pol_t = policy_evict_first();
      const uint64_t pol_f = policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int it = 0; it < nitems && ok; ++it) {
        const int t = it / ptiles, pt = it % ptiles;
        const bool tail_item = tail && pt == ptiles - 1;
        const int v0 = v_lo + t * BN;
        const int n = min(BN, (v_hi - v0 + 31) & ~31);     // MMA N, a multiple of 32
        const int half = n >> 1;
        const int arows = tail_item ? kBM / 2 : kBM;       // this CTA's keyframe rows
        const uint32_t bytes = (arows + half) * kBK * 2;   // per CTA
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&empty[stage]), phase ^ 1, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteProdEmpty);
            ok = false;
            break;
          }
          const uint32_t fb = full0 + (uint32_t)(stage * 8);
          if (rank == 0) mbar_arrive_expect_tx(smem_u32(&full[stage]), 2 * bytes);
          uint8_t* st = ring + stage * C::kStageBytes;
          tma_load_2d_pair(smem_u32(st), tail_item ? &tm_frames64 : &tm_frames, fb, kb * kBK,
                           pt * 2 * kBM + (int)rank * arows, pol_f);
          uint8_t* bsm = st + C::kABytes;
          const int w0 = v0 + (int)rank * half;
          int r = 0;
          for (; r + 64 <= half; r += 64)
            tma_load_2d_pair(smem_u32(bsm + r * 128), &tm_t64, fb, kb * kBK, w0 + r, pol_t);
          for (; r < half; r += 16)
            tma_load_2d_pair(smem_u32(bsm + r * 128), &tm_t16, fb, kb * kBK, w0 + r, pol_t);
          ++issued;
          if (++stage == C::kStagesP) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // rank 0 sees both CTAs' copies complete on its barriers: leave none in flight
      if (rank == 0) {
        const int pend = issued < C::kStagesP ? (int)issued : C::kStagesP;
        for (int i = 0; i < pend; ++i) {
          if (--stage < 0) {
            stage = C::kStagesP - 1;
            phase ^= 1;
          }
          mbar_wait(smem_u32(&full[stage]), phase, limit_ns);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (rank 0)
    if (lane == 0 && rank == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int it = 0; it < nitems && ok; ++it) {
        const int slot = it % C::kSlots;
        const uint32_t use = it / C::kSlots;
        const int t = it / ptiles, pt = it % ptiles;
        const int v0 = v_lo + t * BN;
        const int n = min(BN, (v_hi - v0 + 31) & ~31);
        const uint32_t idesc = idesc_f16_f32((tail && pt == ptiles - 1) ? kBM : 2 * kBM, n);
        if (!mbar_wait_cluster(smem_u32(&tempty[slot]), (use & 1) ^ 1, limit_ns)) {
          record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaTmem);
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&full[stage]), phase, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaFull);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(ring + stage * C::kStageBytes);
          const uint32_t bsm = st + C::kABytes;
          const uint32_t d = tmem_base + (uint32_t)(slot * BN);
#pragma unroll
          for (int k16 = 0; k16 < kBK / 16; ++k16)
            tc_mma_bf16_pair(d, desc_kmajor_sw128(st + k16 * 32), desc_kmajor_sw128(bsm + k16 * 32),
                             idesc, (kb | k16) != 0);
          tc_commit_pair(smem_u32(&empty[stage]), 0x3);
          if (++stage == C::kStagesP) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit_pair(smem_u32(&tfull[slot]), 0x3);
      }
      // every MMA issued by this thread has finished before tensor memory is freed
      tc_commit_pair(smem_u32(drain), 0x1);
      if (!mbar_wait(smem_u32(drain), 0, limit_ns)) record_error(status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;      // this CTA's keyframe inside a pair-tile
    for (int it = 0; it < nitems; ++it) {
      const int slot = it % C::kSlots;
      const uint32_t use = it / C::kSlots;
      const int t = it / ptiles, pt = it % ptiles;
      const bool tail_item = tail && pt == ptiles - 1;
      const int v0 = v_lo + t * BN;
      const int ncols = min(BN, v_hi - v0);
      // this lane's texts: all N columns, or in the M = 128 form half of them
      const int half = min(BN, (v_hi - v0 + 31) & ~31) >> 1;
      const int cbase = tail_item && row >= kBM / 2 ? half : 0;
      const int nc = tail_item ? max(0, min(half, ncols - cbase)) : ncols;
      // the tile's inverse text norms, loaded before the accumulator wait
      float invr[BN / 32];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        const int col = c * 32 + lane;
        invr[c] = col < nc ? __ldg(text_inv_norm + v0 + cbase + col) : 0.f;
      }
      if (!mbar_wait_cluster(smem_u32(&tfull[slot]), use & 1, limit_ns)) {
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteEpiFull);
        break;
      }
      tc_fence_after();
      const int m = tail_item ? pt * 2 * kBM + (int)rank * (kBM / 2) + (row & (kBM / 2 - 1))
                              : pt * 2 * kBM + (int)rank * kBM + row;
      const uint32_t tbase =
          tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(slot * BN);
      row_tile<BN>(tbase, nc, v0 + cbase, m < M, kf, invr, st_sim + (pt * kBM + row) * kf,
                   st_idx + (pt * kBM + row) * kf);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty0 + (uint32_t)(slot * 8));
    }
    // publish this CTA's keyframes' lists (one partial per pair)
    for (int pt = 0; pt < ptiles; ++pt) {
      if (tail && pt == ptiles - 1) {
        // M = 128 form: lanes l and 64 + l hold keyframe l's lists over the two halves
        // of every text tile (disjoint texts); merge them, best first
        asm volatile("bar.sync 1, 128;" ::: "memory");   // the 4 epilogue warps
        const int m = pt * 2 * kBM + (int)rank * (kBM / 2) + row;
        if (row < kBM / 2 && m < M) {
          const float* as = st_sim + (pt * kBM + row) * kf;
          const int32_t* ai = st_idx + (pt * kBM + row) * kf;
          const float* bs = st_sim + (pt * kBM + row + kBM / 2) * kf;
          const int32_t* bi = st_idx + (pt * kBM + row + kBM / 2) * kf;
          int ia = 0, ib = 0;   // ia + ib = p < kf: neither runs past its list
          for (int p = 0; p < kf; ++p) {
            const bool from_a = better(as[ia], ai[ia], bs[ib], bi[ib]);
            part_sim[((size_t)pair * M + m) * kf + p] = from_a ? as[ia] : bs[ib];
            part_idx[((size_t)pair * M + m) * kf + p] = from_a ? ai[ia] : bi[ib];
            if (from_a) ++ia; else ++ib;
          }
        }
        continue;
      }
      const int m = pt * 2 * kBM + (int)rank * kBM + row;
      if (m < M)
        for (int p = 0; p < kf; ++p) {
          part_sim[((size_t)pair * M + m) * kf + p] = st_sim[(pt * kBM + row) * kf + p];
          part_idx[((size_t)pair * M + m) * kf + p] = st_idx[(pt * kBM + row) * kf + p];
        }
    }
  }
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // neither CTA frees tensor memory the other may still use
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, C::kTmemCols);
}

// inv_norm[r] = 1 / |x_r| (0 for a zero row); one warp per row, 16-byte loads.
__global__ void inv_norm_kernel(const __half* __restrict__ x, int rows, int E,
                                float* __restrict__ inv_norm) {
  griddep_wait();
  const int lane = threadIdx.x & 31;
  const int nw = gridDim.x * (blockDim.x >> 5);
  for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += nw) {
    const uint4* p = reinterpret_cast<const uint4*>(x + (size_t)r * E);
    float s = 0.f;
    for (int c = lane; c < E / 8; c += 32) {
      const uint4 u = __ldcs(p + c);
      const __half2* h = reinterpret_cast<const __half2*>(&u);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float2 f = __half22float2(h[k]);
        s = fmaf(f.x, f.x, s);
        s = fmaf(f.y, f.y, s);
      }
    }
    s = warp_sum(s);
    if (lane == 0) inv_norm[r] = s > 0.f ? rsqrtf(s) : 0.f;
  }
  griddep_launch_dependents();
}

// Per keyframe: merge the per-CTA lists (each sorted, ids unique across CTAs)
// into the keyframe's top k_frame and scale by the keyframe's inverse norm.
// One warp per keyframe.
__global__ void frame_merge_kernel(const float* __restrict__ part_sim,
                                   const int32_t* __restrict__ part_idx,
                                   const __half* __restrict__ frames, int M, int E, int kf,
                                   int nparts, int32_t* __restrict__ out_idx,
                                   float* __restrict__ out_sim) {
  griddep_wait();
  griddep_launch_dependents();
  const int m = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= M) return;
  const uint4* p = reinterpret_cast<const uint4*>(frames + (size_t)m * E);
  float s = 0.f;
  for (int c = lane; c < E / 8; c += 32) {
    const uint4 u = p[c];
    const __half2* h = reinterpret_cast<const __half2*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 f = __half22float2(h[k]);
      s = fmaf(f.x, f.x, s);
      s = fmaf(f.y, f.y, s);
    }
  }
  s = warp_sum(s);
  const float inv = s > 0.f ? rsqrtf(s) : 0.f;
  const int n = nparts * kf;          // entries of this keyframe: n <= 256 * 8
  uint64_t taken = 0;                 // bit j: entry lane + 32 j already chosen
  for (int r = 0; r < kf; ++r) {
    float bs = -INFINITY;
    int bi = -1, bpos = -1;
    for (int j = 0, e = lane; e < n; ++j, e += 32) {
      if ((taken >> j) & 1ull) continue;
      const int b = e / kf, pidx = e % kf;
      const size_t a = ((size_t)b * M + m) * kf + pidx;
      const int id = part_idx[a];
      if (id < 0) continue;
      const float v = part_sim[a];
      if (bi < 0 || better(v, id, bs, bi)) {
        bs = v;
        bi = id;
        bpos = e;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float os = __shfl_xor_sync(0xffffffffu, bs, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      const int op = __shfl_xor_sync(0xffffffffu, bpos, o);
      if (oi >= 0 && (bi < 0 || better(os, oi, bs, bi))) {
        bs = os;
        bi = oi;
        bpos = op;
      }
    }
    if (bpos >= 0 && (bpos & 31) == lane) taken |= 1ull << (bpos >> 5);
    if (lane == 0) {
      out_idx[(size_t)m * kf + r] = bi;
      out_sim[(size_t)m * kf + r] = bi >= 0 ? bs * inv : -INFINITY;
    }
  }
}

// Per query: T = the texts its keyframes retrieved, each scored by its best
// retrieving keyframe; out = the k_query best of T.  One warp per query; a text
// chosen in one round marks all its entries dead.
__global__ void query_merge_kernel(const int32_t* __restrict__ fidx, const float* __restrict__ fsim,
                                   const int32_t* __restrict__ frame_offsets, int Qn, int M, int kf,
                                   int Kq, int32_t* __restrict__ out_idx,
                                   float* __restrict__ out_sim) {
  __shared__ uint8_t dead[kMaxState];
  griddep_wait();
  griddep_launch_dependents();
  const int q = blockIdx.x;
  const int lane = threadIdx.x;
  if (q >= Qn) return;
  const int f0 = frame_offsets[q], f1 = frame_offsets[q + 1];
  // offsets outside [0, M] or decreasing (a caller error) read as an empty query
  const bool sane = f0 >= 0 && f1 >= f0 && f1 <= M;
  const int e0 = sane ? f0 * kf : 0;
  const int n = sane ? (f1 - f0) * kf : 0;
  for (int e = lane; e < n; e += 32) dead[e] = fidx[e0 + e] < 0;
  __syncwarp();
  for (int r = 0; r < Kq; ++r) {
    float bs = -INFINITY;
    int bi = -1;
    for (int e = lane; e < n; e += 32) {
      if (dead[e]) continue;
      const float v = fsim[e0 + e];
      const int id = fidx[e0 + e];
      if (bi < 0 || better(v, id, bs, bi)) {
        bs = v;
        bi = id;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float os = __shfl_xor_sync(0xffffffffu, bs, o);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
      if (oi >= 0 && (bi < 0 || better(os, oi, bs, bi))) {
        bs = os;
        bi = oi;
      }
    }
    if (lane == 0) {
      out_idx[(size_t)q * Kq + r] = bi;
      out_sim[(size_t)q * Kq + r] = bi >= 0 ? bs : -INFINITY;
    }
    if (bi >= 0)
      for (int e = lane; e < n; e += 32)
        if (fidx[e0 + e] == bi) dead[e] = 1;
    __syncwarp();
  }
}

struct Plan {
  int ctas, bn, mg;   // mg = 0: the pair form (ctas = pairs, the merge's partial lists)
};

// Pairs (2-CTA clusters) of the pair form that can be resident at once, per device.
static int max_pairs() {
  static std::mutex mu;
  static int cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev] == 0) {
    int n = 0;
    if (cudaFuncSetAttribute(retrieve_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             PairCfg::kSmemBytes) == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      const int sms = std::max(2, sm_count());
      cfg.gridDim = dim3(sms / 2 * 2);
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = PairCfg::kSmemBytes;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&n, retrieve_pair_kernel, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    cached[dev] = std::max(1, std::min(n, std::min(sm_count() / 2, kMaxCtas)));
  }
  return cached[dev];
}

static Plan make_plan(const fvrag_retrieve_desc* d, int sms) {
  Plan p;
  const int mtiles = (d->num_keyframes + kBM - 1) / kBM;
  // one M-tile: <256, 1>, two accumulator sets; more keyframes: the pair form
  p.bn = 256;
  p.mg = mtiles <= 1 ? 1 : 0;
  const int nunits = (d->num_texts + 15) / 16;
  p.ctas = std::max(1, std::min(std::min(sms > 0 ? sms : 148, kMaxCtas), nunits));
  if (p.mg == 0) p.ctas = std::max(1, std::min(max_pairs(), nunits));
  return p;
}

struct WsLayout {
  size_t part_sim, part_idx, frame_idx, frame_sim, inv_norm, total;
};

static WsLayout ws_layout(const fvrag_retrieve_desc* d) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  const size_t lists = (size_t)kMaxCtas * d->num_keyframes * d->k_frame;
  const size_t fl = (size_t)d->num_keyframes * d->k_frame;
  WsLayout w;
  w.part_sim = kWsHeaderBytes;
  w.part_idx = w.part_sim + up(lists * 4);
  w.frame_idx = w.part_idx + up(lists * 4);
  w.frame_sim = w.frame_idx + up(fl * 4);
  w.inv_norm = w.frame_sim + up(fl * 4);
  w.total = w.inv_norm + up((size_t)d->num_texts * 4);
  return w;
}

static bool desc_ok(const fvrag_retrieve_desc* d) {
  return d && d->num_queries >= 1 && d->num_keyframes >= 0 && d->num_texts >= 1 && d->dim >= 8 &&
         d->k_frame >= 1 && d->k_query >= 1 && d->flags == 0;
}

template <int BN, int MG>
static fvrag_status launch(const Plan& p, const CUtensorMap& tf, const CUtensorMap& t64,
                           const CUtensorMap& t16, const float* inv_norm,
                           const fvrag_retrieve_desc* d, int hrows, float* psim, int32_t* pidx,
                           uint32_t* status, cudaStream_t s) {
  using C = Cfg<BN, MG>;
  auto kern = retrieve_kernel<BN, MG>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  if (launch_pdl(kern, dim3(p.ctas), dim3(kThreads), (size_t)C::kSmemBytes, s, tf, t64, t16,
                 inv_norm, d->num_keyframes, d->dim, d->num_texts, d->k_frame, hrows, psim, pidx,
                 status, wait_limit_ns()) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

static fvrag_status launch_pair(const Plan& p, const CUtensorMap& tf, const CUtensorMap& tf64,
                                const CUtensorMap& t64,
                                const CUtensorMap& t16, const float* inv_norm,
                                const fvrag_retrieve_desc* d, float* psim, int32_t* pidx,
                                uint32_t* status, cudaStream_t s) {
  if (cudaFuncSetAttribute(retrieve_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           PairCfg::kSmemBytes) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * p.ctas);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = PairCfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (counted(cudaLaunchKernelEx(&cfg, retrieve_pair_kernel, tf, tf64, t64, t16, inv_norm,
                                 d->num_keyframes, d->dim, d->num_texts, d->k_frame, psim, pidx,
                                 status, wait_limit_ns())) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

static fvrag_status launch_inv_norms(const void* x, int rows, int dim, float* inv, cudaStream_t s) {
  const int sms = sm_count() > 0 ? sm_count() : 148;
  const int blocks = std::max(1, std::min((rows + 7) / 8, sms * 8));
  if (launch_pdl(inv_norm_kernel, dim3(blocks), dim3(256), 0, s, (const __half*)x, rows, dim, inv) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

}  // namespace rt
}  // namespace fvrag

using namespace fvrag;

extern "C" fvrag_status fvrag_embed_inv_norms(const void* x, int32_t rows, int32_t dim,
                                              float* inv_norm, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_embed_inv_norms");
  if (!x || !inv_norm || rows < 1 || dim < 8) return FVRAG_ERR_INVALID_ARG;
  if (dim % 8 != 0 || !aligned16(x)) return FVRAG_ERR_MISALIGNED;
  return rt::launch_inv_norms(x, rows, dim, inv_norm, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" size_t fvrag_retrieve_workspace(const fvrag_retrieve_desc* d) {
  if (!rt::desc_ok(d)) return 0;
  return rt::ws_layout(d).total;
}

extern "C" fvrag_status fvrag_retrieve(const fvrag_retrieve_desc* d, const void* frame_emb,
                                       const int32_t* frame_offsets, const void* text_emb,
                                       const float* text_inv_norm, int32_t* frame_topk,
                                       float* frame_topk_sim, int32_t* out_idx, float* out_sim,
                                       void* ws, size_t ws_size, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_retrieve");
  using namespace rt;
  if (!desc_ok(d) || !frame_offsets || !text_emb || !out_idx || !out_sim)
    return FVRAG_ERR_INVALID_ARG;
  if (d->num_keyframes > 0 && !frame_emb) return FVRAG_ERR_INVALID_ARG;
  if (d->num_keyframes > kMaxMTiles * kBM || d->k_frame > kMaxKf ||
      (long long)((d->num_keyframes + kBM - 1) / kBM) * kBM * d->k_frame > kMaxState ||
      d->k_query > kMaxKq)
    return FVRAG_ERR_UNSUPPORTED;
  if (d->dim % 8 != 0) return FVRAG_ERR_MISALIGNED;
  if ((frame_emb && !aligned16(frame_emb)) || !aligned16(text_emb) ||
      (text_inv_norm && !aligned16(text_inv_norm)))
    return FVRAG_ERR_MISALIGNED;
  const WsLayout w = ws_layout(d);
  if (!ws || ws_size < w.total) return FVRAG_ERR_WORKSPACE;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;

  uint8_t* base = reinterpret_cast<uint8_t*>(ws);
  uint32_t* status = reinterpret_cast<uint32_t*>(base);
  float* psim = reinterpret_cast<float*>(base + w.part_sim);
  int32_t* pidx = reinterpret_cast<int32_t*>(base + w.part_idx);
  int32_t* fidx = frame_topk ? frame_topk : reinterpret_cast<int32_t*>(base + w.frame_idx);
  float* fsim = frame_topk_sim ? frame_topk_sim : reinterpret_cast<float*>(base + w.frame_sim);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int M = d->num_keyframes;

  if (M > 0) {
    const float* inv = text_inv_norm;
    if (!inv) {
      float* tmp = reinterpret_cast<float*>(base + w.inv_norm);
      const fvrag_status st = launch_inv_norms(text_emb, d->num_texts, d->dim, tmp, s);
      if (st != FVRAG_OK) return st;
      inv = tmp;
    }
    const Plan p = make_plan(d, sm_count());
    const uint64_t E = (uint64_t)d->dim, Nt = (uint64_t)d->num_texts;
    const int hrows = M <= kBM ? (M + 15) / 16 * 16 : kBM;
    CUtensorMap tf, tf64, t64, t16;
    {
      const uint64_t dims[2] = {E, (uint64_t)M}, strides[1] = {E * 2};
      const uint32_t box[2] = {(uint32_t)kBK, (uint32_t)hrows}, box64[2] = {(uint32_t)kBK, 64u};
      if (!encode_tmap_f16(&tf, frame_emb, 2, dims, strides, box, true)) return FVRAG_ERR_CUDA;
      if (p.mg == 0 && !encode_tmap_f16(&tf64, frame_emb, 2, dims, strides, box64, true))
        return FVRAG_ERR_CUDA;
    }
    {
      const uint64_t dims[2] = {E, Nt}, strides[1] = {E * 2};
      const uint32_t b64[2] = {(uint32_t)kBK, 64u}, b16[2] = {(uint32_t)kBK, 16u};
      if (!encode_tmap_f16(&t64, text_emb, 2, dims, strides, b64, true)) return FVRAG_ERR_CUDA;
      if (!encode_tmap_f16(&t16, text_emb, 2, dims, strides, b16, true)) return FVRAG_ERR_CUDA;
    }
    fvrag_status st;
    if (p.mg == 1)
      st = launch<256, 1>(p, tf, t64, t16, inv, d, hrows, psim, pidx, status, s);
    else
      st = launch_pair(p, tf, tf64, t64, t16, inv, d, psim, pidx, status, s);
    if (st != FVRAG_OK) return st;
    if (launch_pdl(frame_merge_kernel, dim3((M + 7) / 8), dim3(256), 0, s, (const float*)psim,
                   (const int32_t*)pidx, (const __half*)frame_emb, M, d->dim, d->k_frame, p.ctas,
                   fidx, fsim) != cudaSuccess)
      return FVRAG_ERR_CUDA;
  }
  if (launch_pdl(query_merge_kernel, dim3(d->num_queries), dim3(32), 0, s, (const int32_t*)fidx,
                 (const float*)fsim, frame_offsets, d->num_queries, M, d->k_frame, d->k_query,
                 out_idx, out_sim) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}
