// K2: verifier LM-head log-probabilities (Eq. 11; the verifier likelihood of
// Section 4.6) as one tcgen05 GEMM with a fused online log-sum-exp and target
// gather, so the [rows x vocab] logits never leave the SM.
//
// Shape of the work: z = hidden[M x H] * W[V x H]^T with M (candidate tokens)
// small (32 .. ~1300) and V x H large (152064 x 3584 bf16 = 1.09 GB).  W is read
// from HBM exactly once; hidden (<= a few MB) stays in L2 and is re-read by
// every CTA.
//
// Persistent grid, one CTA per SM.  CTA b owns a contiguous vocabulary range
// (multiples of 16 rows, balanced to within 16 rows) and walks it in tiles of
// BN rows.  Per tile it accumulates, for a group of MG M-tiles of 128 hidden rows,
// D[128 x BN] = hidden_tile * W_tile^T in tensor memory (fp32), K-loop over H
// in blocks of 64 (one 128-byte swizzled row per operand row).
//
// Warp roles (192 threads):
//   warp 0     TMA producer: hidden tiles (box 64 x 128) and W tiles (boxes of
//              64 x 64 rows, 64 x 16 rows for the remainder) into a STAGES-deep
//              shared-memory ring, completion via mbarrier transaction counts.
//   warp 1     allocates tensor memory; one lane issues tcgen05.mma
//              (M = 128, N = tile rows, K = 16) and tcgen05.commit.
//   warps 2-5  epilogue: tcgen05.ld of 32 columns at a time (one hidden row per
//              thread), online max / sum of exp over the CTA's vocabulary slice,
//              and the gather of target logits that fall in the slice.
// Forms by row count M:
//   M <= 128        <256, 1>: one M-tile, two accumulator sets, so the epilogue of
//                   tile t overlaps the MMAs of tile t+1 (HBM-bound: W streams once);
//   129 .. 256      the pair form with one 256-row pair-tile (two accumulator sets);
//   257 .. 384      the vocabulary-major pair form: W rows along the MMA's M axis, the
//                   hidden rows along N (no padding of 320 rows to 384);
//   385 .. 2048     the pair form with two pair-tiles (512 rows) per pass over W.
// The pair form (lm_head_pair_kernel) runs on clusters of two CTAs with tcgen05
// cta_group::2 MMAs of M = 256, each SM loading half of every W tile.
//
// A second small kernel merges the per-CTA (max, sum) partials of every row into
// lse and writes logprob = z_target - lse (NaN for ids outside [0, V)).
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {
namespace lm {

constexpr int kThreads = 192;
constexpr int kBK = 64;            // bf16 elements per 128-byte swizzled row
constexpr int kBM = 128;           // hidden rows per M-tile (MMA M)
constexpr int kMaxCtas = 256;      // workspace is sized for this many partials
constexpr int kMaxMTiles = 16;     // rows <= 2048
constexpr int kMaxGathers = 8;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// wait-site ids recorded in the workspace header on a timeout
enum : uint32_t { kSiteProdEmpty = 0x201, kSiteMmaTmem = 0x202, kSiteMmaFull = 0x203,
                  kSiteEpiFull = 0x204, kSiteDrain = 0x205 };

// BN vocabulary rows per tile and MG M-tiles per pass; the accumulators of one item take
// MG * BN tensor-memory columns.  The one form built, <256, 1> (one M-tile), double-buffers
// them; more rows take the pair forms below.
template <int BN, int MG>
struct Cfg {
  static constexpr int kABytes = kBM * kBK * 2;           // 16 KB per M-tile
  static constexpr int kBBytes = BN * kBK * 2;            // BN rows x 128 B
  static constexpr int kStageBytes = MG * kABytes + kBBytes;
  static constexpr int kSlots = 512 / (MG * BN);
  static constexpr int kStages = MG * BN > 256 ? 3 : 4;  // ring depth within shared memory
  static constexpr int kTmemCols = 512;                   // allocation: a power of two
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 /*align*/ + 256 /*barriers*/ +
                                    2 * kMaxMTiles * kBM * 4 /*row state*/;
  static_assert(kSlots >= 1 && kSlots * MG * BN <= kTmemCols, "accumulators fit tensor memory");
  static_assert(BN % 32 == 0 && BN <= 256, "epilogue reads 32-column chunks; MMA N <= 256");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Online (max, sum of exp2) update of one row's state with a 32-column chunk of logits
// (natural units in r).  FULL: all 32 columns are valid (no per-element tests).  The max
// is a tree and the sum four interleaved partial sums, so neither is one long dependency
// chain.
template <bool FULL>
__device__ __forceinline__ void lse_chunk(const uint32_t (&r)[32], int nvalid, float& rmax,
                                          float& rsum) {
  float mx[8];
#pragma unroll
  for (int u = 0; u < 8; ++u) mx[u] = -INFINITY;
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (FULL || i < nvalid) mx[i & 7] = fmaxf(mx[i & 7], __uint_as_float(r[i]));
  const float cmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                           fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7]))) * kLog2e;
  const float nmax = fmaxf(rmax, cmax);
  float sp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (FULL || i < nvalid) sp[i & 3] += ex2(fmaf(__uint_as_float(r[i]), kLog2e, -nmax));
  rsum = rsum * ex2(rmax - nmax) + ((sp[0] + sp[1]) + (sp[2] + sp[3]));
  rmax = nmax;
}

// The epilogue of one row over `ncols` accumulator columns at tensor-memory address tbase
// (this warp's lane quarter), whose column c is vocabulary id v0 + c: folds them into the
// row's (rmax, rsum) and writes the logits of the row's targets found among them.
__device__ __forceinline__ void lse_row(uint32_t tbase, int ncols, int v0, bool live, int m,
                                        int G, const int32_t* __restrict__ targets,
                                        float* __restrict__ tgt_logit, float& rmax, float& rsum) {
  int tg[kMaxGathers];
#pragma unroll
  for (int g = 0; g < kMaxGathers; ++g)
    tg[g] = (live && g < G) ? __ldg(&targets[(size_t)m * G + g]) - v0 : -1;
  for (int c0 = 0; c0 < ncols; c0 += 32) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tbase + c0, r);
    tmem_wait_ld();
    const int nvalid = min(32, ncols - c0);
    if (nvalid == 32)
      lse_chunk<true>(r, 32, rmax, rsum);
    else
      lse_chunk<false>(r, nvalid, rmax, rsum);
#pragma unroll
    for (int g = 0; g < kMaxGathers; ++g) {
      const int c = tg[g] - c0;
      if (c >= 0 && c < nvalid) {
        float val = 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (i == c) val = __uint_as_float(r[i]);
        tgt_logit[(size_t)m * G + g] = val;
      }
    }
  }
}

template <int BN, int MG>
__global__ void __launch_bounds__(kThreads, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap tm_hidden,
                   const __grid_constant__ CUtensorMap tm_w64,
                   const __grid_constant__ CUtensorMap tm_w16, const int32_t* __restrict__ targets,
                   int M, int H, int V, int G, int hrows, float* __restrict__ part_max,
                   float* __restrict__ part_sum, float* __restrict__ tgt_logit, uint32_t* status,
                   uint64_t limit_ns) {
  using C = Cfg<BN, MG>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStageBytes);
  uint64_t* full = bars;                    // [C::kStages]
  uint64_t* empty = bars + C::kStages;         // [C::kStages]
  uint64_t* tfull = bars + 2 * C::kStages;     // [kSlots]
  uint64_t* tempty = tfull + C::kSlots;     // [kSlots]
  uint64_t* drain = tempty + C::kSlots;     // [1]
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* st_max = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);
  float* st_sum = st_max + kMaxMTiles * kBM;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // ---- this CTA's vocabulary range, in units of 16 rows
  const int nunits = (V + 15) >> 4;
  const int u_lo = (int)(((long long)blockIdx.x * nunits) / gridDim.x);
  const int u_hi = (int)(((long long)(blockIdx.x + 1) * nunits) / gridDim.x);
  const int v_lo = u_lo * 16;
  const int v_hi = min(u_hi * 16, V);
  const int ntiles = (v_hi - v_lo + BN - 1) / BN;
  const int mtiles = (M + kBM - 1) / kBM;
  const int ngroups = (mtiles + MG - 1) / MG;
  const int nitems = ntiles * ngroups;
  const int kblocks = (H + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    for (int s = 0; s < C::kSlots; ++s) {
      mbar_init(smem_u32(&tfull[s]), 1);
      mbar_init(smem_u32(&tempty[s]), 4);  // one arrival per epilogue warp
    }
    mbar_init(smem_u32(drain), 1);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_hidden);
    tma_prefetch_desc(&tm_w64);
    tma_prefetch_desc(&tm_w16);
  }
  for (int i = threadIdx.x; i < mtiles * kBM; i += kThreads) {
    st_max[i] = -INFINITY;
    st_sum[i] = 0.f;
  }
  if (hrows < kBM) {
    // A-tile rows the hidden box never fills: zero them once so the (discarded)
    // accumulator rows they produce stay finite
    for (int i = threadIdx.x; i < C::kStages * MG * (kBM - hrows) * 8; i += kThreads) {
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
  griddep_wait();                 // the prologue above touched no global memory

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
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
            tma_load_2d(smem_u32(st + j * C::kABytes), &tm_hidden, fb, kb * kBK,
                        (grp * MG + j) * kBM, pol_h);
          uint8_t* bsm = st + MG * C::kABytes;
          int r = 0;
          for (; r + 64 <= rows16; r += 64)
            tma_load_2d(smem_u32(bsm + r * 128), &tm_w64, fb, kb * kBK, v0 + r, pol_w);
          for (; r < rows16; r += 16)
            tma_load_2d(smem_u32(bsm + r * 128), &tm_w16, fb, kb * kBK, v0 + r, pol_w);
          ++issued;
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // leave no copy in flight: wait for the last (up to C::kStages) loads issued
      const int pend = issued < C::kStages ? (int)issued : C::kStages;
      for (int i = 0; i < pend; ++i) {
        if (--stage < 0) {
          stage = C::kStages - 1;
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
        const uint32_t idesc = idesc_bf16_f32(kBM, rows16);
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
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit(smem_u32(&tfull[slot]));
      }
      // every MMA issued by this thread has finished before tensor memory is freed
      tc_commit(smem_u32(drain));
      if (!mbar_wait(smem_u32(drain), 0, limit_ns))
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3;             // tensor-memory lanes this warp may access
    const int row = quarter * 32 + lane;      // row inside an M-tile
    for (int it = 0; it < nitems; ++it) {
      const int slot = it % C::kSlots;
      const uint32_t use = it / C::kSlots;
      const int t = it / ngroups, grp = it % ngroups;
      const int v0 = v_lo + t * BN;
      const int ncols = min(BN, v_hi - v0);
      const int mcount = min(MG, mtiles - grp * MG);
      if (!mbar_wait(smem_u32(&tfull[slot]), use & 1, limit_ns)) {
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteEpiFull);
        break;
      }
      tc_fence_after();
      for (int j = 0; j < mcount; ++j) {
        const int mt = grp * MG + j;
        const int m = mt * kBM + row;
        float rmax = st_max[mt * kBM + row];  // running max of z * log2(e)
        float rsum = st_sum[mt * kBM + row];
        const uint32_t tbase =
            tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((slot * MG + j) * BN);
        lse_row(tbase, ncols, v0, m < M, m, G, targets, tgt_logit, rmax, rsum);
        st_max[mt * kBM + row] = rmax;
        st_sum[mt * kBM + row] = rsum;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&tempty[slot]));
    }
    // publish this CTA's partials (row state in the log2 domain)
    for (int mt = 0; mt < mtiles; ++mt) {
      const int m = mt * kBM + row;
      if (m < M) {
        part_max[(size_t)blockIdx.x * M + m] = st_max[mt * kBM + row];
        part_sum[(size_t)blockIdx.x * M + m] = st_sum[mt * kBM + row];
      }
    }
  }
  griddep_launch_dependents();    // the merge kernel may start launching
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, C::kTmemCols);
}

// ---------------------------------------------------------------------------
// Pair form for many rows (more than three M-tiles).  A cluster of two CTAs on two SMs
// runs the GEMM with tcgen05 cta_group::2 MMAs of M = 256: CTA r of the pair holds hidden
// rows [128 r, 128 r + 128) of every 256-row pair-tile and W rows [v0 + N/2 r, v0 + N/2 (r + 1))
// of every N-row vocabulary tile, and its tensor memory receives the accumulators of its
// own 128 rows against all N columns (rank 0's W rows first).  Each SM thus loads half of
// every W tile, and one pass over W serves PG pair-tiles (PG = 2: 512 rows).  Rank 0
// issues the MMAs; both CTAs load (their copies complete on rank 0's barriers), and both
// run the epilogue over their own rows.  The pair owns one contiguous vocabulary range
// and writes one partial per row.
template <int PG>
struct PairCfg {
  static constexpr int BN = 256;                           // vocabulary rows per tile (MMA N)
  static constexpr int kABytes = kBM * kBK * 2;            // this CTA's 128 rows of a pair-tile
  static constexpr int kBBytes = (BN / 2) * kBK * 2;       // this CTA's half of a W tile
  static constexpr int kStageBytes = PG * kABytes + kBBytes;
  static constexpr int kSlots = 512 / (PG * BN);
  static constexpr int kStages = PG == 2 ? 4 : 6;
  static constexpr int kTmemCols = 512;
  static constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 256 + 2 * kMaxMTiles * kBM * 4;
  static_assert(kSlots >= 1 && kSlots * PG * BN <= kTmemCols, "accumulators fit tensor memory");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
  static_assert(kSmemBytes <= 232448, "shared memory per CTA");
};

template <int PG>
__global__ void __launch_bounds__(kThreads, 1)
    lm_head_pair_kernel(const __grid_constant__ CUtensorMap tm_hidden,
                        const __grid_constant__ CUtensorMap tm_w64,
                        const __grid_constant__ CUtensorMap tm_w16, const int32_t* __restrict__ targets,
                        int M, int H, int V, int G, float* __restrict__ part_max,
                        float* __restrict__ part_sum, float* __restrict__ tgt_logit, uint32_t* status,
                        uint64_t limit_ns) {
  using C = PairCfg<PG>;
  constexpr int BN = C::BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + C::kStages * C::kStageBytes);
  uint64_t* full = bars;                       // [kStages]  rank 0: both CTAs' copies
  uint64_t* empty = bars + C::kStages;         // [kStages]  each CTA: its stage is free
  uint64_t* tfull = bars + 2 * C::kStages;     // [kSlots]   each CTA: accumulators ready
  uint64_t* tempty = tfull + C::kSlots;        // [kSlots]   rank 0: both epilogues done
  uint64_t* drain = tempty + C::kSlots;        // [1]        rank 0: every MMA done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* st_max = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);
  float* st_sum = st_max + kMaxMTiles * kBM;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

  // ---- this pair's vocabulary range, in units of 16 rows
  const int nunits = (V + 15) >> 4;
  const int u_lo = (int)(((long long)pair * nunits) / npairs);
  const int u_hi = (int)(((long long)(pair + 1) * nunits) / npairs);
  const int v_lo = u_lo * 16;
  const int v_hi = min(u_hi * 16, V);
  const int ntiles = (v_hi - v_lo + BN - 1) / BN;
  const int ptiles = (M + 2 * kBM - 1) / (2 * kBM);        // 256-row pair-tiles
  const int ngroups = (ptiles + PG - 1) / PG;
  const int nitems = ntiles * ngroups;
  const int kblocks = (H + kBK - 1) / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
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
    tma_prefetch_desc(&tm_hidden);
    tma_prefetch_desc(&tm_w64);
    tma_prefetch_desc(&tm_w16);
  }
  for (int i = threadIdx.x; i < ptiles * kBM; i += kThreads) {
    st_max[i] = -INFINITY;
    st_sum[i] = 0.f;
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
  griddep_wait();                 // the prologue above touched no global memory

  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int it = 0; it < nitems && ok; ++it) {
        const int t = it / ngroups, grp = it % ngroups;
        const int v0 = v_lo + t * BN;
        const int n = min(BN, (v_hi - v0 + 31) & ~31);    // MMA N, a multiple of 32
        const int half = n >> 1;
        const int pcount = min(PG, ptiles - grp * PG);
        const uint32_t bytes = pcount * C::kABytes + half * kBK * 2;   // per CTA
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&empty[stage]), phase ^ 1, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteProdEmpty);
            ok = false;
            break;
          }
          const uint32_t fb = full0 + (uint32_t)(stage * 8);
          if (rank == 0) mbar_arrive_expect_tx(smem_u32(&full[stage]), 2 * bytes);
          uint8_t* st = ring + stage * C::kStageBytes;
          for (int j = 0; j < pcount; ++j)
            tma_load_2d_pair(smem_u32(st + j * C::kABytes), &tm_hidden, fb, kb * kBK,
                             (grp * PG + j) * 2 * kBM + (int)rank * kBM, pol_h);
          uint8_t* bsm = st + PG * C::kABytes;
          const int w0 = v0 + (int)rank * half;
          int r = 0;
          for (; r + 64 <= half; r += 64)
            tma_load_2d_pair(smem_u32(bsm + r * 128), &tm_w64, fb, kb * kBK, w0 + r, pol_w);
          for (; r < half; r += 16)
            tma_load_2d_pair(smem_u32(bsm + r * 128), &tm_w16, fb, kb * kBK, w0 + r, pol_w);
          ++issued;
          if (++stage == C::kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // rank 0 sees both CTAs' copies complete on its barriers: leave none in flight
      if (rank == 0) {
        const int pend = issued < C::kStages ? (int)issued : C::kStages;
        for (int i = 0; i < pend; ++i) {
          if (--stage < 0) {
            stage = C::kStages - 1;
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
        const int t = it / ngroups, grp = it % ngroups;
        const int v0 = v_lo + t * BN;
        const int n = min(BN, (v_hi - v0 + 31) & ~31);
        const int pcount = min(PG, ptiles - grp * PG);
        const uint32_t idesc = idesc_bf16_f32(2 * kBM, n);
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
          const uint32_t bsm = st + PG * C::kABytes;
          for (int j = 0; j < pcount; ++j) {
            const uint32_t d = tmem_base + (uint32_t)((slot * PG + j) * BN);
#pragma unroll
            for (int k16 = 0; k16 < kBK / 16; ++k16)
              tc_mma_bf16_pair(d, desc_kmajor_sw128(st + j * C::kABytes + k16 * 32),
                               desc_kmajor_sw128(bsm + k16 * 32), idesc, (kb | k16) != 0);
          }
          tc_commit_pair(smem_u32(&empty[stage]), 0x3);
          if (++stage == C::kStages) {
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
    const int row = quarter * 32 + lane;      // this CTA's row inside a pair-tile
    for (int it = 0; it < nitems; ++it) {
      const int slot = it % C::kSlots;
      const uint32_t use = it / C::kSlots;
      const int t = it / ngroups, grp = it % ngroups;
      const int v0 = v_lo + t * BN;
      const int ncols = min(BN, v_hi - v0);
      const int pcount = min(PG, ptiles - grp * PG);
      if (!mbar_wait_cluster(smem_u32(&tfull[slot]), use & 1, limit_ns)) {
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteEpiFull);
        break;
      }
      tc_fence_after();
      for (int j = 0; j < pcount; ++j) {
        const int pt = grp * PG + j;
        const int m = pt * 2 * kBM + (int)rank * kBM + row;
        float rmax = st_max[pt * kBM + row];
        float rsum = st_sum[pt * kBM + row];
        const uint32_t tbase =
            tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((slot * PG + j) * BN);
        lse_row(tbase, ncols, v0, m < M, m, G, targets, tgt_logit, rmax, rsum);
        st_max[pt * kBM + row] = rmax;
        st_sum[pt * kBM + row] = rsum;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tempty0 + (uint32_t)(slot * 8));
    }
    // publish this CTA's rows of the pair's partials (log2 domain)
    for (int pt = 0; pt < ptiles; ++pt) {
      const int m = pt * 2 * kBM + (int)rank * kBM + row;
      if (m < M) {
        part_max[(size_t)pair * M + m] = st_max[pt * kBM + row];
        part_sum[(size_t)pair * M + m] = st_sum[pt * kBM + row];
      }
    }
  }
  griddep_launch_dependents();    // the merge kernel may start launching
  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // neither CTA frees tensor memory the other may still use
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, C::kTmemCols);
}

// ---------------------------------------------------------------------------
// Vocabulary-major pair form for 257 .. 384 rows.  An MMA's M axis comes in 128 rows per
// SM, so 257-384 hidden rows as the A operand cost 384 rows of tensor work (320 rows: a
// ceiling of 83 %).  Here the operands swap: W is A (M = 256 vocabulary rows per pair MMA,
// 128 per CTA) and the hidden rows lie along N, which comes in steps of 16: Mp = rows
// rounded up to 32, issued as two MMAs of N = Mp / 2 per K step.  Each CTA of the pair loads
// its 128 W rows of a tile and a quarter Mp / 4 of the hidden rows of each of the two MMAs.
//
// Tensor memory then holds z with vocabulary ids in lanes and hidden rows in columns, so
// the log-sum-exp over the vocabulary runs across the lanes of a warp.  Per 32-column chunk
// a transposed butterfly of 31 shuffles leaves lane c with the sum over the warp's 32 ids of
// column c.  Every (lane quarter, column) keeps a reference max R in the log2 domain, raised
// only when a value passes it by more than 2^8 (one warp vote per chunk), so an ordinary
// chunk takes no max reduction at all.  Consecutive tiles alternate their accumulators
// between columns [0, Mp) and [512 - Mp, 512); the next tile's MMAs wait only until the
// epilogue has read the columns the two ranges share, which it reads first.  Eight epilogue
// warps (two per lane quarter) split the chunks.  The target logits are direct dot products
// of the hidden row with the target's W row (the definition of z_target), taken by the
// epilogue warps while the first tile's MMAs run.
namespace vt {
constexpr int kThreads = 320;                   // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr int kEpiWarps = 8;
constexpr int kMaxRows = 384;
constexpr int kStages = 5;
constexpr int kTile = 256;                      // vocabulary rows per pair MMA (128 per CTA)
constexpr int kABytes = kBM * kBK * 2;          // this CTA's 128 W rows x 64 K: 16 KB
constexpr int kStageBytes = kABytes + kMaxRows / 2 * kBK * 2;   // + up to 192 hidden rows
constexpr int kSmemBytes = kStages * kStageBytes + 1024 + 256 + 2 * 4 * kMaxRows * 4;
constexpr float kLazy = 8.f;                    // R is raised once a value exceeds it by 2^8
static_assert(kStageBytes % 1024 == 0, "stages must keep 1024-byte alignment");
static_assert(kSmemBytes <= 232448, "shared memory per CTA");
}  // namespace vt

// On entry v[i] is this lane's value of column i of a 32 x 32 block (lanes x columns); on
// exit v[0] holds the reduction over the 32 lanes of column `lane`.  Each step halves the
// columns a lane keeps and combines them with the partner's across the step's lane bit.
template <bool MAX>
__device__ __forceinline__ float warp_transpose_reduce(float (&v)[32], int lane) {
#pragma unroll
  for (int w = 16; w >= 1; w >>= 1) {
    const bool hi = (lane & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float send = hi ? v[i] : v[i + w];
      const float keep = hi ? v[i + w] : v[i];
      const float got = __shfl_xor_sync(0xffffffffu, send, w);
      v[i] = MAX ? fmaxf(keep, got) : keep + got;
    }
  }
  return v[0];
}

// One 32-column chunk of a vocabulary-major accumulator: lanes are vocabulary ids, columns
// hidden rows.  nR / S: this lane quarter's -R and running sums of the chunk's 32 columns
// (lane c owns column c).  MASKED: lanes with `valid` false lie past the pair's range.
template <bool MASKED>
__device__ __forceinline__ void vt_chunk(uint32_t taddr, bool valid, float* nR, float* S, int lane) {
  uint32_t r[32];
  tmem_ld_32x32b_x32(taddr, r);
  tmem_wait_ld();
  float nr[32], e[32];
  const float4* nr4 = reinterpret_cast<const float4*>(nR);
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const float4 x = nr4[q];
    nr[4 * q] = x.x;
    nr[4 * q + 1] = x.y;
    nr[4 * q + 2] = x.z;
    nr[4 * q + 3] = x.w;
  }
  float dmax = -INFINITY;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    float d = fmaf(__uint_as_float(r[i]), kLog2e, nr[i]);
    if (MASKED && !valid) d = -INFINITY;
    dmax = fmaxf(dmax, d);
    e[i] = ex2(d);
  }
  if (__any_sync(0xffffffffu, dmax > vt::kLazy)) {
    // rare: some value passed its column's R by more than 2^8 (always on the first tile,
    // where R = -inf): raise R to the column max and redo the chunk
#pragma unroll
    for (int i = 0; i < 32; ++i)
      e[i] = (MASKED && !valid) ? -INFINITY : __uint_as_float(r[i]) * kLog2e;
    const float cmax = warp_transpose_reduce<true>(e, lane);
    const float rold = -nR[lane];
    const float rnew = fmaxf(rold, cmax);
    if (rnew > rold) {
      S[lane] *= ex2(rold - rnew);
      nR[lane] = -rnew;
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 x = nr4[q];
      nr[4 * q] = x.x;
      nr[4 * q + 1] = x.y;
      nr[4 * q + 2] = x.z;
      nr[4 * q + 3] = x.w;
    }
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      float d = fmaf(__uint_as_float(r[i]), kLog2e, nr[i]);
      if (MASKED && !valid) d = -INFINITY;
      e[i] = ex2(d);
    }
  }
  const float csum = warp_transpose_reduce<false>(e, lane);
  S[lane] += csum;
}

// Sum of the products of eight bf16 pairs packed in two 16-byte vectors, in fp32.
__device__ __forceinline__ float dot8_bf16(const uint4 a, const uint4 b) {
  const uint32_t av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    s = fmaf(__uint_as_float(av[i] << 16), __uint_as_float(bv[i] << 16), s);
    s = fmaf(__uint_as_float(av[i] & 0xffff0000u), __uint_as_float(bv[i] & 0xffff0000u), s);
  }
  return s;
}

__global__ void __launch_bounds__(vt::kThreads, 1)
    lm_head_vt_kernel(const __grid_constant__ CUtensorMap tm_hb,
                      const __grid_constant__ CUtensorMap tm_w64,
                      const __grid_constant__ CUtensorMap tm_w16, const uint16_t* __restrict__ hidden,
                      const uint16_t* __restrict__ weight, const int32_t* __restrict__ targets, int M,
                      int Mp, int H, int V, int G, float* __restrict__ part_max,
                      float* __restrict__ part_sum, float* __restrict__ tgt_logit, uint32_t* status,
                      uint64_t limit_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* ring = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + vt::kStages * vt::kStageBytes);
  uint64_t* full = bars;                       // [vt::kStages]  rank 0: both CTAs' copies
  uint64_t* empty = bars + vt::kStages;            // [vt::kStages]  each CTA: its stage is free
  uint64_t* tfull = bars + 2 * vt::kStages;        // each CTA: the tile's accumulators are ready
  uint64_t* ovl = tfull + 1;                   // rank 0: both epilogues read the shared columns
  uint64_t* drain = ovl + 1;                   // rank 0: every MMA done
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
  float* negR = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);  // [4][vt::kMaxRows]
  float* Ssum = negR + 4 * vt::kMaxRows;                                                // [4][vt::kMaxRows]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

  // ---- this pair's vocabulary range, in units of 16 rows
  const int nunits = (V + 15) >> 4;
  const int u_lo = (int)(((long long)pair * nunits) / npairs);
  const int u_hi = (int)(((long long)(pair + 1) * nunits) / npairs);
  const int v_lo = u_lo * 16;
  const int v_hi = min(u_hi * 16, V);
  const int ntiles = (v_hi - v_lo + vt::kTile - 1) / vt::kTile;
  const int kblocks = (H + kBK - 1) / kBK;
  const int N = Mp >> 1, nb = Mp >> 2, nch = Mp >> 5;

  if (threadIdx.x == 0) {
    for (int s = 0; s < vt::kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), 1);
    }
    mbar_init(smem_u32(tfull), 1);
    mbar_init(smem_u32(ovl), 2 * vt::kEpiWarps);   // every epilogue warp of both CTAs
    mbar_init(smem_u32(drain), 1);
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_hb);
    tma_prefetch_desc(&tm_w64);
    tma_prefetch_desc(&tm_w16);
  }
  for (int i = threadIdx.x; i < 4 * vt::kMaxRows; i += vt::kThreads) {
    negR[i] = INFINITY;     // R = -inf
    Ssum[i] = 0.f;
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(tmem_holder), 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // the peer's barriers are initialised before any remote use
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  const uint32_t full0 = mapa_shared(smem_u32(&full[0]), 0);
  const uint32_t ovl0 = mapa_shared(smem_u32(ovl), 0);
  griddep_wait();                 // the prologue above touched no global memory

  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first();
      const uint64_t pol_h = policy_evict_last();
      const uint32_t hbytes = (uint32_t)Mp * kBK;       // per CTA: Mp / 2 hidden rows
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int t = 0; t < ntiles && ok; ++t) {
        // each CTA loads the W rows of its half that lie in the pair's range (rounded up to
        // 16); the A rows past them hold stale data and feed only masked lanes
        const int t0 = v_lo + t * vt::kTile;
        auto w_rows = [&](int r) { return (min(max(v_hi - t0 - r * kBM, 0), kBM) + 15) & ~15; };
        const int w0 = t0 + (int)rank * kBM, wr = w_rows((int)rank);
        const uint32_t bytes2 = (uint32_t)(w_rows(0) + w_rows(1)) * kBK * 2 + 2 * hbytes;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&empty[stage]), phase ^ 1, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteProdEmpty);
            ok = false;
            break;
          }
          const uint32_t fb = full0 + (uint32_t)(stage * 8);
          if (rank == 0) mbar_arrive_expect_tx(smem_u32(&full[stage]), bytes2);
          const uint32_t st = smem_u32(ring + stage * vt::kStageBytes);
          int r = 0;
          for (; r + 64 <= wr; r += 64)
            tma_load_2d_pair(st + r * 128, &tm_w64, fb, kb * kBK, w0 + r, pol_w);
          for (; r < wr; r += 16)
            tma_load_2d_pair(st + r * 128, &tm_w16, fb, kb * kBK, w0 + r, pol_w);
          tma_load_2d_pair(st + vt::kABytes, &tm_hb, fb, kb * kBK, (int)rank * nb, pol_h);
          tma_load_2d_pair(st + vt::kABytes + nb * 128, &tm_hb, fb, kb * kBK, N + (int)rank * nb, pol_h);
          ++issued;
          if (++stage == vt::kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (rank == 0) {
        const int pend = issued < vt::kStages ? (int)issued : vt::kStages;
        for (int i = 0; i < pend; ++i) {
          if (--stage < 0) {
            stage = vt::kStages - 1;
            phase ^= 1;
          }
          mbar_wait(smem_u32(&full[stage]), phase, limit_ns);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (rank 0)
    if (lane == 0 && rank == 0) {
      const uint32_t idesc = idesc_bf16_f32(2 * kBM, (uint32_t)N);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = 0; t < ntiles && ok; ++t) {
        // the previous tile's epilogue has read the columns this tile shares with it (and,
        // before that, all of the tile before it, whose columns this one reuses)
        if (t > 0 && !mbar_wait_cluster(smem_u32(ovl), (uint32_t)((t - 1) & 1), limit_ns)) {
          record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaTmem);
          break;
        }
        tc_fence_after();
        const uint32_t d0 = tmem_base + (uint32_t)((t & 1) ? 512 - Mp : 0);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&full[stage]), phase, limit_ns)) {
            record_error(status, FVRAG_ERR_TIMEOUT, kSiteMmaFull);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(ring + stage * vt::kStageBytes);
#pragma unroll
          for (int k16 = 0; k16 < kBK / 16; ++k16) {
            const uint64_t a = desc_kmajor_sw128(st + k16 * 32);
            tc_mma_bf16_pair(d0, a, desc_kmajor_sw128(st + vt::kABytes + k16 * 32), idesc,
                             (kb | k16) != 0);
            tc_mma_bf16_pair(d0 + (uint32_t)N, a,
                             desc_kmajor_sw128(st + vt::kABytes + nb * 128 + k16 * 32), idesc,
                             (kb | k16) != 0);
          }
          tc_commit_pair(smem_u32(&empty[stage]), 0x3);
          if (++stage == vt::kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        tc_commit_pair(smem_u32(tfull), 0x3);
      }
      tc_commit_pair(smem_u32(drain), 0x1);
      if (!mbar_wait(smem_u32(drain), 0, limit_ns)) record_error(status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int ew = warp - 2, quarter = warp & 3, grp = ew >> 2;
    // target logits z[m, t] = <hidden[m], W[t]>, split over every epilogue warp of the grid
    for (int i = (int)blockIdx.x * vt::kEpiWarps + ew; i < M * G; i += (int)gridDim.x * vt::kEpiWarps) {
      const int tg = __ldg(&targets[i]);
      if (tg < 0 || tg >= V) continue;          // the merge writes NaN for these
      const uint4* hp = reinterpret_cast<const uint4*>(hidden + (size_t)(i / G) * H);
      const uint4* wp = reinterpret_cast<const uint4*>(weight + (size_t)tg * H);
      float acc = 0.f;
      for (int c = lane; c < (H >> 3); c += 32) acc += dot8_bf16(__ldg(hp + c), __ldg(wp + c));
      acc = warp_sum(acc);
      if (lane == 0) tgt_logit[i] = acc;
    }
    float* nRq = negR + quarter * vt::kMaxRows;
    float* Sq = Ssum + quarter * vt::kMaxRows;
    const int vl = (int)rank * kBM + quarter * 32 + lane;   // this thread's row inside a tile
    const uint32_t lane_addr = tmem_base + ((uint32_t)(quarter * 32) << 16);
    for (int t = 0; t < ntiles; ++t) {
      if (!mbar_wait_cluster(smem_u32(tfull), (uint32_t)(t & 1), limit_ns)) {
        record_error(status, FVRAG_ERR_TIMEOUT, kSiteEpiFull);
        break;
      }
      tc_fence_after();
      const int v0 = v_lo + t * vt::kTile;
      const bool masked = v0 + vt::kTile > v_hi;
      const bool valid = v0 + vl < v_hi;
      const uint32_t tb = lane_addr + (uint32_t)((t & 1) ? 512 - Mp : 0);
      // chunks whose columns the next tile's accumulators share: [16 - nch, nch) of an even
      // tile, [0, 2 nch - 16) of an odd one
      const int lo = (t & 1) ? 0 : 16 - nch, hi = (t & 1) ? 2 * nch - 16 : nch;
      for (int pass = 0; pass < 2; ++pass) {
        for (int k = grp; k < nch; k += 2) {
          if ((k >= lo && k < hi) != (pass == 0)) continue;
          if (masked)
            vt_chunk<true>(tb + (uint32_t)(32 * k), valid, nRq + 32 * k, Sq + 32 * k, lane);
          else
            vt_chunk<false>(tb + (uint32_t)(32 * k), valid, nRq + 32 * k, Sq + 32 * k, lane);
        }
        if (pass == 0) {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(ovl0);
        }
      }
    }
    // fold the four lane quarters of every column into this CTA's partial (log2 domain)
    asm volatile("bar.sync 1, %0;" ::"n"(vt::kEpiWarps * 32) : "memory");
    for (int m = ew * 32 + lane; m < M; m += vt::kEpiWarps * 32) {
      float mx = -INFINITY;
#pragma unroll
      for (int q = 0; q < 4; ++q) mx = fmaxf(mx, -negR[q * vt::kMaxRows + m]);
      float s = 0.f;
      if (mx != -INFINITY) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float rq = -negR[q * vt::kMaxRows + m];
          if (rq != -INFINITY) s += Ssum[q * vt::kMaxRows + m] * ex2(rq - mx);
        }
      }
      part_max[(size_t)blockIdx.x * M + m] = mx;
      part_sum[(size_t)blockIdx.x * M + m] = s;
    }
  }
  griddep_launch_dependents();    // the merge kernel may start launching
  tc_fence_before();
  __syncthreads();
  cluster_sync();                 // neither CTA frees tensor memory the other may still use
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, 512);
}

// One warp per row: lse = ln 2 * (M2 + log2 S) with M2 = max_b max_b and
// S = sum_b sum_b * 2^(max_b - M2) (partials in the log2 domain); logprob = z_target - lse.
__global__ void lm_merge_kernel(const float* __restrict__ part_max, const float* __restrict__ part_sum,
                                const float* __restrict__ tgt_logit,
                                const int32_t* __restrict__ targets, int M, int V, int G, int nparts,
                                float* __restrict__ logprob, float* __restrict__ lse_out) {
  griddep_wait();
  griddep_launch_dependents();
  const int m = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= M) return;
  // one pass over the partials: each lane folds its (max, sum) pairs online, then the
  // warp combines the 32 lane states
  float mx = -INFINITY, s = 0.f;
#pragma unroll 4
  for (int b = lane; b < nparts; b += 32) {
    const float pm = part_max[(size_t)b * M + m];
    const float ps = part_sum[(size_t)b * M + m];
    if (pm > mx) {
      s = s * ex2(mx - pm) + ps;
      mx = pm;
    } else if (pm != -INFINITY) {
      s += ps * ex2(pm - mx);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, mx, o);
    const float os = __shfl_xor_sync(0xffffffffu, s, o);
    const float nm = fmaxf(mx, om);
    s = (mx == -INFINITY ? 0.f : s * ex2(mx - nm)) + (om == -INFINITY ? 0.f : os * ex2(om - nm));
    mx = nm;
  }
  const float l = kLn2 * (mx + __log2f(s));
  if (lane == 0 && lse_out) lse_out[m] = l;
  for (int g = lane; g < G; g += 32) {
    const int32_t t = targets[(size_t)m * G + g];
    logprob[(size_t)m * G + g] =
        (t >= 0 && t < V) ? tgt_logit[(size_t)m * G + g] - l : __int_as_float(0x7fc00000);
  }
}

struct Plan {
  int ctas;       // CTAs of the 1-CTA forms; pairs of the pair forms
  int parts;      // per-row partials the merge folds: one per CTA, or per pair
  int bn, mg;     // mg = 0 / -1: the pair form with two / one pair-tiles per pass;
                  // mg = 2: the vocabulary-major pair form
};

// Pairs (2-CTA clusters) of a pair-form kernel that can be resident at once on the current
// device; `cache` holds one entry per device.
static int resident_pairs(const void* kern, int threads, int smem, int* cache, std::mutex& mu) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) ==
        cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      const int sms = std::max(2, sm_count());
      cfg.gridDim = dim3(sms / 2 * 2);
      cfg.blockDim = dim3(threads);
      cfg.dynamicSmemBytes = smem;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();
    cache[dev] = std::max(1, std::min(n, std::min(sm_count() / 2, kMaxCtas / 2)));
  }
  return cache[dev];
}

static int max_pairs() {
  static std::mutex mu;
  static int cache[64] = {0};
  return resident_pairs(reinterpret_cast<const void*>(lm_head_pair_kernel<2>), kThreads,
                        PairCfg<2>::kSmemBytes, cache, mu);
}

static int max_pairs_vt() {
  static std::mutex mu;
  static int cache[64] = {0};
  return resident_pairs(reinterpret_cast<const void*>(lm_head_vt_kernel), vt::kThreads,
                        vt::kSmemBytes, cache, mu);
}

// `sms`: the most SMs the grid may occupy (the device's count, or the caller's budget).
static Plan make_plan(const fvrag_lm_desc* d, int sms) {
  Plan p;
  const int mtiles = (d->rows + kBM - 1) / kBM;
  p.bn = 256;
  // one M-tile: <256, 1>; two: the pair form with one pair-tile and two accumulator sets;
  // three: the vocabulary-major pair form (hidden rows along N, no padding to 384); more:
  // the pair form with two pair-tiles per pass
  p.mg = mtiles == 1 ? 1 : mtiles == 3 ? 2 : mtiles == 2 ? -1 : 0;
  const int nunits = (d->vocab + 15) / 16;
  const int budget = sms > 0 ? sms : 148;
  if (p.mg == 1) {
    p.ctas = std::max(1, std::min(std::min(budget, kMaxCtas), nunits));
    p.parts = p.ctas;
  } else {
    const int pairs = p.mg == 2 ? max_pairs_vt() : max_pairs();
    p.ctas = std::max(1, std::min(std::min(pairs, std::max(1, budget / 2)), nunits));
    p.parts = p.mg == 2 ? 2 * p.ctas : p.ctas;
  }
  return p;
}

template <int PG>
static fvrag_status launch_pair(const Plan& p, const CUtensorMap& th, const CUtensorMap& tw64,
                                const CUtensorMap& tw16, const int32_t* targets,
                                const fvrag_lm_desc* d, float* pmax, float* psum, float* ptgt,
                                uint32_t* status, cudaStream_t s) {
  using C = PairCfg<PG>;
  auto kern = lm_head_pair_kernel<PG>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * p.ctas);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::kSmemBytes;
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
  if (counted(cudaLaunchKernelEx(&cfg, kern, th, tw64, tw16, targets, d->rows, d->hidden,
                                 d->vocab, d->gathers, pmax, psum, ptgt, status,
                                 wait_limit_ns())) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

static fvrag_status launch_vt(const Plan& p, const CUtensorMap& thb, const CUtensorMap& tw64,
                              const CUtensorMap& tw16, const void* hidden, const void* weight, const int32_t* targets,
                              const fvrag_lm_desc* d, int Mp, float* pmax, float* psum,
                              float* ptgt, uint32_t* status, cudaStream_t s) {
  auto kern = lm_head_vt_kernel;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, vt::kSmemBytes) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * p.ctas);
  cfg.blockDim = dim3(vt::kThreads);
  cfg.dynamicSmemBytes = vt::kSmemBytes;
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
  if (counted(cudaLaunchKernelEx(&cfg, kern, thb, tw64, tw16, static_cast<const uint16_t*>(hidden),
                                 static_cast<const uint16_t*>(weight), targets, d->rows, Mp,
                                 d->hidden, d->vocab, d->gathers, pmax, psum, ptgt, status,
                                 wait_limit_ns())) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

// 0 (every SM) or 1 .. the device's SM count.
static bool budget_ok(int32_t budget) {
  const int s = sm_count();
  return budget >= 0 && (s <= 0 || budget <= s);
}

static size_t ws_bytes(const fvrag_lm_desc* d) {
  const size_t M = (size_t)d->rows;
  return kWsHeaderBytes + 2 * (size_t)kMaxCtas * M * 4 + M * (size_t)d->gathers * 4;
}

template <int BN, int MG>
static fvrag_status launch(const Plan& p, const CUtensorMap& th, const CUtensorMap& tw64,
                           const CUtensorMap& tw16, const int32_t* targets, const fvrag_lm_desc* d,
                           int hrows, float* pmax, float* psum, float* ptgt, uint32_t* status,
                           cudaStream_t s) {
  using C = Cfg<BN, MG>;
  auto kern = lm_head_kernel<BN, MG>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  if (launch_pdl(kern, dim3(p.ctas), dim3(kThreads), (size_t)C::kSmemBytes, s, th, tw64, tw16, targets,
                 d->rows, d->hidden, d->vocab, d->gathers, hrows, pmax, psum, ptgt, status,
                 wait_limit_ns()) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

}  // namespace lm
}  // namespace fvrag

using namespace fvrag;

extern "C" size_t fvrag_score_logprobs_workspace(const fvrag_lm_desc* d) {
  if (!d || d->rows < 1 || d->hidden < 8 || d->vocab < 1 || d->gathers < 1 ||
      !lm::budget_ok(d->sm_budget))
    return 0;
  return lm::ws_bytes(d);
}

extern "C" fvrag_status fvrag_score_logprobs(const fvrag_lm_desc* d, const void* hidden,
                                             const void* weight, const int32_t* targets,
                                             float* logprob, float* lse, void* ws, size_t ws_size,
                                             fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_score_logprobs");
  using namespace lm;
  if (!d || !hidden || !weight || !targets || !logprob) return FVRAG_ERR_INVALID_ARG;
  if (d->rows < 1 || d->hidden < 1 || d->vocab < 1 || d->gathers < 1 || d->flags != 0 ||
      !budget_ok(d->sm_budget))
    return FVRAG_ERR_INVALID_ARG;
  if (d->gathers > kMaxGathers || d->rows > kMaxMTiles * kBM) return FVRAG_ERR_UNSUPPORTED;
  if (d->hidden % 8 != 0) return FVRAG_ERR_MISALIGNED;
  if (!aligned16(hidden) || !aligned16(weight)) return FVRAG_ERR_MISALIGNED;
  if (!ws || ws_size < ws_bytes(d)) return FVRAG_ERR_WORKSPACE;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;

  const Plan p = make_plan(d, sm_plan(d->sm_budget));
  const uint64_t H = (uint64_t)d->hidden, M = (uint64_t)d->rows, V = (uint64_t)d->vocab;
  CUtensorMap th, tw64, tw16;
  // one M-tile: load only the rows that exist (rounded to 16), not all 128
  const int hrows = M <= (uint64_t)kBM ? (int)((M + 15) / 16 * 16) : kBM;
  {
    const uint64_t dims[2] = {H, M}, strides[1] = {H * 2};
    const uint32_t box[2] = {(uint32_t)kBK, (uint32_t)hrows};
    if (!encode_tmap_bf16(&th, hidden, 2, dims, strides, box, true)) return FVRAG_ERR_CUDA;
  }
  {
    const uint64_t dims[2] = {H, V}, strides[1] = {H * 2};
    const uint32_t box64[2] = {(uint32_t)kBK, 64u}, box16[2] = {(uint32_t)kBK, 16u};
    if (!encode_tmap_bf16(&tw64, weight, 2, dims, strides, box64, true)) return FVRAG_ERR_CUDA;
    if (!encode_tmap_bf16(&tw16, weight, 2, dims, strides, box16, true)) return FVRAG_ERR_CUDA;
  }
  uint8_t* base = reinterpret_cast<uint8_t*>(ws);
  uint32_t* status = reinterpret_cast<uint32_t*>(base);
  float* pmax = reinterpret_cast<float*>(base + kWsHeaderBytes);
  float* psum = pmax + (size_t)kMaxCtas * M;
  float* ptgt = psum + (size_t)kMaxCtas * M;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  fvrag_status st;
  if (p.mg == 2) {
    // vocabulary-major form: hidden rows in boxes of Mp / 4 (a quarter of the padded rows)
    const int Mp = (int)((M + 31) / 32 * 32);
    CUtensorMap thb;
    const uint64_t dims[2] = {H, M}, strides[1] = {H * 2};
    const uint32_t box[2] = {(uint32_t)kBK, (uint32_t)(Mp / 4)};
    if (!encode_tmap_bf16(&thb, hidden, 2, dims, strides, box, true)) return FVRAG_ERR_CUDA;
    st = launch_vt(p, thb, tw64, tw16, hidden, weight, targets, d, Mp, pmax, psum, ptgt, status, s);
  } else if (p.mg == 0)
    st = launch_pair<2>(p, th, tw64, tw16, targets, d, pmax, psum, ptgt, status, s);
  else if (p.mg == -1)
    st = launch_pair<1>(p, th, tw64, tw16, targets, d, pmax, psum, ptgt, status, s);
  else
    st = launch<256, 1>(p, th, tw64, tw16, targets, d, hrows, pmax, psum, ptgt, status, s);
  if (st != FVRAG_OK) return st;
  const int rows_per_block = 8;
  if (launch_pdl(lm_merge_kernel, dim3((d->rows + rows_per_block - 1) / rows_per_block),
                 dim3(32 * rows_per_block), 0, s, (const float*)pmax, (const float*)psum,
                 (const float*)ptgt, targets, d->rows, d->vocab, d->gathers, p.parts, logprob,
                 lse) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

// ---------------------------------------------------------------------------
// Allocation-free variant of fvrag_score_logprobs.
//
// Some callers cannot call cudaMalloc: a host runtime that hands out only
// pre-registered buffers, an embedded engine whose allocator is owned by
// someone else, or a caller working under a memory budget that forbids new
// device allocations after start-up.  For them this entry point keeps the LM
// head's scratch (the workspace header and the per-CTA partial max / sum and
// gathered target logits) in a file-scope device array of fixed size instead of
// a caller-provided workspace.  Every GPU that loads the library holds the
// array until the process exits.
namespace fvrag {
namespace lm {

constexpr int kNoAllocMaxRows = 1024;
constexpr size_t kNoAllocBytes = kWsHeaderBytes + 2 * (size_t)kMaxCtas * kNoAllocMaxRows * 4 +
                                 (size_t)kNoAllocMaxRows * kMaxGathers * 4;

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocBytes];

// Device address of g_noalloc_scratch in the current context.  In host code the
// array's name is only a host-side stand-in, so the address is looked up with the
// device current (the first call on a device) and cached per device together with
// the context it was found in: when that context changes (after cudaDeviceReset the
// module is loaded again, possibly elsewhere) the address is looked up again.
static void* noalloc_scratch_address() {
  static std::mutex mu;
  static void* addr[64] = {nullptr};
  static CUcontext ctx[64] = {nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] && ctx[dev] != nullptr && ctx[dev] == current_cu_context()) return addr[dev];
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
  addr[dev] = p;
  ctx[dev] = current_cu_context();   // current now: the lookup initialised the runtime
  return p;
}

}  // namespace lm
}  // namespace fvrag

extern "C" fvrag_status fvrag_score_logprobs_noalloc(const fvrag_lm_desc* d, const void* hidden,
                                                     const void* weight, const int32_t* targets,
                                                     float* logprob, float* lse,
                                                     fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_score_logprobs_noalloc");
  using namespace lm;
  // reject bad arguments before anything is enqueued
  if (!d || !hidden || !weight || !targets || !logprob) return FVRAG_ERR_INVALID_ARG;
  if (d->rows < 1 || d->hidden < 1 || d->vocab < 1 || d->gathers < 1 || d->flags != 0 ||
      !budget_ok(d->sm_budget))
    return FVRAG_ERR_INVALID_ARG;
  if (d->rows > kNoAllocMaxRows || d->gathers > kMaxGathers) return FVRAG_ERR_UNSUPPORTED;
  if (d->hidden % 8 != 0 || !aligned16(hidden) || !aligned16(weight)) return FVRAG_ERR_MISALIGNED;
  void* scratch = noalloc_scratch_address();
  if (!scratch) return FVRAG_ERR_CUDA;
  // the status word reports this call only
  if (cudaMemsetAsync(scratch, 0, kWsHeaderBytes, reinterpret_cast<cudaStream_t>(stream)) !=
      cudaSuccess)
    return FVRAG_ERR_CUDA;
  return fvrag_score_logprobs(d, hidden, weight, targets, logprob, lse, scratch, kNoAllocBytes,
                              stream);
}

// Status of the last fvrag_score_logprobs_noalloc call on the current device: its
// device-side status word lives in the static array, out of the caller's reach.
extern "C" fvrag_status fvrag_score_logprobs_noalloc_status(fvrag_stream_t stream) {
  using namespace lm;
  void* scratch = noalloc_scratch_address();
  if (!scratch) return FVRAG_ERR_CUDA;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  uint32_t v = 0;
  if (cudaMemcpy(&v, scratch, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return status_of_word(v);
}
