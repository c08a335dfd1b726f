// K1: one attention layer of the verifier forward over all candidate rows
// (Eq. 6 / Eq. 11): every token l of candidate k attends to the P_q tokens of
// the shared prefix and to tokens 0..l of its own candidate.
//
// The prefix part dominates (P up to 32768 keys vs L <= 64 tail keys) and is
// shared by every candidate row, so it is computed as a split-KV flash pass in
// which ALL K x L x (hq/hkv) query rows that use one KV head are packed into
// the rows of the tensor-core tiles (GQA packing): each prefix K/V tile is read
// from HBM once per (KV head, key split) and reused by every candidate row.
//
// prefix kernel  grid = Qn x hkv x key-splits x row-tiles; one CTA computes 128
//                query rows (T tokens x the hq/hkv heads of one KV head) against
//                one key range.  Warp 8 streams 64-key K/V tiles with TMA (3-D
//                maps over [keys][hkv][D], 128-byte swizzle) into a 3-stage ring;
//                warps 0-7 (16 rows each) run S = Q K^T and O += P V on the tensor
//                cores (bf16 mma.sync m16n8k16, fp32 accumulate) with an online
//                softmax in registers, then write the normalised partial O and
//                its log-sum-exp to the workspace.
// tail+merge     one warp per (token, head): attention over the candidate's own
//                tokens 0..l (at most 64 keys, CUDA cores), then a log-sum-exp
//                merge of the tail with every prefix split; writes bf16 out and
//                the fp32 lse.
#include <cuda_bf16.h>

#include <algorithm>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {
namespace attn {

constexpr int kConsumerWarps = 8;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kRowsPerTile = 128;
constexpr int kKeysPerBlock = 64;
constexpr int kStages = 3;
constexpr int kTargetCtas = 304;   // split plan aims at ~2 CTAs per SM (fixed: plan is device-independent)
constexpr int kMaxTail = 64;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

enum : uint32_t { kSiteQ = 0x101, kSiteFull = 0x102, kSiteEmpty = 0x103 };

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Address of 16-byte chunk c (0 .. D/8-1) of row i in a tile stored as D/64
// column halves of `rows_per_half` rows x 128 B, each with the 128-byte swizzle
// (chunk index XOR row mod 8, the layout TMA writes).
__device__ __forceinline__ uint32_t sw128(uint32_t base, int rows_per_half, int i, int c) {
  return base + (uint32_t)((c >> 3) * rows_per_half * 128 + i * 128 + (((c & 7) ^ (i & 7)) << 4));
}

struct PrefixArgs {
  const int32_t* offs;
  float* part_o;      // [nsplit][Qn*K*L][hq][D]
  float* part_lse;    // [nsplit][Qn*K*L][hq]
  uint32_t* status;
  uint64_t limit_ns;
  int Qn, KL, hq, hkv, grp, T, mtiles, nsplit, chunk;
  float scale_log2;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_attn_kernel(const __grid_constant__ CUtensorMap tm_q,
                       const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, const PrefixArgs a) {
  constexpr int NH = D / 64;                               // 128-byte column halves
  constexpr int kQBytes = NH * kRowsPerTile * 128;          // Q tile
  constexpr int kKVHalf = kKeysPerBlock * 128;              // one half of a K or V tile
  constexpr int kStageBytes = 2 * NH * kKVHalf;             // K + V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* q_s = smem;
  uint8_t* ring = smem + kQBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(ring + kStages * kStageBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + kStages;
  uint64_t* qbar = bars + 2 * kStages;

  int b = blockIdx.x;
  const int mt = b % a.mtiles;
  b /= a.mtiles;
  const int split = b % a.nsplit;
  b /= a.nsplit;
  const int g = b % a.hkv;
  const int qi = b / a.hkv;
  const int P = a.offs[qi + 1] - a.offs[qi];
  const int key_lo = split * a.chunk;
  const int key_hi = min(P, key_lo + a.chunk);
  const int nblocks = key_hi > key_lo ? (key_hi - key_lo + kKeysPerBlock - 1) / kKeysPerBlock : 0;
  const int tok0 = mt * a.T;                                // first token of this row tile
  const int rows = min(a.T, a.KL - tok0) * a.grp;           // valid rows in the tile

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&full[s]), 1);
      mbar_init(smem_u32(&empty[s]), kConsumerWarps);
    }
    mbar_init(smem_u32(qbar), 1);
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0 && nblocks > 0) {
      const uint64_t pol_kv = policy_evict_last();   // re-read by the other row tiles
      const uint64_t pol_q = policy_evict_first();
      const uint32_t qb = smem_u32(qbar);
      mbar_arrive_expect_tx(qb, NH * a.grp * a.T * 128);
      for (int h = 0; h < NH; ++h)
        tma_load_3d(smem_u32(q_s + h * kRowsPerTile * 128), &tm_q, qb, h * 64, g * a.grp,
                    qi * a.KL + tok0, pol_q);
      int stage = 0;
      uint32_t phase = 0;
      const int kbase = a.offs[qi] + key_lo;
      for (int blk = 0; blk < nblocks; ++blk) {
        if (!mbar_wait(smem_u32(&empty[stage]), phase ^ 1, a.limit_ns)) {
          record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteEmpty);
          break;
        }
        const uint32_t fb = smem_u32(&full[stage]);
        mbar_arrive_expect_tx(fb, kStageBytes);
        uint8_t* st = ring + stage * kStageBytes;
        const int key = kbase + blk * kKeysPerBlock;
        for (int h = 0; h < NH; ++h) {
          tma_load_3d(smem_u32(st + h * kKVHalf), &tm_k, fb, h * 64, g, key, pol_kv);
          tma_load_3d(smem_u32(st + (NH + h) * kKVHalf), &tm_v, fb, h * 64, g, key, pol_kv);
        }
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1;
        }
      }
      // drain: no copy may still be in flight when the CTA exits
      mbar_wait(qb, 0, a.limit_ns);
      const int pend = min(nblocks, kStages);
      for (int i = 0; i < pend; ++i) {
        if (--stage < 0) {
          stage = kStages - 1;
          phase ^= 1;
        }
        mbar_wait(smem_u32(&full[stage]), phase, a.limit_ns);
      }
    }
    return;
  }

  // ------------------------------------------------------------ consumers
  const int r0 = warp * 16;              // first tile row of this warp
  const int gq = lane >> 2, tq = lane & 3;
  float o[D / 8][4];
#pragma unroll
  for (int n = 0; n < D / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

  if (nblocks > 0) {
    bool ok = mbar_wait(smem_u32(qbar), 0, a.limit_ns);
    if (!ok) record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteQ);
    uint32_t qf[D / 16][4];
    const uint32_t qbase = smem_u32(q_s);
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks)
      ldsm_x4(sw128(qbase, kRowsPerTile, r0 + (lane & 15), 2 * ks + (lane >> 4)), qf[ks]);

    int stage = 0;
    uint32_t phase = 0;
    for (int blk = 0; blk < nblocks && ok; ++blk) {
      if (!mbar_wait(smem_u32(&full[stage]), phase, a.limit_ns)) {
        record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteFull);
        break;
      }
      const uint32_t kb = smem_u32(ring + stage * kStageBytes);
      const uint32_t vb = kb + NH * kKVHalf;
      // S = Q K^T over 64 keys: 8 n-tiles of 8 keys
      float s[8][4];
#pragma unroll
      for (int n = 0; n < 8; ++n) s[n][0] = s[n][1] = s[n][2] = s[n][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t kf[4];
          ldsm_x4(sw128(kb, kKeysPerBlock, 16 * np + (lane & 7) + ((lane >> 4) << 3),
                        2 * ks + ((lane >> 3) & 1)),
                  kf);
          mma_bf16(s[2 * np], qf[ks], kf[0], kf[1]);
          mma_bf16(s[2 * np + 1], qf[ks], kf[2], kf[3]);
        }
      }
      // online softmax (base-2 domain)
      const int kfirst = key_lo + blk * kKeysPerBlock;
      float bmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
      for (int n = 0; n < 8; ++n) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kfirst + 8 * n + 2 * tq + (e & 1);
          const float v = key < key_hi ? s[n][e] * a.scale_log2 : -INFINITY;
          s[n][e] = v;
          bmax[e >> 1] = fmaxf(bmax[e >> 1], v);
        }
      }
      float corr[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        bmax[h] = fmaxf(bmax[h], __shfl_xor_sync(0xffffffffu, bmax[h], 1));
        bmax[h] = fmaxf(bmax[h], __shfl_xor_sync(0xffffffffu, bmax[h], 2));
        const float nm = fmaxf(mrow[h], bmax[h]);
        corr[h] = ex2(mrow[h] - nm);
        mrow[h] = nm;
      }
      float bsum[2] = {0.f, 0.f};
#pragma unroll
      for (int n = 0; n < 8; ++n) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float p = ex2(s[n][e] - mrow[e >> 1]);
          s[n][e] = p;
          bsum[e >> 1] += p;
        }
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) lrow[h] = lrow[h] * corr[h] + bsum[h];
#pragma unroll
      for (int n = 0; n < D / 8; ++n) {
        o[n][0] *= corr[0];
        o[n][1] *= corr[0];
        o[n][2] *= corr[1];
        o[n][3] *= corr[1];
      }
      // O += P V over the 64 keys (4 k-steps of 16)
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t pa[4];
        pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
        pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
        pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
        pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
          uint32_t vf[4];
          ldsm_x4_t(sw128(vb, kKeysPerBlock, 16 * kk + (lane & 7) + (((lane >> 3) & 1) << 3),
                          2 * dp + (lane >> 4)),
                    vf);
          mma_bf16(o[2 * dp], pa, vf[0], vf[1]);
          mma_bf16(o[2 * dp + 1], pa, vf[2], vf[3]);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[stage]));
      if (++stage == kStages) {
        stage = 0;
        phase ^= 1;
      }
    }
  }
  // finish the row sums across the quad, write the normalised partial
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    lrow[h] += __shfl_xor_sync(0xffffffffu, lrow[h], 1);
    lrow[h] += __shfl_xor_sync(0xffffffffu, lrow[h], 2);
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int r = r0 + gq + 8 * h;
    if (r >= rows) continue;
    const int tok = tok0 + r / a.grp;
    const int head = g * a.grp + r % a.grp;
    const size_t row = ((size_t)split * a.Qn * a.KL + (size_t)qi * a.KL + tok) * a.hq + head;
    const bool any = lrow[h] > 0.f;
    const float inv = any ? 1.f / lrow[h] : 0.f;
    float* dst = a.part_o + row * D;
#pragma unroll
    for (int n = 0; n < D / 8; ++n) {
      float2 v = make_float2(o[n][2 * h] * inv, o[n][2 * h + 1] * inv);
      *reinterpret_cast<float2*>(dst + 8 * n + 2 * tq) = v;
    }
    if (tq == 0) a.part_lse[row] = any ? kLn2 * (mrow[h] + __log2f(lrow[h])) : -INFINITY;
  }
}

// One warp per (query, candidate, token l, head h).  Lane j (< l+1) scores tail
// key j; the weighted sum over tail values is split over lanes by D; then the
// tail result is merged with every prefix split by log-sum-exp weights.
template <int D>
__global__ void tail_merge_kernel(const __nv_bfloat16* __restrict__ q,
                                  const __nv_bfloat16* __restrict__ k_tail,
                                  const __nv_bfloat16* __restrict__ v_tail,
                                  const float* __restrict__ part_o, const float* __restrict__ part_lse,
                                  int nsplit, int Qn, int K, int L, int hq, int hkv, float scale,
                                  __nv_bfloat16* __restrict__ out, float* __restrict__ lse_out) {
  constexpr int DPL = D / 32;  // elements per lane
  const long long rowid = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const long long nrows = (long long)Qn * K * L * hq;
  if (rowid >= nrows) return;
  const int lane = threadIdx.x & 31;
  const int h = (int)(rowid % hq);
  const long long tok = rowid / hq;           // (qi*K + k)*L + l
  const int l = (int)(tok % L);
  const long long cand = tok / L;             // qi*K + k
  const int g = h / (hq / hkv);

  // q row in fp32, DPL elements per lane (contiguous)
  float qv[DPL];
  {
    const __nv_bfloat16* qr = q + rowid * D + lane * DPL;
#pragma unroll
    for (int i = 0; i < DPL; i += 2) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(qr + i));
      qv[i] = f.x;
      qv[i + 1] = f.y;
    }
  }
  // scores of tail keys 0..l: each key's dot is a warp reduction
  float my_s[kMaxTail / 32] = {-INFINITY, -INFINITY};
  float tmax = -INFINITY;
  for (int j = 0; j <= l; ++j) {
    const __nv_bfloat16* kr = k_tail + ((cand * L + j) * hkv + g) * D + lane * DPL;
    float dot = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; i += 2) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(kr + i));
      dot = fmaf(qv[i], f.x, fmaf(qv[i + 1], f.y, dot));
    }
    dot = warp_sum(dot) * scale;
    if ((j & 31) == lane) my_s[j >> 5] = dot;
    tmax = fmaxf(tmax, dot);
  }
  float acc[DPL];
#pragma unroll
  for (int i = 0; i < DPL; ++i) acc[i] = 0.f;
  float tsum = 0.f;
  for (int j = 0; j <= l; ++j) {
    const float sj = __shfl_sync(0xffffffffu, my_s[j >> 5], j & 31);
    const float p = __expf(sj - tmax);
    tsum += p;
    const __nv_bfloat16* vr = v_tail + ((cand * L + j) * hkv + g) * D + lane * DPL;
#pragma unroll
    for (int i = 0; i < DPL; i += 2) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(vr + i));
      acc[i] = fmaf(p, f.x, acc[i]);
      acc[i + 1] = fmaf(p, f.y, acc[i + 1]);
    }
  }
  const float tail_lse = tmax + __logf(tsum);
  // merge: weights exp(lse_i - LSE)
  float M = tail_lse;
  for (int s = 0; s < nsplit; ++s) M = fmaxf(M, part_lse[(size_t)s * nrows + rowid]);
  float wt = __expf(tail_lse - M);
  float den = wt;
  float res[DPL];
#pragma unroll
  for (int i = 0; i < DPL; ++i) res[i] = acc[i] / tsum * wt;
  for (int s = 0; s < nsplit; ++s) {
    const float ls = part_lse[(size_t)s * nrows + rowid];
    if (ls == -INFINITY) continue;
    const float w = __expf(ls - M);
    den += w;
    const float* po = part_o + ((size_t)s * nrows + rowid) * D + lane * DPL;
#pragma unroll
    for (int i = 0; i < DPL; i += 2) {
      const float2 f = *reinterpret_cast<const float2*>(po + i);
      res[i] = fmaf(w, f.x, res[i]);
      res[i + 1] = fmaf(w, f.y, res[i + 1]);
    }
  }
  const float inv = 1.f / den;
  __nv_bfloat16* orow = out + rowid * D + lane * DPL;
#pragma unroll
  for (int i = 0; i < DPL; i += 2)
    *reinterpret_cast<__nv_bfloat162*>(orow + i) = __floats2bfloat162_rn(res[i] * inv, res[i + 1] * inv);
  if (lane == 0 && lse_out) lse_out[rowid] = M + __logf(den);
}

struct Plan {
  int grp, T, mtiles, nsplit, chunk;
};

static Plan make_plan(const fvrag_attn_desc* d) {
  Plan p;
  p.grp = d->hq / d->hkv;
  p.T = std::max(1, kRowsPerTile / p.grp);
  const int KL = d->num_cand * d->cand_len;
  p.mtiles = (KL + p.T - 1) / p.T;
  if (d->max_prefix <= 0) {
    p.nsplit = 0;
    p.chunk = 0;
    return p;
  }
  const long long base = (long long)d->num_queries * d->hkv * p.mtiles;
  const int max_blocks = (d->max_prefix + kKeysPerBlock - 1) / kKeysPerBlock;
  int ns = (int)std::min<long long>((kTargetCtas + base - 1) / base, max_blocks);
  ns = std::max(ns, 1);
  const int per = (max_blocks + ns - 1) / ns;   // key blocks per split
  p.chunk = per * kKeysPerBlock;
  p.nsplit = (max_blocks + per - 1) / per;
  return p;
}

static size_t ws_bytes(const fvrag_attn_desc* d) {
  const Plan p = make_plan(d);
  const size_t rows = (size_t)d->num_queries * d->num_cand * d->cand_len * d->hq;
  return kWsHeaderBytes + (size_t)p.nsplit * rows * ((size_t)d->head_dim + 1) * 4;
}

template <int D>
static size_t smem_bytes() {
  return (size_t)(D / 64) * kRowsPerTile * 128 + (size_t)kStages * 2 * (D / 64) * kKeysPerBlock * 128 +
         1024 + 256;
}

}  // namespace attn
}  // namespace fvrag

using namespace fvrag;

extern "C" size_t fvrag_verify_attn_workspace(const fvrag_attn_desc* d) {
  if (!d || d->num_queries < 1 || d->num_cand < 1 || d->cand_len < 1 || d->hq < 1 || d->hkv < 1 ||
      d->hq % d->hkv || (d->head_dim != 64 && d->head_dim != 128) || d->max_prefix < 0)
    return 0;
  return attn::ws_bytes(d);
}

extern "C" fvrag_status fvrag_verify_attn(const fvrag_attn_desc* d, const void* q,
                                          const void* k_prefix, const void* v_prefix,
                                          const int32_t* prefix_offsets, const void* k_tail,
                                          const void* v_tail, void* out, float* lse, void* ws,
                                          size_t ws_size, fvrag_stream_t stream) {
  using namespace attn;
  if (!d || !q || !prefix_offsets || !k_tail || !v_tail || !out) return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_cand < 1 || d->cand_len < 1 || d->hq < 1 || d->hkv < 1 ||
      d->max_prefix < 0 || d->total_prefix < 0 || d->flags != 0)
    return FVRAG_ERR_INVALID_ARG;
  if (d->total_prefix > 0 && (!k_prefix || !v_prefix)) return FVRAG_ERR_INVALID_ARG;
  if (d->hq % d->hkv != 0 || (d->head_dim != 64 && d->head_dim != 128) ||
      d->cand_len > kMaxTail || d->hq / d->hkv > kRowsPerTile)
    return FVRAG_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k_tail) || !aligned16(v_tail) || !aligned16(out) ||
      (k_prefix && !aligned16(k_prefix)) || (v_prefix && !aligned16(v_prefix)))
    return FVRAG_ERR_MISALIGNED;
  const size_t need = ws_bytes(d);
  if (!ws || ws_size < need) return FVRAG_ERR_WORKSPACE;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;

  const Plan p = make_plan(d);
  const int D = d->head_dim;
  const float scale = d->softmax_scale != 0.f ? d->softmax_scale : 1.f / sqrtf((float)D);
  const int KL = d->num_cand * d->cand_len;
  uint8_t* base = reinterpret_cast<uint8_t*>(ws);
  uint32_t* status = reinterpret_cast<uint32_t*>(base);
  const size_t nrows = (size_t)d->num_queries * KL * d->hq;
  float* part_o = reinterpret_cast<float*>(base + kWsHeaderBytes);
  float* part_lse = part_o + (size_t)p.nsplit * nrows * D;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  const bool run_prefix = p.nsplit > 0 && d->total_prefix > 0;
  if (run_prefix) {
    CUtensorMap tq, tk, tv;
    {
      const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d->hq, (uint64_t)d->num_queries * KL};
      const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d->hq * D * 2};
      const uint32_t box[3] = {64u, (uint32_t)p.grp, (uint32_t)p.T};
      if (!encode_tmap_bf16(&tq, q, 3, dims, strides, box, true)) return FVRAG_ERR_CUDA;
    }
    {
      const uint64_t dims[3] = {(uint64_t)D, (uint64_t)d->hkv, (uint64_t)d->total_prefix};
      const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)d->hkv * D * 2};
      const uint32_t box[3] = {64u, 1u, (uint32_t)kKeysPerBlock};
      if (!encode_tmap_bf16(&tk, k_prefix, 3, dims, strides, box, true)) return FVRAG_ERR_CUDA;
      if (!encode_tmap_bf16(&tv, v_prefix, 3, dims, strides, box, true)) return FVRAG_ERR_CUDA;
    }
    PrefixArgs a;
    a.offs = prefix_offsets;
    a.part_o = part_o;
    a.part_lse = part_lse;
    a.status = status;
    a.limit_ns = wait_limit_ns();
    a.Qn = d->num_queries;
    a.KL = KL;
    a.hq = d->hq;
    a.hkv = d->hkv;
    a.grp = p.grp;
    a.T = p.T;
    a.mtiles = p.mtiles;
    a.nsplit = p.nsplit;
    a.chunk = p.chunk;
    a.scale_log2 = scale * kLog2e;
    const long long grid = (long long)d->num_queries * d->hkv * p.nsplit * p.mtiles;
    if (grid > 0x7fffffffLL) return FVRAG_ERR_UNSUPPORTED;
    if (D == 128) {
      const size_t sm = smem_bytes<128>();
      if (cudaFuncSetAttribute(prefix_attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)sm) != cudaSuccess)
        return FVRAG_ERR_CUDA;
      prefix_attn_kernel<128><<<(unsigned)grid, kThreads, sm, s>>>(tq, tk, tv, a);
    } else {
      const size_t sm = smem_bytes<64>();
      if (cudaFuncSetAttribute(prefix_attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)sm) != cudaSuccess)
        return FVRAG_ERR_CUDA;
      prefix_attn_kernel<64><<<(unsigned)grid, kThreads, sm, s>>>(tq, tk, tv, a);
    }
    if (cudaGetLastError() != cudaSuccess) return FVRAG_ERR_CUDA;
  }
  const int nsplit = run_prefix ? p.nsplit : 0;
  const int warps_per_block = 8;
  const long long blocks = ((long long)nrows + warps_per_block - 1) / warps_per_block;
  if (D == 128)
    tail_merge_kernel<128><<<(unsigned)blocks, 32 * warps_per_block, 0, s>>>(
        reinterpret_cast<const __nv_bfloat16*>(q), reinterpret_cast<const __nv_bfloat16*>(k_tail),
        reinterpret_cast<const __nv_bfloat16*>(v_tail), part_o, part_lse, nsplit, d->num_queries,
        d->num_cand, d->cand_len, d->hq, d->hkv, scale, reinterpret_cast<__nv_bfloat16*>(out), lse);
  else
    tail_merge_kernel<64><<<(unsigned)blocks, 32 * warps_per_block, 0, s>>>(
        reinterpret_cast<const __nv_bfloat16*>(q), reinterpret_cast<const __nv_bfloat16*>(k_tail),
        reinterpret_cast<const __nv_bfloat16*>(v_tail), part_o, part_lse, nsplit, d->num_queries,
        d->num_cand, d->cand_len, d->hq, d->hkv, scale, reinterpret_cast<__nv_bfloat16*>(out), lse);
  return launch_status();
}
