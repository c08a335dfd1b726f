// K1: one attention layer of the verifier forward over all candidate rows
// (Eq. 6 / Eq. 11): token l of candidate k attends to the P_q tokens of the
// shared prefix and to tokens 0..l of its own candidate.  The same kernel runs
// one decode step of the drafts (Eq. 5, Eq. 8-10): the newest token of each
// draft attends to the shared prefix and to the draft's own cached tokens.
//
// General form: every candidate owns C own-token slots of which the first n_k
// are valid, and its Lq query tokens are the last Lq of those n_k (query l sits
// at slot n_k - Lq + l and sees own slots 0 .. n_k - Lq + l).  Verification is
// Lq = C = n_k = L; a decode step is Lq = 1 with n_k read from the device.
//
// The prefix (up to 32768 keys) is shared by every candidate row, so all
// query rows that use one KV head are packed into the rows of the tensor-core
// tiles (GQA packing): a row tile is T query tokens x the hq/hkv query heads of
// one KV head (T = floor(128 / (hq/hkv))), and every prefix K/V block that a
// CTA loads feeds all of them.
//
// Key blocks of 128: the query's prefix blocks, then the blocks of the tile's
// candidates' own slots (concatenated) that hold at least one valid slot.  The
// list is cut into equal runs of blocks, one run per CTA (split-KV): the same
// number of runs for every tile when the tiles' lists are alike (verification),
// or, when their lengths differ with data known only on the device (decode: n_k),
// runs of one length R for all tiles, chosen so that all runs fit one grid of CTAs;
// every CTA makes that plan in its prologue and takes its own (tile, run).
//
// attn_kernel: one CTA = one row tile x one run of key blocks.
//   warp 0     TMA: the Q tile once (3-D map over [tokens][hq][D]), then K and V
//              blocks (3-D maps over [keys][hkv][D], 128-byte swizzle) into a 2-deep
//              K ring and a 3-deep V ring, in block order, each once its slot is free.
//              Warps 0 and 1 wait with blocking mbarrier waits in a fixed order, so they
//              take no issue slots from the softmax warps on their sub-partitions.
//   warp 1     allocates tensor memory and issues the PV tcgen05.mma:
//                O   += P_j V_j   (M = 128, N = D, K = 128 keys; P_j read from tensor
//                                  memory, V MN-major from shared memory)
//   warp 10    issues the S tcgen05.mma:
//                S_j  = Q K_j^T   (M = 128 rows, N = 128 keys, K = D; both K-major)
//              into three S/P buffers; O accumulates in tensor memory.  Two issuing
//              threads keep the tensor pipe fed: S_{j+3} waits for PV_j to finish
//              (it overwrites P_j) while PV_{j+1} is already queued.
//   warps 2-9  two warps per tensor-memory lane quarter, one query row per thread and
//              half of the block's keys per warp: tcgen05.ld of S_j, masking (prefix
//              length, or the row's own visible slots; full blocks skip it), online
//              softmax in base 2 against a lazily moved reference max (O and l are
//              rescaled in place only when a row's max grows by more than 2^8; the block
//              max is only computed, and shared by the two halves through shared memory,
//              when a row has no reference yet or a partial sum shows a term past that
//              limit), and P_j written back as bf16 pairs over S_j in tensor memory.
//   One run: the CTA writes the bf16 output and the lse directly.  Several runs:
//   normalised partials go to the workspace (fp16: the outputs are convex combinations
//   of V rows, so 11 mantissa bits keep them well inside the bf16 output's rounding) and
//   merge_kernel combines them with
//   log-sum-exp weights.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <cmath>
#include <type_traits>

#include "fvrag_common.cuh"
#include "fvrag_internal.h"

namespace fvrag {
namespace attn {

constexpr int kThreads = 352;      // producer, PV issuer, 8 softmax warps, S issuer
constexpr int kWarpS = 10;         // the warp whose lane 0 issues the S MMAs
constexpr int kBM = 128;          // query rows per tile (MMA M)
constexpr int kBN = 128;          // keys per block (MMA N of S, K of PV)
constexpr int kKStages = 2;       // depth of the K ring (K_j is consumed early, by S_j)
constexpr int kVStages = 3;       // depth of the V ring (V_j is read by PV_j, after softmax_j)
constexpr int kMaxTail = 64;            // verification: tokens per candidate
constexpr int kMaxCand = kBM + 1;       // candidates a row tile can touch
constexpr uint32_t kTmemCols = 512;
// tensor-memory columns: kSP S/P buffers of 128 columns (S_j as fp32 in 128 columns, then
// P_j as packed bf16: keys 0-63 in columns 0-31, keys 64-127 in columns 64-95, each half over
// the S columns its own softmax warp has read), the O accumulator after them.  Three buffers let
// S_{j+2} be computed while PV_j still reads P_j.
constexpr int kSP = 3;
__device__ __forceinline__ uint32_t col_s(int b) { return (uint32_t)b * 128u; }
constexpr uint32_t kColO = kSP * 128;
static_assert(kColO + 128 <= kTmemCols, "S/P buffers and O must fit in tensor memory");
constexpr float kRescaleLog2 = 8.f;   // lazy-rescale threshold (P stays < 2^8)
constexpr float kSumLimit = 256.f;    // 2^kRescaleLog2: a partial sum above it may hold a term past the limit
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// balanced plan (see plan_run): shared-memory capacity
constexpr int kMaxPlanTiles = 1024;   // tiles the plan holds in shared memory
constexpr int kMaxPlanQueries = 1024; // queries whose offsets it stages
constexpr int kMaxPlanOwn = 2048;     // Qn * K own lengths it stages
constexpr int kMaxRuns = 64;          // runs of one tile that merge_kernel combines
constexpr int kPlanScratch = 256;     // reduction and control words
constexpr int kMaxStreamQueries = 64; // streamed plan: queries and row tiles per KV head
constexpr int kMaxStreamMtiles = 64;  // whose prefix sums it keeps in shared memory
constexpr int kStreamPlanBytes = 1024;
constexpr int kPlanInts = kPlanScratch + kMaxPlanTiles + kMaxPlanQueries + 4 + kMaxPlanOwn;

enum : uint32_t { kSiteQ = 0x101, kSiteMma = 0x102, kSiteProducer = 0x103, kSiteSFull = 0x107,
                  kSitePvDone = 0x109, kSiteDrain = 0x10A, kSitePlan = 0x10B };

template <int D>
struct Layout {
  static constexpr int NH = D / 64;                 // 128-byte column halves of a row
  static constexpr int kQ = NH * kBM * 128;         // Q tile
  static constexpr int kKVHalf = kBN * 128;         // 128 keys x 64 elements
  static constexpr int kStage = NH * kKVHalf;       // one K block or one V block
  // + row-max exchange [2 slots][2 halves][128 rows], row-sum exchange [2][128] floats and
  // the slow-path flags [2 slots][2 halves][4 quarters]
  static constexpr int kBytes =
      kQ + (kKStages + kVStages) * kStage + 1024 + 256 + kMaxCand * 4 + 6 * kBM * 4 + 64 +
      kStreamPlanBytes;
  static_assert(kPlanInts * 4 <= kVStages * kStage, "plan scratch fits the V ring");
  static_assert(kBytes <= 232448, "shared memory per CTA");
};

struct Args {
  int2* tile_runs;         // balanced plan: [tiles] {first slot, runs}, written here; or null
  const int32_t* offs;
  const int32_t* own_len;  // [Qn][K] valid own slots n_k, or null (n_k = C)
  __nv_bfloat16* out;     // final output (one split)
  float* lse;             // final lse (one split), may be null
  __half* part_o;         // [nsplit][rows][D] fp16 (several splits)
  float* part_lse;        // [nsplit][rows]
  uint32_t* status;
  uint64_t limit_ns;
  int Qn, K, Lq, C, KL, hq, hkv, grp, T, mtiles, nsplit;
  int slot_rows;           // balanced and streamed plans: rows per partial slot (T * grp)
  int maxparts;            // streamed plan: partial slots per tile
  float scale_log2;
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed pairs of fp32 (the sm_100 family's two-lane FMA / ADD) and a three-input max:
// the softmax issues half as many FMA, ADD and MAX instructions per key.
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}

__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}

__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

// Makes this thread's generic-proxy shared-memory writes visible to the async
// proxy (the tensor cores read Q from shared memory).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// MN-major operand with the 128-byte swizzle (V read as B of O = P V, N = D
// contiguous in memory): 64-element MN chunks `lbo` bytes apart (leading
// byte offset), 8-row K groups 1024 B apart (stride byte offset).
__device__ __forceinline__ uint64_t desc_mnmajor_sw128(uint32_t smem_addr, uint32_t lbo) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo & 0x3FFFFu) >> 4) << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// ---------------------------------------------------------------------------
// Balanced plan, for tiles whose block lists differ in length by data on the device
// (decode: n_k).  Every CTA of the grid makes the same plan from the same inputs in its
// prologue: the smallest run length R (in blocks) such that the runs of all tiles,
// ns_t = max(1, ceil(nb_t / R)) each, fit in the grid (and ns_t <= kMaxRuns); tile t's
// list is cut into ns_t equal runs held by consecutive CTAs.

// Length of tile t's block list: its query's prefix blocks plus the own blocks that hold a
// valid slot, i.e. the union over its candidates c with n_c > 0 of the blocks
// [c C / 128, (c C + n_c - 1) / 128] (the count the kernel makes with own_valid).
// offs_s and own_s are the prefix offsets and own lengths staged in shared memory.
__device__ int tile_blocks(const Args& a, const int* offs_s, const int* own_s, int t) {
  const int mt = t % a.mtiles;
  const int qi = t / a.mtiles / a.hkv;
  const int P = max(0, offs_s[qi + 1] - offs_s[qi]);
  int nb = (P + kBN - 1) / kBN;
  const int tok0 = mt * a.T;
  const int ntok = min(a.T, a.KL - tok0);
  const int c_lo = tok0 / a.Lq;
  const int ncand = (tok0 + ntok - 1) / a.Lq - c_lo + 1;
  int last = -1;                                  // highest own block counted so far
  for (int c = 0; c < ncand; ++c) {
    int n = a.own_len ? own_s[qi * a.K + c_lo + c] : a.C;
    n = n < 0 ? 0 : (n > a.C ? a.C : n);
    if (n == 0) continue;
    const int lo = (c * a.C) / kBN, hi = (c * a.C + n - 1) / kBN;
    if (hi > last) {
      nb += hi - max(lo, last + 1) + 1;
      last = hi;
    }
  }
  return nb;
}

// Called by all NT threads of the CTA.  Returns this CTA's run {tile, first block, blocks,
// 1 if the tile has a single run}, or tile -1 when the plan leaves the CTA idle; the CTA
// holding a tile's first run records {first slot (CTA), runs} of the tile for the merge.
template <int NT>
__device__ int4 plan_run(const Args& a, int* ps) {
  constexpr int NW = NT / 32;
  long long* red_sum = reinterpret_cast<long long*>(ps);   // [NW]
  int* red_max = ps + 64;
  int* red_r = ps + 96;
  int* red_ok = ps + 128;
  int* scan_s = ps + 160;
  int* ctl = ps + 192;             // [0], [1] search range of R; [2..5] this CTA's run
  int* nb_s = ps + kPlanScratch;
  int* offs_s = nb_s + kMaxPlanTiles;
  int* own_s = offs_s + kMaxPlanQueries + 4;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ntiles = a.Qn * a.hkv * a.mtiles;
  for (int i = tid; i <= a.Qn; i += NT) offs_s[i] = __ldg(&a.offs[i]);
  if (a.own_len)
    for (int i = tid; i < a.Qn * a.K; i += NT) own_s[i] = __ldg(&a.own_len[i]);
  if (tid == 0) ctl[2] = -1;
  __syncthreads();
  long long sum = 0;
  int mx = 0;
  for (int t = tid; t < ntiles; t += NT) {
    const int nb = tile_blocks(a, offs_s, own_s, t);
    nb_s[t] = nb;
    sum += nb;
    mx = max(mx, nb);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sum += __shfl_xor_sync(0xffffffffu, sum, o);
    mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == 0) {
    red_sum[warp] = sum;
    red_max[warp] = mx;
  }
  __syncthreads();
  if (tid == 0) {
    long long total = 0;
    int m = 0;
    for (int w = 0; w < NW; ++w) {
      total += red_sum[w];
      m = max(m, red_max[w]);
    }
    // any R >= total / (grid - tiles) fits: the run count is at most total / R + tiles
    const int rmin = max(1, (m + kMaxRuns - 1) / kMaxRuns);
    const long long slack = (long long)gridDim.x - ntiles;
    ctl[0] = rmin;
    ctl[1] = (int)max((long long)rmin, (total + slack - 1) / slack);
  }
  __syncthreads();
  // NW-ary search: warp w tests R_w = lo + (hi - lo) w / (NW - 1) (R_{NW-1} = hi fits)
  while (ctl[0] < ctl[1]) {
    const int lo = ctl[0], hi = ctl[1];
    const int rw = lo + (int)((long long)(hi - lo) * warp / (NW - 1));
    long long cnt = 0;
    for (int t = lane; t < ntiles; t += 32) cnt += max(1, (nb_s[t] + rw - 1) / rw);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
    if (lane == 0) {
      red_r[warp] = rw;
      red_ok[warp] = cnt <= (long long)gridDim.x;
    }
    __syncthreads();
    if (tid == 0) {
      int w = 0;
      while (!red_ok[w]) ++w;
      ctl[0] = w > 0 ? red_r[w - 1] + 1 : lo;
      ctl[1] = red_r[w];
    }
    __syncthreads();
  }
  const int R = ctl[1];
  // runs per tile over a contiguous chunk of tiles per thread; exclusive scan of the counts
  const int per = (ntiles + NT - 1) / NT;
  const int t0 = min(ntiles, tid * per), t1 = min(ntiles, t0 + per);
  int local = 0;
  for (int t = t0; t < t1; ++t) local += max(1, (nb_s[t] + R - 1) / R);
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) scan_s[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int v = lane < NW ? scan_s[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int u = __shfl_up_sync(0xffffffffu, v, o);
      if (lane >= o) v += u;
    }
    if (lane < NW) scan_s[lane] = v;   // inclusive over warps
  }
  __syncthreads();
  int start = incl - local + (warp > 0 ? scan_s[warp - 1] : 0);
  const int b = blockIdx.x;
  for (int t = t0; t < t1; ++t) {
    const int nb = nb_s[t];
    const int ns = max(1, (nb + R - 1) / R);
    if (b >= start && b < start + ns) {
      const int bps = (nb + ns - 1) / ns;
      const int lo = (b - start) * bps;
      ctl[2] = t;
      ctl[3] = lo;
      ctl[4] = max(0, min(nb, lo + bps) - lo);
      ctl[5] = ns == 1 ? 1 : 0;
      if (b == start) a.tile_runs[t] = make_int2(start, ns);
    }
    start += ns;
  }
  __syncthreads();
  return make_int4(ctl[2], ctl[3], ctl[4], ctl[5]);
}

// ---------------------------------------------------------------------------
// Streamed plan (verification, own lengths all C).  The block lists of all tiles, in tile
// order (query, KV head, row tile), form one sequence of W blocks; CTA c takes the blocks
// [c W / grid, (c + 1) W / grid): the tail of one tile, whole tiles and the head of another,
// run as consecutive segments in one pass of its pipelines.  Every SM then does the same
// number of blocks (to within one) in a single wave, whatever the number of tiles, and pays
// the pipeline fill once.  A tile cut between CTAs leaves one normalised partial per CTA in
// slots [t * maxparts, t * maxparts + parts) of the balanced plan's layout, merged by
// merge_kernel; a tile that lies inside one CTA's range is written directly.
//
// The sequence position of tile t (query qi, KV head g, row tile mt) is closed-form:
// tile t has npb(qi) prefix blocks and ntb(mt) own blocks, so with the prefix sums qcum over
// queries and tcum over row tiles (NTB = tcum[mtiles]),
//   G0(t) = hkv (mtiles qcum[qi] + qi NTB) + g (mtiles npb(qi) + NTB) + mt npb(qi) + tcum[mt].
struct StreamPlan {
  long long W;                         // blocks in all
  int t0;                              // first tile of this CTA's range
  int qcum[kMaxStreamQueries + 1];
  int npb[kMaxStreamQueries];
  int tcum[kMaxStreamMtiles + 1];
};
static_assert(sizeof(StreamPlan) + 16 <= kStreamPlanBytes, "the streamed plan fits its space");

// Own blocks of row tile mt: the 128-key blocks over its candidates' C slots each.
__device__ __forceinline__ int tile_own_blocks(const Args& a, int mt) {
  const int tok0 = mt * a.T;
  const int ntok = min(a.T, a.KL - tok0);
  const int c_lo = tok0 / a.Lq;
  const int ncand = (tok0 + ntok - 1) / a.Lq - c_lo + 1;
  return (ncand * a.C + kBN - 1) / kBN;
}

__device__ __forceinline__ long long stream_g0(const Args& a, const StreamPlan& sp, int t) {
  if (t >= a.Qn * a.hkv * a.mtiles) return sp.W;
  const int mt = t % a.mtiles;
  const int g = (t / a.mtiles) % a.hkv;
  const int qi = t / a.mtiles / a.hkv;
  const long long ntb_all = sp.tcum[a.mtiles];
  return (long long)a.hkv * ((long long)a.mtiles * sp.qcum[qi] + (long long)qi * ntb_all) +
         (long long)g * ((long long)a.mtiles * sp.npb[qi] + ntb_all) +
         (long long)mt * sp.npb[qi] + sp.tcum[mt];
}

// The CTA whose range holds sequence position x: the largest c with c W / grid <= x.
__device__ __forceinline__ int stream_cta(long long x, long long W, int grid) {
  return (int)(((x + 1) * grid + W - 1) / W) - 1;
}

// One contiguous run of a tile's block list that a CTA processes.
struct Seg {
  int t;            // tile
  int blk_lo;       // first block of the tile's list
  int nblk;         // blocks
  bool direct;      // the run is the whole list: the CTA writes the output itself
  int pslot;        // partial slot (runs that are not direct), or the static plan's split
};

// MODE 0: static split (verification: tile x nsplit runs, one per CTA); 1: balanced plan
// (decode: runs fitted on the device into one grid); 2: streamed plan (verification: a
// share of the concatenated block lists per CTA).  Separate instantiations keep each plan's
// code out of the other kernels.
template <int D, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kp,
                const __grid_constant__ CUtensorMap tm_vp, const __grid_constant__ CUtensorMap tm_kt,
                const __grid_constant__ CUtensorMap tm_vt, const Args a) {
  constexpr bool BAL = MODE == 1, STREAM = MODE == 2;
  using Lay = Layout<D>;
  constexpr int NH = Lay::NH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* q_s = smem;
  uint8_t* k_ring = q_s + Lay::kQ;                     // [kKStages][kStage]
  uint8_t* v_ring = k_ring + kKStages * Lay::kStage;   // [kVStages][kStage]
  float* xmax = reinterpret_cast<float*>(v_ring + kVStages * Lay::kStage);  // [2][2][kBM]
  float* xsum = xmax + 4 * kBM;                                             // [2][kBM]
  int* xflag = reinterpret_cast<int*>(xsum + 2 * kBM);                      // [2][2][4]
  uint64_t* bars = reinterpret_cast<uint64_t*>(xflag + 16);
  uint64_t* k_full = bars;                        // [kKStages]  TMA -> MMA
  uint64_t* k_empty = bars + kKStages;            // [kKStages]  MMA (S done) -> TMA
  uint64_t* v_full = k_empty + kKStages;          // [kVStages]  TMA -> MMA
  uint64_t* v_empty = v_full + kVStages;          // [kVStages]  MMA (PV done) -> TMA
  uint64_t* s_full = v_empty + kVStages;          // [kSP]  S_j in tensor memory
  uint64_t* p_full = s_full + kSP;                // [kSP]  P_j in tensor memory (4 warps)
  uint64_t* pv_done = s_full + 2 * kSP;           // [kSP]  PV_j done: S/P buffer free
  uint64_t* q_full = s_full + 3 * kSP;            // the segment's Q tile is in
  uint64_t* drain = q_full + 1;                   // every PV MMA done
  uint64_t* drain_s = drain + 1;                  // every S MMA done
  uint64_t* q_empty = drain_s + 1;                // the segment's S MMAs are done: Q may be reloaded
  uint64_t* o_free = q_empty + 1;                 // the softmax warps have read the segment's O
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(o_free + 1);
  // valid own slots of the tile's candidates (single-segment plans; the own blocks with
  // none are skipped)
  int* n_own = reinterpret_cast<int*>(o_free + 1) + 4;
  StreamPlan* sp = reinterpret_cast<StreamPlan*>(
      (reinterpret_cast<uintptr_t>(n_own + kMaxCand) + 15) & ~uintptr_t(15));

  griddep_wait();                 // inputs may come from the previous kernel
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // ---- work: one run (static, balanced plans) or this CTA's share of the sequence
  Seg seg0 = {0, 0, 0, false, 0};
  int4 wk = make_int4(0, 0, 0, 0);
  if constexpr (BAL) {
    // the plan's scratch is the V ring, whose first writer is the TMA after the prologue
    wk = plan_run<kThreads>(a, reinterpret_cast<int*>(v_ring));
    fence_proxy_async_smem();
    if (wk.x < 0) return;         // the plan left this CTA without a run
    seg0.t = wk.x;
  } else if constexpr (!STREAM) {
    int b = blockIdx.x;
    const int mt = b % a.mtiles;
    b /= a.mtiles;
    seg0.pslot = b % a.nsplit;    // the split
    b /= a.nsplit;
    seg0.t = b * a.mtiles + mt;   // (qi, g) then mt
  } else {
    const int ntiles = a.Qn * a.hkv * a.mtiles;
    for (int i = threadIdx.x; i < a.Qn; i += kThreads)
      sp->npb[i] = (max(0, __ldg(&a.offs[i + 1]) - __ldg(&a.offs[i])) + kBN - 1) / kBN;
    for (int i = threadIdx.x; i < a.mtiles; i += kThreads) sp->tcum[i + 1] = tile_own_blocks(a, i);
    __syncthreads();
    if (threadIdx.x == 0) {
      sp->qcum[0] = 0;
      for (int i = 0; i < a.Qn; ++i) sp->qcum[i + 1] = sp->qcum[i] + sp->npb[i];
      sp->tcum[0] = 0;
      for (int i = 0; i < a.mtiles; ++i) sp->tcum[i + 1] += sp->tcum[i];
      sp->W = (long long)a.hkv *
              ((long long)a.mtiles * sp->qcum[a.Qn] + (long long)a.Qn * sp->tcum[a.mtiles]);
      const long long W = sp->W, grid = gridDim.x;
      const long long x0 = (long long)blockIdx.x * W / grid, x1 = ((long long)blockIdx.x + 1) * W / grid;
      // first tile whose list reaches past x0
      int lo = 0, hi = ntiles;            // G0(lo) <= x0 < G0(hi)
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (stream_g0(a, *sp, mid) <= x0) lo = mid; else hi = mid;
      }
      sp->t0 = lo;
      // record {first slot, runs} of every tile whose first block lies in this range
      for (int t = lo; t < ntiles; ++t) {
        const long long g0 = stream_g0(a, *sp, t);
        if (g0 >= x1) break;
        if (g0 < x0) continue;
        const long long g1 = stream_g0(a, *sp, t + 1);
        const int parts = g1 > g0 ? stream_cta(g1 - 1, W, (int)grid) - stream_cta(g0, W, (int)grid) + 1 : 1;
        a.tile_runs[t] = make_int2(t * a.maxparts, parts);
      }
    }
  }
  // segment s of this CTA (s = 0 only for the static and balanced plans); false past the last
  auto segment = [&](int s, Seg& sg) -> bool {
    if constexpr (!STREAM) {
      if (s > 0) return false;
      sg = seg0;
      return true;
    } else {
      const int ntiles = a.Qn * a.hkv * a.mtiles;
      const long long W = sp->W, grid = gridDim.x;
      const long long x0 = (long long)blockIdx.x * W / grid, x1 = ((long long)blockIdx.x + 1) * W / grid;
      const int t = sp->t0 + s;
      if (t >= ntiles) return false;
      const long long g0 = stream_g0(a, *sp, t);
      if (g0 >= x1) return false;
      const long long g1 = stream_g0(a, *sp, t + 1);
      const long long lo = max(x0, g0), hi = min(x1, g1);
      if (hi <= lo) return false;   // an empty range (more CTAs than blocks)
      sg.t = t;
      sg.blk_lo = (int)(lo - g0);
      sg.nblk = (int)max(0LL, hi - lo);
      const int cf = stream_cta(g0, W, (int)grid);
      const int parts = g1 > g0 ? stream_cta(g1 - 1, W, (int)grid) - cf + 1 : 1;
      sg.direct = parts == 1;
      const int part = (int)blockIdx.x - cf;
      sg.pslot = part < a.maxparts ? t * a.maxparts + part : -1;   // -1: no room (bad plan)
      return true;
    }
  };
  // the tile a segment covers
  struct TileInfo {
    int mt, g, qi, P, nbp, tok0, ntok, rows, c_lo, ncand, ntb;
  };
  auto tile_info = [&](int t) {
    TileInfo ti;
    ti.mt = t % a.mtiles;
    ti.g = (t / a.mtiles) % a.hkv;
    ti.qi = t / a.mtiles / a.hkv;
    ti.P = max(0, __ldg(&a.offs[ti.qi + 1]) - __ldg(&a.offs[ti.qi]));
    ti.nbp = (ti.P + kBN - 1) / kBN;               // prefix blocks of this query
    ti.tok0 = ti.mt * a.T;
    ti.ntok = min(a.T, a.KL - ti.tok0);
    ti.rows = ti.ntok * a.grp;
    ti.c_lo = ti.tok0 / a.Lq;
    ti.ncand = (ti.tok0 + ti.ntok - 1) / a.Lq - ti.c_lo + 1;
    ti.ntb = (ti.ncand * a.C + kBN - 1) / kBN;     // blocks over the candidates' own slots
    return ti;
  };

  if constexpr (!STREAM) {
    const TileInfo ti = tile_info(seg0.t);
    for (int c = threadIdx.x; c < ti.ncand; c += kThreads) {
      int n = a.own_len ? __ldg(&a.own_len[ti.qi * a.K + ti.c_lo + c]) : a.C;
      n_own[c] = n < 0 ? 0 : (n > a.C ? a.C : n);
    }
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < kKStages; ++s) {
      mbar_init(smem_u32(&k_full[s]), 1);
      mbar_init(smem_u32(&k_empty[s]), 1);
    }
    for (int s = 0; s < kVStages; ++s) {
      mbar_init(smem_u32(&v_full[s]), 1);
      mbar_init(smem_u32(&v_empty[s]), 1);
    }
    for (int s = 0; s < kSP; ++s) {
      mbar_init(smem_u32(&s_full[s]), 1);
      mbar_init(smem_u32(&p_full[s]), 8);   // one arrival per softmax warp
      mbar_init(smem_u32(&pv_done[s]), 1);
    }
    mbar_init(smem_u32(q_full), 1);
    mbar_init(smem_u32(drain), 1);
    mbar_init(smem_u32(drain_s), 1);
    mbar_init(smem_u32(q_empty), 1);
    mbar_init(smem_u32(o_free), 8);         // one arrival per softmax warp
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_holder), kTmemCols);
    tmem_relinquish();
  }
  if (warp >= 2 && warp < 6) {
    // Rows past the T x grp rows the Q box fills are never loaded: zero them so their
    // (discarded) scores stay finite and every lane of a warp takes the same code path.
    const int r = (warp & 3) * 32 + lane;
    if (r >= a.T * a.grp) {
      for (int h = 0; h < NH; ++h)
        for (int c = 0; c < 8; ++c)
          st_shared_v4(smem_u32(q_s + h * kBM * 128 + r * 128 + c * 16), 0u, 0u, 0u, 0u);
      fence_proxy_async_smem();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;
  // own block tb of a tile holds a valid slot when some candidate c it overlaps has n_c > 0
  // and c * C + n_c > tb * kBN (each candidate's valid slots are its first n_c); under the
  // streamed plan every candidate has C valid slots, so every own block does
  auto own_valid = [&](const TileInfo& ti, int tb) {
    if constexpr (STREAM) {
      return tb < ti.ntb;
    } else {
      const int s0 = tb * kBN;
      const int s1 = min(s0 + kBN, ti.ncand * a.C);
      for (int c = s0 / a.C; c * a.C < s1; ++c)
        if (n_own[c] > 0 && c * a.C + n_own[c] > s0) return true;
      return false;
    }
  };
  auto own_next = [&](const TileInfo& ti, int tb) {   // first valid own block >= tb
    while (tb < ti.ntb && !own_valid(ti, tb)) ++tb;
    return tb;
  };
  // Single-run plans: every warp computes the run and its first own block (the valid own
  // blocks of earlier runs of the tile are skipped) with the same warp votes.  The static
  // split cuts the tile's list of nb blocks into nsplit equal runs here; the balanced plan
  // fixed the run already.  The streamed plan's segments carry their runs, and every own
  // block is valid there.
  int tb_first0 = 0;
  if constexpr (!STREAM) {
    const TileInfo ti = tile_info(seg0.t);
    int nvt = 0;
    for (int base = 0; base < ti.ntb; base += 32)
      nvt += __popc(__ballot_sync(0xffffffffu, base + lane < ti.ntb && own_valid(ti, base + lane)));
    const int nb = ti.nbp + nvt;
    if constexpr (BAL) {            // plan_run counted the same nb for this tile
      seg0.blk_lo = wk.y;
      seg0.nblk = wk.z;
      seg0.direct = wk.w != 0;
      seg0.pslot = blockIdx.x;
    } else {
      const int bps = (nb + a.nsplit - 1) / a.nsplit;
      seg0.blk_lo = seg0.pslot * bps;
      seg0.nblk = max(0, min(nb, seg0.blk_lo + bps) - seg0.blk_lo);
      seg0.direct = a.nsplit == 1;
    }
    tb_first0 = ti.ntb;
    int skip = max(0, seg0.blk_lo - ti.nbp);
    for (int base = 0; base < ti.ntb; base += 32) {
      const uint32_t m = __ballot_sync(0xffffffffu, base + lane < ti.ntb && own_valid(ti, base + lane));
      const int cnt = __popc(m);
      if (skip < cnt) {
        uint32_t mm = m;
        for (int i = 0; i < skip; ++i) mm &= mm - 1u;
        tb_first0 = base + __ffs(mm) - 1;
        break;
      }
      skip -= cnt;
    }
  }
  auto first_own = [&](const TileInfo& ti, const Seg& sg) {
    return STREAM ? max(0, sg.blk_lo - ti.nbp) : tb_first0;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // Per segment: its Q tile (once the previous segment's S MMAs are done with the last
    // one), then K_0, V_0, K_1, V_1, ... (K is recycled after its S MMA, V after its PV MMA).
    // The rings and their phases run on over the CTA's whole sequence of blocks.
    Seg sg;
    int nk = 0, nv = 0, nq = 0;
    bool fine = true;
    for (int s = 0; fine && segment(s, sg); ++s) {
      if (lane != 0 || sg.nblk == 0) continue;
      const TileInfo ti = tile_info(sg.t);
      const int tb_first = first_own(ti, sg);
      const uint64_t pol_kv = policy_evict_last();   // re-read by the other row tiles
      const uint64_t pol_q = policy_evict_first();
      const uint32_t qb = smem_u32(q_full);
      if (nq > 0 && !mbar_wait(smem_u32(q_empty), (nq - 1) & 1, a.limit_ns)) {
        fine = false;
        break;
      }
      mbar_arrive_expect_tx(qb, NH * a.grp * a.T * 128);
      for (int h = 0; h < NH; ++h)
        tma_load_3d(smem_u32(q_s + h * kBM * 128), &tm_q, qb, h * 64, ti.g * a.grp,
                    ti.qi * a.KL + ti.tok0, pol_q);
      ++nq;
      const int pbase = __ldg(&a.offs[ti.qi]);
      const int tbase = (ti.qi * a.K + ti.c_lo) * a.C;   // own slot 0 of candidate c_lo
      int tbk = tb_first, tbv = tb_first;               // own-block cursors of the two rings
      // Fixed order K_j, V_j with blocking waits (the waiting thread takes no issue slots
      // from the softmax warps on its sub-partition): K_j's slot frees when S_{j-2} is done,
      // V_j's when PV_{j-3} is done, both well before the block is needed.
      auto load = [&](bool is_v, int jj, int j, int& tb) {
        const uint32_t fb = smem_u32(is_v ? &v_full[jj % kVStages] : &k_full[jj % kKStages]);
        mbar_arrive_expect_tx(fb, Lay::kStage);
        uint8_t* dst = is_v ? v_ring + (jj % kVStages) * Lay::kStage : k_ring + (jj % kKStages) * Lay::kStage;
        const int bi = sg.blk_lo + j;
        const bool pre = bi < ti.nbp;
        int key;
        if (pre) {
          key = pbase + bi * kBN;
        } else {
          tb = own_next(ti, tb);
          key = tbase + tb * kBN;
          ++tb;
        }
        const CUtensorMap* tm = is_v ? (pre ? &tm_vp : &tm_vt) : (pre ? &tm_kp : &tm_kt);
        for (int h = 0; h < NH; ++h)
          tma_load_3d(smem_u32(dst + h * Lay::kKVHalf), tm, fb, h * 64, ti.g, key, pol_kv);
      };
      for (int j = 0; j < sg.nblk; ++j) {
        if (!mbar_wait(smem_u32(&k_empty[nk % kKStages]), ((nk / kKStages) & 1) ^ 1, a.limit_ns)) {
          fine = false;
          break;
        }
        load(false, nk, j, tbk);
        ++nk;
        if (!mbar_wait(smem_u32(&v_empty[nv % kVStages]), ((nv / kVStages) & 1) ^ 1, a.limit_ns)) {
          fine = false;
          break;
        }
        load(true, nv, j, tbv);
        ++nv;
      }
    }
    if (lane == 0) {
      if (!fine) record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteProducer);
      // no copy may still be in flight when the CTA exits
      if (nq > 0) mbar_wait(smem_u32(q_full), (nq - 1) & 1, a.limit_ns);
      for (int i = max(0, nk - kKStages); i < nk; ++i)
        mbar_wait(smem_u32(&k_full[i % kKStages]), (i / kKStages) & 1, a.limit_ns);
      for (int i = max(0, nv - kVStages); i < nv; ++i)
        mbar_wait(smem_u32(&v_full[i % kVStages]), (i / kVStages) & 1, a.limit_ns);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ PV issuer
    //   O += P_j V_j   with P_j read from tensor memory, once the softmax warps published
    //                  P_j and V_j is in; its commit frees V_j's stage and S/P buffer j.
    // The S MMAs come from another thread (warp kWarpS), so neither kind of MMA waits
    // behind the other's inputs: the S issuer waits for PV_j to finish before it reuses
    // P_j's buffer while this thread already has PV_{j+1} queued, and the tensor pipe is
    // never drained between blocks.  A segment's first PV starts O afresh, once the
    // softmax warps have read the previous segment's O.
    if (lane == 0) {
      const uint32_t idPV = idesc_bf16_f32(kBM, D) | (1u << 16);   // B (= V) MN-major
      bool fine = true;
      Seg sg;
      int np = 0, nseg = 0;
      for (int s = 0; fine && segment(s, sg); ++s) {
        if (sg.nblk == 0) continue;
        if (nseg > 0 && !mbar_wait(smem_u32(o_free), (nseg - 1) & 1, a.limit_ns)) {
          fine = false;
          break;
        }
        ++nseg;
        for (int j = 0; j < sg.nblk; ++j, ++np) {
          if (!mbar_wait(smem_u32(&p_full[np % kSP]), (np / kSP) & 1, a.limit_ns) ||
              !mbar_wait(smem_u32(&v_full[np % kVStages]), (np / kVStages) & 1, a.limit_ns)) {
            fine = false;
            break;
          }
          tc_fence_after();
          const uint32_t pa = tmem_base + col_s(np % kSP);
          const uint32_t vs = smem_u32(v_ring + (np % kVStages) * Lay::kStage);
#pragma unroll
          for (int k16 = 0; k16 < kBN / 16; ++k16)   // P of keys 64-127 starts at column 64
            tc_mma_bf16_ts(tmem_base + kColO, pa + (uint32_t)(k16 * 8 + (k16 >= 4 ? 32 : 0)),
                           desc_mnmajor_sw128(vs + k16 * 2048, Lay::kKVHalf), idPV,
                           (j | k16) != 0);
          tc_commit(smem_u32(&pv_done[np % kSP]));
          tc_commit(smem_u32(&v_empty[np % kVStages]));
        }
      }
      if (!fine) record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteMma);
      tc_commit(smem_u32(drain));
      if (!mbar_wait(smem_u32(drain), 0, a.limit_ns))
        record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else if (warp == kWarpS) {
    // ------------------------------------------------------------ S issuer
    //   S_j = Q K_j^T  into S/P buffer j % kSP, once K_j is in and PV_{j-kSP} (the previous
    //                  user of that buffer) is done; its commit frees K_j's stage.  After a
    //                  segment's last S its Q tile is released for the next segment's.
    if (lane == 0) {
      const uint32_t idS = idesc_bf16_f32(kBM, kBN);
      const uint32_t qa = smem_u32(q_s);
      bool fine = true;
      Seg sg;
      int ns = 0, nq = 0;
      for (int s = 0; fine && segment(s, sg); ++s) {
        if (sg.nblk == 0) continue;
        if (!mbar_wait(smem_u32(q_full), nq & 1, a.limit_ns)) {
          record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteQ);
          fine = false;
          break;
        }
        ++nq;
        for (int j = 0; j < sg.nblk; ++j, ++ns) {
          if (!mbar_wait(smem_u32(&k_full[ns % kKStages]), (ns / kKStages) & 1, a.limit_ns) ||
              !mbar_wait(smem_u32(&pv_done[ns % kSP]), ((ns / kSP) & 1) ^ 1, a.limit_ns)) {
            record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteMma);
            fine = false;
            break;
          }
          tc_fence_after();
          const uint32_t ks = smem_u32(k_ring + (ns % kKStages) * Lay::kStage);
#pragma unroll
          for (int h = 0; h < NH; ++h)
#pragma unroll
            for (int k16 = 0; k16 < 4; ++k16)
              tc_mma_bf16(tmem_base + col_s(ns % kSP), desc_kmajor_sw128(qa + h * kBM * 128 + k16 * 32),
                          desc_kmajor_sw128(ks + h * Lay::kKVHalf + k16 * 32), idS, (h | k16) != 0);
          tc_commit(smem_u32(&s_full[ns % kSP]));
          tc_commit(smem_u32(&k_empty[ns % kKStages]));
        }
        tc_commit(smem_u32(q_empty));
      }
      tc_commit(smem_u32(drain_s));
      if (!mbar_wait(smem_u32(drain_s), 0, a.limit_ns))
        record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteDrain);
    }
  } else {
    // ------------------------------------------------------------ softmax / epilogue
    // Two warps per tensor-memory lane quarter: warp w (2..9) serves rows 32 (w % 4) ..
    // +31 and the key half `half` = (w - 2) / 4 of every block (64 keys, written back as
    // 32 columns of packed bf16 P), and the same half of O's columns.  The two halves
    // of a row keep one reference max (agreed through shared memory and a named barrier
    // per quarter when it has to move) and separate partial sums, added at the end.
    // Online softmax in base 2 with a lazily updated reference max: P_j is taken
    // relative to m_ref, which only moves when a row's block max exceeds it by more than
    // kRescaleLog2 (then O in tensor memory and l are rescaled once).  P values stay below
    // 2^kRescaleLog2; the result is the same softmax.
    constexpr int kHalf = kBN / 2;                     // keys per warp and block
    constexpr int kOHalf = D / 2;                      // O columns per warp
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int r = quarter * 32 + lane;                 // tile row = tensor-memory lane
    const uint32_t lane_base = tmem_base + ((uint32_t)(quarter * 32) << 16);
    auto pair_sync = [&]() {                           // the two warps of this quarter
      asm volatile("bar.sync %0, 64;" ::"r"(1 + quarter) : "memory");
    };
    bool ok = true;
    Seg sg;
    int J = 0;                                         // blocks of earlier segments
    for (int s = 0; segment(s, sg); ++s) {
      const TileInfo ti = tile_info(sg.t);
      const int tb_first = first_own(ti, sg);
      const bool rvalid = r < ti.rows;
      const int tok = ti.tok0 + r / a.grp;
      const int crow = min(tok / a.Lq - ti.c_lo, ti.ncand - 1);  // rows past the tile: any candidate
      const int lrow = tok % a.Lq;
      // visible own slots of this row, in the tile's concatenated own-slot space
      const int tlo = crow * a.C;
      const int thi = tlo + max(0, (STREAM ? a.C : n_own[crow]) - a.Lq + lrow + 1);
      int tbs = tb_first;                                // own-block cursor
      float m_ref = -INFINITY, l = 0.f;
      for (int j = 0; j < sg.nblk; ++j) {
        const int jj = J + j;                            // position in the CTA's sequence
        const int sb = jj % kSP;
        // `ok` stays warp-uniform (the warp votes on every bounded wait), so a timed-out
        // warp still meets its partner at every barrier below and the kernel drains
        if (ok && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&s_full[sb]), (jj / kSP) & 1, a.limit_ns))) {
          record_error(a.status, FVRAG_ERR_TIMEOUT, kSiteSFull);
          ok = false;
        }
        tc_fence_after();
        uint32_t sr[kHalf];
        if (ok) {
          static_assert(kHalf == 64, "one 64-column load per warp and block");
          tmem_ld_32x32b_x64(lane_base + col_s(sb) + half * kHalf, sr);
          tmem_wait_ld();
        } else {
#pragma unroll
          for (int c = 0; c < kHalf; ++c) sr[c] = 0u;
        }
        int vlo, vhi;   // valid columns of this block for this row
        if (sg.blk_lo + j < ti.nbp) {
          vlo = 0;
          vhi = min(kBN, ti.P - (sg.blk_lo + j) * kBN);
        } else {
          tbs = own_next(ti, tbs);
          const int base = tbs * kBN;
          ++tbs;
          vlo = max(0, tlo - base);
          vhi = min(kBN, thi - base);
        }
        // this warp's columns are [c_off, c_off + kHalf) of the block
        const int c_off = half * kHalf;
        vlo -= c_off;
        vhi -= c_off;
        // rows without output (r >= rows) are not masked: their values are finite and
        // discarded, and masking them would split the warp between the two paths below
        const bool full = vlo <= 0 && vhi >= kHalf;
        // P_j relative to the reference `mref`: bf16 pairs into pk (written over the first 32
        // of this warp's own S columns of the buffer; S_j is in registers), the partial sum
        // into rs
        uint32_t pk[32];
        float rs = 0.f;
        // kMask: 0 = no masking, 1 = mask every element, 2 = mask when the block is not full
        auto exp_pass_t = [&](float mref, auto mask_mode) {
          constexpr int kMask = decltype(mask_mode)::value;
          const float ms = mref == -INFINITY ? 0.f : mref;
          // exponent arguments s * scale - m and the running sums in packed pairs
          const uint64_t sc2 = f2_pack(a.scale_log2, a.scale_log2), nm2 = f2_pack(-ms, -ms);
          uint64_t rsp2[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) rsp2[u] = 0ull;   // (+0.f, +0.f)
#pragma unroll
          for (int c = 0; c < kHalf; c += 2) {
            float t0, t1;
            f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])), sc2, nm2),
                      t0, t1);
            float e0 = ex2(t0);
            float e1 = ex2(t1);
            if (kMask == 1 || (kMask == 2 && !full)) {
              e0 = (c >= vlo && c < vhi) ? e0 : 0.f;
              e1 = (c + 1 >= vlo && c + 1 < vhi) ? e1 : 0.f;
            }
            rsp2[(c / 2) & 3] = f2_add(rsp2[(c / 2) & 3], f2_pack(e0, e1));
            pk[c / 2] = pack_bf16(e0, e1);
          }
          float rsp[8];
#pragma unroll
          for (int u = 0; u < 4; ++u) f2_unpack(rsp2[u], rsp[2 * u], rsp[2 * u + 1]);
          rs = ((rsp[0] + rsp[1]) + (rsp[2] + rsp[3])) + ((rsp[4] + rsp[5]) + (rsp[6] + rsp[7]));
        };
        // Verification: full blocks (almost all of them) run a copy of the loop without the
        // masking selects, which the compiler otherwise keeps in the loop as predicated
        // instructions (long 145.9 -> 133.6 us per call).  Decode (the balanced plan), whose own
        // blocks are mostly partial, keeps the one loop with the test inside (74.2 us
        // unswitched against 71.7).
        auto exp_pass = [&](float mref) {
          if constexpr (BAL) {
            exp_pass_t(mref, std::integral_constant<int, 2>{});
          } else {
            if (full)
              exp_pass_t(mref, std::integral_constant<int, 0>{});
            else
              exp_pass_t(mref, std::integral_constant<int, 1>{});
          }
        };
        // Once every row of the warp has a reference, the block max is not computed: all
        // terms of the partial sum are positive, so rs <= 2^kRescaleLog2 shows that no term
        // of this half ran past the limit.  A row without a reference, or a larger sum, in
        // either warp of the quarter sends both into the path that computes the block max
        // (the two halves of a row must keep one reference).
        const bool fresh = __any_sync(0xffffffffu, m_ref == -INFINITY);
        if (!fresh) exp_pass(m_ref);
        const bool mine = fresh || __any_sync(0xffffffffu, !(rs <= kSumLimit));
        int* xf = xflag + ((jj & 1) * 2 + half) * 4;     // [2 slots][2 halves][4 quarters]
        if (lane == 0) xf[quarter] = mine ? 1 : 0;
        // Each warp writes its P over its own S columns, so this exchange orders no tensor-
        // memory access between the two; the fences stay because without them the compiler
        // scheduled the streamed form's loop worse (72b 154 -> 156 us per call).
        tc_fence_before();
        pair_sync();
        tc_fence_after();
        const uint32_t pcol = lane_base + col_s(sb) + (uint32_t)(half * kHalf);   // this warp's P
        const bool slow = mine || xflag[((jj & 1) * 2 + (half ^ 1)) * 4 + quarter] != 0;
        bool resc = false;
        float corr = 1.f;
        if (slow) {
          float pm[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) pm[u] = -INFINITY;
          if (full) {
#pragma unroll
            for (int c = 0; c < kHalf; c += 2)
              pm[(c / 2) & 7] = max3(pm[(c / 2) & 7], __uint_as_float(sr[c]), __uint_as_float(sr[c + 1]));
          } else {
#pragma unroll
            for (int c = 0; c < kHalf; ++c)
              if (c >= vlo && c < vhi) pm[c & 7] = fmaxf(pm[c & 7], __uint_as_float(sr[c]));
          }
          float hmax = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                             fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7])));
          // block max over both halves (slots by block parity: the next use of a slot comes
          // after two more flag barriers)
          float* xs = xmax + (jj & 1) * 2 * kBM;
          xs[half * kBM + r] = hmax;
          pair_sync();
          hmax = fmaxf(hmax, xs[(half ^ 1) * kBM + r]);
          const float bmax = a.scale_log2 * hmax;
          const float m_old = m_ref;
          if (bmax > m_ref + kRescaleLog2) m_ref = bmax;   // also the first finite block
          resc = m_ref != m_old && m_old != -INFINITY;
          corr = resc ? ex2(m_old - m_ref) : 1.f;
          if (fresh || __any_sync(0xffffffffu, m_ref != m_old)) exp_pass(m_ref);
          if (ok) tmem_st_32x32b_x32(pcol, pk);
        } else if (ok) {
          // the same store, kept on each path: with one store after the branch the compiler
          // scheduled the loop worse (72b 154 -> 157 us per call)
          tmem_st_32x32b_x32(pcol, pk);
        }
        l = l * corr + rs;
        if (ok && __any_sync(0xffffffffu, resc)) {
          // O holds blocks < j relative to the old reference: wait for PV_{j-1}, then scale
          const int i = jj - 1;
          if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&pv_done[i % kSP]), (i / kSP) & 1, a.limit_ns))) {
            record_error(a.status, FVRAG_ERR_TIMEOUT, kSitePvDone);
            ok = false;
          } else {
            tc_fence_after();
#pragma unroll
            for (int c0 = 0; c0 < kOHalf; c0 += 32) {
              uint32_t o[32];
              tmem_ld_32x32b_x32(lane_base + kColO + half * kOHalf + c0, o);
              tmem_wait_ld();
#pragma unroll
              for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * corr);
              tmem_st_32x32b_x32(lane_base + kColO + half * kOHalf + c0, o);
            }
          }
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&p_full[sb]));
      }
      // ---- epilogue: wait for the last PV, add the two halves' sums, normalise O by l
      if (ok && sg.nblk > 0) {
        const int i = J + sg.nblk - 1;
        if (!mbar_wait(smem_u32(&pv_done[i % kSP]), (i / kSP) & 1, a.limit_ns))
          record_error(a.status, FVRAG_ERR_TIMEOUT, kSitePvDone);
        tc_fence_after();
      }
      xsum[half * kBM + r] = l;
      pair_sync();
      l += xsum[(half ^ 1) * kBM + r];
      const int head = ti.g * a.grp + r % a.grp;
      const size_t rowid = ((size_t)ti.qi * a.KL + tok) * a.hq + head;
      const size_t nrows = (size_t)a.Qn * a.KL * a.hq;
      // partial slot of this row: [slot][row of the tile] (balanced and streamed plans) or
      // [split][row] (static split)
      const bool store = sg.direct || MODE == 0 || sg.pslot >= 0;
      const size_t pidx = MODE == 0 ? (size_t)sg.pslot * nrows + rowid
                                    : (size_t)max(sg.pslot, 0) * a.slot_rows + r;
      const bool any = l > 0.f;
      const float inv = any ? 1.f / l : 0.f;
      const float lse = any ? kLn2 * (m_ref + __log2f(l)) : -INFINITY;
#pragma unroll
      for (int c0 = 0; c0 < kOHalf; c0 += 32) {
        const int oc = half * kOHalf + c0;               // O column of this chunk
        uint32_t o[32];
        if (sg.nblk > 0) {
          tmem_ld_32x32b_x32(lane_base + kColO + oc, o);
          tmem_wait_ld();
        } else {
#pragma unroll
          for (int c = 0; c < 32; ++c) o[c] = 0u;
        }
        if (rvalid && store) {
          if (sg.direct) {
            uint4* dst = reinterpret_cast<uint4*>(a.out + rowid * D + oc);
#pragma unroll
            for (int c = 0; c < 32; c += 8)
              dst[c / 8] = make_uint4(
                  pack_bf16(__uint_as_float(o[c]) * inv, __uint_as_float(o[c + 1]) * inv),
                  pack_bf16(__uint_as_float(o[c + 2]) * inv, __uint_as_float(o[c + 3]) * inv),
                  pack_bf16(__uint_as_float(o[c + 4]) * inv, __uint_as_float(o[c + 5]) * inv),
                  pack_bf16(__uint_as_float(o[c + 6]) * inv, __uint_as_float(o[c + 7]) * inv));
          } else {
            uint4* dst = reinterpret_cast<uint4*>(a.part_o + pidx * D + oc);
#pragma unroll
            for (int c = 0; c < 32; c += 8)
              dst[c / 8] = make_uint4(
                  pack_f16(__uint_as_float(o[c]) * inv, __uint_as_float(o[c + 1]) * inv),
                  pack_f16(__uint_as_float(o[c + 2]) * inv, __uint_as_float(o[c + 3]) * inv),
                  pack_f16(__uint_as_float(o[c + 4]) * inv, __uint_as_float(o[c + 5]) * inv),
                  pack_f16(__uint_as_float(o[c + 6]) * inv, __uint_as_float(o[c + 7]) * inv));
          }
        }
      }
      if (rvalid && half == 0 && store) {
        if (sg.direct) {
          if (a.lse) a.lse[rowid] = lse;
        } else {
          a.part_lse[pidx] = lse;
        }
      }
      if (!store && lane == 0 && half == 0 && quarter == 0)
        record_error(a.status, FVRAG_ERR_UNSUPPORTED, kSitePlan);
      // O has been read: the next segment's first PV may overwrite it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(o_free));
      J += sg.nblk;
    }
  }
  griddep_launch_dependents();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, kTmemCols);
}

// Where the partials of a tile live under the balanced plan (null otherwise).
struct RunTable {
  const int2* tile_runs;   // [tiles] {first slot, runs}
  int slot_rows, KL, hq, grp, T, mtiles, hkv;
};

// One warp per output row: out = sum_s w_s o_s / sum_s w_s with w_s = exp(lse_s - max lse),
// lse = max + log(sum_s w_s).  Lane s holds split s's weight (and s + 32); all partial
// loads of a group of 8 splits are issued before any is used.  Partial s of the row sits
// at index first + s * stride: [split][row] (static plan), or [slot][row of the tile]
// with the tile's runs in consecutive slots (balanced plan; a tile with one run was
// written by its CTA directly).
template <int D>
__global__ void merge_kernel(const __half* __restrict__ part_o, const float* __restrict__ part_lse,
                             int nsplit, long long nrows, __nv_bfloat16* __restrict__ out,
                             float* __restrict__ lse_out, const RunTable rt) {
  constexpr int DPL = D / 32;
  griddep_wait();
  griddep_launch_dependents();
  const long long row = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= nrows) return;
  long long first = row, stride = nrows;
  if (rt.tile_runs) {
    const int head = (int)(row % rt.hq);
    const long long tq = row / rt.hq;
    const int tok = (int)(tq % rt.KL);
    const int qi = (int)(tq / rt.KL);
    const int g = head / rt.grp;
    const int mt = tok / rt.T;
    const int r = (tok - mt * rt.T) * rt.grp + head % rt.grp;
    const int2 tr = rt.tile_runs[((long long)qi * rt.hkv + g) * rt.mtiles + mt];
    if (tr.y <= 1) return;
    nsplit = tr.y;
    first = (long long)tr.x * rt.slot_rows + r;
    stride = rt.slot_rows;
  }
  const float l0 = lane < nsplit ? part_lse[first + lane * stride] : -INFINITY;
  const float l1 = lane + 32 < nsplit ? part_lse[first + (lane + 32) * stride] : -INFINITY;
  const float mx = warp_max(fmaxf(l0, l1));
  const float w0 = l0 == -INFINITY ? 0.f : __expf(l0 - mx);
  const float w1 = l1 == -INFINITY ? 0.f : __expf(l1 - mx);
  const float den = warp_sum(w0 + w1);
  float res[DPL];
#pragma unroll
  for (int i = 0; i < DPL; ++i) res[i] = 0.f;
  const __half* base = part_o + (size_t)first * D + lane * DPL;
  for (int s0 = 0; s0 < nsplit; s0 += 8) {
    float v[8][DPL];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      if (s0 + u < nsplit) {
        const __half2* po = reinterpret_cast<const __half2*>(base + (size_t)(s0 + u) * stride * D);
        if constexpr (DPL == 4) {
          const uint2 raw = *reinterpret_cast<const uint2*>(po);
          const float2 f0 = __half22float2(*reinterpret_cast<const __half2*>(&raw.x));
          const float2 f1 = __half22float2(*reinterpret_cast<const __half2*>(&raw.y));
          v[u][0] = f0.x;
          v[u][1] = f0.y;
          v[u][2] = f1.x;
          v[u][3] = f1.y;
        } else {
#pragma unroll
          for (int i = 0; i < DPL; i += 2) {
            const float2 f = __half22float2(po[i / 2]);
            v[u][i] = f.x;
            v[u][i + 1] = f.y;
          }
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int sp = s0 + u;
      if (sp < nsplit) {
        const float w = __shfl_sync(0xffffffffu, sp < 32 ? w0 : w1, sp & 31);
#pragma unroll
        for (int i = 0; i < DPL; ++i) res[i] = fmaf(w, v[u][i], res[i]);
      }
    }
  }
  const float inv = den > 0.f ? 1.f / den : 0.f;
  __nv_bfloat16* o = out + row * D + lane * DPL;
#pragma unroll
  for (int i = 0; i < DPL; i += 2)
    *reinterpret_cast<__nv_bfloat162*>(o + i) = __floats2bfloat162_rn(res[i] * inv, res[i + 1] * inv);
  if (lane == 0 && lse_out) lse_out[row] = den > 0.f ? mx + __logf(den) : -INFINITY;
}

// One attention problem in the general form of the kernel (see the top of the file).
struct Problem {
  int Qn, K, Lq, C, hq, hkv, D, max_prefix, total_prefix;
  float scale;                 // 0 => 1/sqrt(D)
  const int32_t* own_len;      // device [Qn][K] or null (every candidate has C valid slots)
  bool ragged;                 // the valid own slots n_k are read from the device
  uint32_t split;              // FVRAG_ATTN_SPLIT_* request (verification), 0 = by the cost model
};

struct Plan {
  int grp, T, mtiles, nsplit;
  bool stream;             // the streamed plan (grid CTAs, maxparts partial slots per tile)
  int grid, maxparts;
  bool unsupported;        // the streamed plan was requested but cannot serve the problem
};

// L2 capacity of the current device (cached per device; 126.5 MB if it cannot be read).
static double l2_bytes() {
  static double cached[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 126.5e6;
  if (cached[dev] == 0) {
    int v = 0;
    cached[dev] = cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev) == cudaSuccess && v > 0
                      ? (double)v : 126.5e6;
  }
  return cached[dev];
}

// Own blocks of row tile mt (every candidate with all C slots valid).
static int own_blocks(const Problem& pr, const Plan& p, int mt) {
  const int KL = pr.K * pr.Lq;
  const int tok0 = mt * p.T;
  const int ntok = std::min(p.T, KL - tok0);
  const int c_lo = tok0 / pr.Lq;
  const int ncand = (tok0 + ntok - 1) / pr.Lq - c_lo + 1;
  return (ncand * pr.C + kBN - 1) / kBN;
}

// Key-split plan.  Static split: every row tile's block list (its query's prefix blocks
// plus the own blocks of its candidates) is cut on the device into nsplit equal runs, one
// CTA each, so a short ragged prefix gives short CTAs that the block scheduler backfills.
// Streamed plan (verification only): each of `grid` CTAs takes an equal share of all tiles'
// blocks in one wave.  Pick the plan with the smaller estimate of the time: for the static
// split the larger of the mean work per SM (waves x mean run, three blocks added per run for
// its prologue and epilogue) and the longest run, for the streamed plan its share; plus the
// cost of writing and merging the fp16 partials.  The constants (~0.8 us per 128-key block;
// per split count, a fixed 20 us and the partials written and read at ~3 TB/s) were fitted
// on GB300 to per-call times of the static split measured at every split count from 1 to 12
// on the 72B-class, long-context and batch-16 workloads; the streamed plan's terms to its
// times on the same workloads (72B-class: 158 us against the static split's 181 us; long
// context: 117 against 111 us; batch-16, whose K/V does not fit L2: 233 against 177 us).
static Plan make_plan(const Problem& pr, int sms) {
  Plan p;
  p.grp = pr.hq / pr.hkv;
  p.T = std::max(1, kBM / p.grp);
  const int KL = pr.K * pr.Lq;
  p.mtiles = (KL + p.T - 1) / p.T;
  p.stream = false;
  p.grid = 0;
  p.maxparts = 1;
  p.unsupported = false;
  const long long base = (long long)pr.Qn * pr.hkv * p.mtiles;
  const int ncand = std::min(pr.K, (p.T + pr.Lq - 1) / pr.Lq + 1);
  const int nb_own = (int)(((long long)ncand * pr.C + kBN - 1) / kBN);
  const int nb = (std::max(pr.max_prefix, 0) + kBN - 1) / kBN + nb_own;
  const double nb_mean = std::ceil((double)std::max(pr.total_prefix, 0) / pr.Qn / kBN) + nb_own;
  p.nsplit = 1;
  if (sms <= 0) sms = 148;
  if (nb <= 1 && pr.split != FVRAG_ATTN_SPLIT_STREAM) return p;
  const double rows = (double)pr.Qn * KL * pr.hq;
  auto merge_us = [&](double ns) { return 20.0 + ns * rows * (pr.D * 2 + 4) * 2.0 / 3.0e6; };
  double best = 1e30;
  for (int ns = 1; ns <= std::min(nb, 64); ++ns) {
    const long long ctas = base * ns;
    const double waves = (double)((ctas + sms - 1) / sms);
    const double t_mean = waves * (std::ceil(nb_mean / ns) + 3);
    const double t_max = std::ceil((double)nb / ns) + 3;
    double t = std::max(t_mean, t_max) * 0.8;
    if (ns > 1) t += merge_us(ns);
    if (t < best - 1e-9) {
      best = t;
      p.nsplit = ns;
    }
  }
  // the streamed plan's CTAs read different K/V blocks of a KV head at the same time, so it
  // needs every query's prefix K/V resident in L2 (3/4 of it) to keep one HBM read per block
  const double kv_bytes = 4.0 * pr.hkv * pr.D * (double)std::max(pr.total_prefix, 0);
  const bool want_stream = pr.split == FVRAG_ATTN_SPLIT_STREAM;
  if (want_stream) best = 1e30;            // requested: no comparison with the static split
  if (pr.split == FVRAG_ATTN_SPLIT_STATIC) {
    // requested: the static split as chosen above
  } else if (!pr.ragged && pr.Qn <= kMaxStreamQueries && p.mtiles <= kMaxStreamMtiles &&
             (want_stream || kv_bytes <= 0.75 * l2_bytes())) {
    long long ntb_all = 0;
    int ntb_max = 0;
    for (int mt = 0; mt < p.mtiles; ++mt) {
      const int b = own_blocks(pr, p, mt);
      ntb_all += b;
      ntb_max = std::max(ntb_max, b);
    }
    // sum over queries of ceil(P_q / 128) lies between these two (P_q sum to total_prefix)
    const long long tp = std::max(pr.total_prefix, 0);
    const long long pre_lb = (tp + kBN - 1) / kBN;
    const long long pre_ub = (tp + (long long)pr.Qn * (kBN - 1)) / kBN;
    const long long w_lb = (long long)pr.hkv * (p.mtiles * pre_lb + (long long)pr.Qn * ntb_all);
    const long long w_ub = (long long)pr.hkv * (p.mtiles * pre_ub + (long long)pr.Qn * ntb_all);
    const int grid = (int)std::max(1LL, std::min<long long>(sms, w_lb));
    const long long range = std::max(1LL, w_lb / grid);       // fewest blocks of a share
    const int nbmax = (std::max(pr.max_prefix, 0) + kBN - 1) / kBN + ntb_max;
    const long long maxparts = (nbmax - 1 + range - 1) / range + 1;
    if (maxparts <= kMaxRuns) {
      // per block ~7 % above the static split's (measured: its row tiles of a KV head do not
      // read a block in lockstep), plus two blocks per change of tile within a share
      const double share = std::ceil((double)w_ub / grid);
      const double segs = std::ceil(share / std::max(1.0, nb_mean)) + 1;
      double t = (share + 3 + 2 * segs) * 0.8 * 1.07;
      if (maxparts > 1) t += merge_us(std::min<double>(maxparts, 2.0));
      if (t < best - 1e-9) {
        p.stream = true;
        p.grid = grid;
        p.maxparts = (int)maxparts;
      }
    }
  }
  p.unsupported = want_stream && !p.stream;
  return p;
}

// The balanced plan serves problems whose tiles' block lists differ by the n_k on the
// device (decode): one grid of CTAs, a whole number of waves over the SMs with room for
// every tile's first run and a quarter more.
static bool balanced_grid(const Problem& pr, const Plan& p, int sms, int* grid) {
  if (!pr.ragged) return false;
  const long long ntiles = (long long)pr.Qn * pr.hkv * p.mtiles;
  if (ntiles > kMaxPlanTiles || pr.Qn > kMaxPlanQueries || (long long)pr.Qn * pr.K > kMaxPlanOwn)
    return false;
  const long long waves = (ntiles + ntiles / 4) / sms + 1;
  if (waves > 8) return false;
  *grid = (int)(waves * sms);
  return true;
}

// Workspace of the balanced and streamed plans: header | tile runs [tiles] | partial O
// [slots][T * grp][D] | partial lse [slots][T * grp], with one slot per CTA (balanced) or
// maxparts slots per tile (streamed).
struct BalancedWs {
  size_t runs, part_o, part_lse, total;
};

static BalancedWs balanced_ws(const Problem& pr, const Plan& p, long long nslots) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  const size_t ntiles = (size_t)pr.Qn * pr.hkv * p.mtiles;
  const size_t slots = (size_t)nslots * p.grp * p.T;
  BalancedWs w;
  w.runs = up(kWsHeaderBytes);
  w.part_o = w.runs + up(ntiles * sizeof(int2));
  w.part_lse = w.part_o + up(slots * pr.D * 2);
  w.total = w.part_lse + up(slots * 4);
  return w;
}

static long long stream_slots(const Problem& pr, const Plan& p) {
  return (long long)pr.Qn * pr.hkv * p.mtiles * p.maxparts;
}

static size_t ws_bytes(const Problem& pr, int sms) {
  const Plan p = make_plan(pr, sms);
  if (p.unsupported) return 0;
  int grid = 0;
  if (balanced_grid(pr, p, sms, &grid)) return balanced_ws(pr, p, grid).total;
  if (p.stream) return balanced_ws(pr, p, stream_slots(pr, p)).total;
  const size_t rows = (size_t)pr.Qn * pr.K * pr.Lq * pr.hq;
  // partial outputs fp16 [nsplit][rows][D], then their lse fp32 [nsplit][rows]
  return kWsHeaderBytes + (p.nsplit > 1 ? (size_t)p.nsplit * rows * ((size_t)pr.D * 2 + 4) : 0);
}

static int device_sms() {
  const int s = sm_count();
  return s > 0 ? s : 148;
}

// The SMs a verification call plans for; -1 when the budget is outside 0 .. the SM count.
static int budget_sms(int32_t budget) {
  const int s = sm_count();
  if (budget < 0 || (s > 0 && budget > s)) return -1;
  return budget > 0 ? budget : device_sms();
}

template <int D, int MODE>
static fvrag_status launch(const CUtensorMap* maps, const Args& a, long long grid, cudaStream_t s) {
  const int sm = Layout<D>::kBytes;
  auto kern = attn_kernel<D, MODE>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, sm) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  if (launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), (size_t)sm, s, maps[0], maps[1],
                 maps[2], maps[3], maps[4], a) != cudaSuccess)
    return FVRAG_ERR_CUDA;
  return launch_status();
}

// Shape checks shared by both entry points (after their own argument checks).
static fvrag_status check_problem(const Problem& pr) {
  if (pr.hq % pr.hkv != 0 || (pr.D != 64 && pr.D != 128) || pr.hq / pr.hkv > kBM)
    return FVRAG_ERR_UNSUPPORTED;
  if ((long long)pr.Qn * pr.K * pr.C >= (1LL << 31) || (long long)pr.Qn * pr.K * pr.Lq >= (1LL << 31) ||
      (long long)pr.total_prefix + kBN >= (1LL << 31))
    return FVRAG_ERR_UNSUPPORTED;
  return FVRAG_OK;
}

// q [Qn][K][Lq][hq][D]; own K/V [Qn][K][C][hkv][D]; out like q.
// `sms`: the SMs the split is planned for (the device's count, or the caller's budget).
static fvrag_status run(const Problem& pr, int sms, const void* q, const void* k_prefix,
                        const void* v_prefix, const int32_t* prefix_offsets, const void* k_own,
                        const void* v_own, void* out, float* lse, void* ws, size_t ws_size,
                        cudaStream_t s) {
  const size_t need = ws_bytes(pr, sms);
  if (need == 0) return FVRAG_ERR_UNSUPPORTED;   // a requested streamed plan cannot serve it
  if (!ws || ws_size < need) return FVRAG_ERR_WORKSPACE;
  if (!aligned16(ws)) return FVRAG_ERR_MISALIGNED;

  const Plan p = make_plan(pr, sms);
  const int D = pr.D;
  const float scale = pr.scale != 0.f ? pr.scale : 1.f / sqrtf((float)D);
  const int KL = pr.K * pr.Lq;
  const long long nrows = (long long)pr.Qn * KL * pr.hq;
  uint8_t* base = reinterpret_cast<uint8_t*>(ws);

  CUtensorMap maps[5];
  {
    const uint64_t dims[3] = {(uint64_t)D, (uint64_t)pr.hq, (uint64_t)pr.Qn * KL};
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)pr.hq * D * 2};
    const uint32_t box[3] = {64u, (uint32_t)p.grp, (uint32_t)p.T};
    if (!encode_tmap_bf16(&maps[0], q, 3, dims, strides, box, true)) return FVRAG_ERR_CUDA;
  }
  {
    const uint64_t strides[2] = {(uint64_t)D * 2, (uint64_t)pr.hkv * D * 2};
    const uint32_t box[3] = {64u, 1u, (uint32_t)kBN};
    const uint64_t tdims[3] = {(uint64_t)D, (uint64_t)pr.hkv, (uint64_t)pr.Qn * pr.K * pr.C};
    if (!encode_tmap_bf16(&maps[3], k_own, 3, tdims, strides, box, true)) return FVRAG_ERR_CUDA;
    if (!encode_tmap_bf16(&maps[4], v_own, 3, tdims, strides, box, true)) return FVRAG_ERR_CUDA;
    if (pr.total_prefix > 0) {
      const uint64_t pdims[3] = {(uint64_t)D, (uint64_t)pr.hkv, (uint64_t)pr.total_prefix};
      if (!encode_tmap_bf16(&maps[1], k_prefix, 3, pdims, strides, box, true)) return FVRAG_ERR_CUDA;
      if (!encode_tmap_bf16(&maps[2], v_prefix, 3, pdims, strides, box, true)) return FVRAG_ERR_CUDA;
    } else {
      maps[1] = maps[3];   // never read: no query has prefix keys
      maps[2] = maps[4];
    }
  }
  int bgrid = 0;
  const bool bal = balanced_grid(pr, p, sms, &bgrid);
  const bool strm = !bal && p.stream;
  const BalancedWs bw = bal ? balanced_ws(pr, p, bgrid)
                            : strm ? balanced_ws(pr, p, stream_slots(pr, p)) : BalancedWs{};
  Args a;
  a.tile_runs = (bal || strm) ? reinterpret_cast<int2*>(base + bw.runs) : nullptr;
  a.offs = prefix_offsets;
  a.own_len = pr.own_len;
  a.out = reinterpret_cast<__nv_bfloat16*>(out);
  a.lse = lse;
  if (bal || strm) {
    a.part_o = reinterpret_cast<__half*>(base + bw.part_o);
    a.part_lse = reinterpret_cast<float*>(base + bw.part_lse);
  } else {
    a.part_o = reinterpret_cast<__half*>(base + kWsHeaderBytes);
    a.part_lse = reinterpret_cast<float*>(a.part_o + (size_t)p.nsplit * nrows * D);
  }
  a.status = reinterpret_cast<uint32_t*>(base);
  a.limit_ns = wait_limit_ns();
  a.Qn = pr.Qn;
  a.K = pr.K;
  a.Lq = pr.Lq;
  a.C = pr.C;
  a.KL = KL;
  a.hq = pr.hq;
  a.hkv = pr.hkv;
  a.grp = p.grp;
  a.T = p.T;
  a.mtiles = p.mtiles;
  a.nsplit = p.nsplit;
  a.slot_rows = p.grp * p.T;
  a.maxparts = p.maxparts;
  a.scale_log2 = scale * kLog2e;
  RunTable rt{nullptr, a.slot_rows, KL, pr.hq, p.grp, p.T, p.mtiles, pr.hkv};
  long long grid = (long long)pr.Qn * pr.hkv * p.nsplit * p.mtiles;
  if (bal || strm) {
    rt.tile_runs = a.tile_runs;
    grid = bal ? bgrid : p.grid;
  }
  if (grid > 0x7fffffffLL) return FVRAG_ERR_UNSUPPORTED;
  fvrag_status st;
  if (bal)
    st = D == 128 ? launch<128, 1>(maps, a, grid, s) : launch<64, 1>(maps, a, grid, s);
  else if (strm)
    st = D == 128 ? launch<128, 2>(maps, a, grid, s) : launch<64, 2>(maps, a, grid, s);
  else
    st = D == 128 ? launch<128, 0>(maps, a, grid, s) : launch<64, 0>(maps, a, grid, s);
  if (st != FVRAG_OK) return st;
  if (!bal && !(strm && p.maxparts > 1) && !(!strm && p.nsplit > 1)) return st;
  const int wpb = 8;
  const long long blocks = (nrows + wpb - 1) / wpb;
  const cudaError_t e =
      D == 128 ? launch_pdl(merge_kernel<128>, dim3((unsigned)blocks), dim3(32 * wpb), 0, s,
                            (const __half*)a.part_o, (const float*)a.part_lse, p.nsplit, nrows, a.out,
                            lse, rt)
               : launch_pdl(merge_kernel<64>, dim3((unsigned)blocks), dim3(32 * wpb), 0, s,
                            (const __half*)a.part_o, (const float*)a.part_lse, p.nsplit, nrows, a.out,
                            lse, rt);
  if (e != cudaSuccess) return FVRAG_ERR_CUDA;
  return launch_status();
}

static Problem verify_problem(const fvrag_attn_desc* d) {
  return Problem{d->num_queries, d->num_cand, d->cand_len, d->cand_len, d->hq, d->hkv,
                 d->head_dim, d->max_prefix, d->total_prefix, d->softmax_scale, nullptr, false,
                 d->flags};
}

static Problem decode_problem(const fvrag_decode_desc* d, const int32_t* cache_len) {
  return Problem{d->num_queries, d->num_drafts, 1, d->cache_cap, d->hq, d->hkv,
                 d->head_dim, d->max_prefix, d->total_prefix, d->softmax_scale, cache_len, true,
                 0u};
}

static bool split_flags_ok(uint32_t f) {
  return f == 0 || f == FVRAG_ATTN_SPLIT_STATIC || f == FVRAG_ATTN_SPLIT_STREAM;
}

}  // namespace attn
}  // namespace fvrag

using namespace fvrag;

extern "C" size_t fvrag_verify_attn_workspace(const fvrag_attn_desc* d) {
  if (!d || d->num_queries < 1 || d->num_cand < 1 || d->cand_len < 1 || d->hq < 1 || d->hkv < 1 ||
      d->hq % d->hkv || (d->head_dim != 64 && d->head_dim != 128) || d->max_prefix < 0 ||
      !attn::split_flags_ok(d->flags))
    return 0;
  const int sms = attn::budget_sms(d->sm_budget);
  if (sms < 0) return 0;
  return attn::ws_bytes(attn::verify_problem(d), sms);
}

extern "C" fvrag_status fvrag_verify_attn(const fvrag_attn_desc* d, const void* q,
                                          const void* k_prefix, const void* v_prefix,
                                          const int32_t* prefix_offsets, const void* k_tail,
                                          const void* v_tail, void* out, float* lse, void* ws,
                                          size_t ws_size, fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_verify_attn");
  using namespace attn;
  if (!d || !q || !prefix_offsets || !k_tail || !v_tail || !out) return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_cand < 1 || d->cand_len < 1 || d->hq < 1 || d->hkv < 1 ||
      d->max_prefix < 0 || d->total_prefix < 0 || !split_flags_ok(d->flags) ||
      !(d->softmax_scale >= 0.f) || d->softmax_scale == INFINITY)
    return FVRAG_ERR_INVALID_ARG;
  if (d->total_prefix > 0 && (!k_prefix || !v_prefix)) return FVRAG_ERR_INVALID_ARG;
  const int sms = budget_sms(d->sm_budget);
  if (sms < 0) return FVRAG_ERR_INVALID_ARG;
  if (d->cand_len > kMaxTail) return FVRAG_ERR_UNSUPPORTED;
  const Problem pr = verify_problem(d);
  const fvrag_status cs = check_problem(pr);
  if (cs != FVRAG_OK) return cs;
  if (!aligned16(q) || !aligned16(k_tail) || !aligned16(v_tail) || !aligned16(out) ||
      (k_prefix && !aligned16(k_prefix)) || (v_prefix && !aligned16(v_prefix)))
    return FVRAG_ERR_MISALIGNED;
  return run(pr, sms, q, k_prefix, v_prefix, prefix_offsets, k_tail, v_tail, out, lse, ws,
             ws_size, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" size_t fvrag_decode_attn_workspace(const fvrag_decode_desc* d) {
  if (!d || d->num_queries < 1 || d->num_drafts < 1 || d->cache_cap < 1 || d->hq < 1 ||
      d->hkv < 1 || d->hq % d->hkv || (d->head_dim != 64 && d->head_dim != 128) || d->max_prefix < 0)
    return 0;
  return attn::ws_bytes(attn::decode_problem(d, nullptr), attn::device_sms());
}

extern "C" fvrag_status fvrag_decode_attn(const fvrag_decode_desc* d, const void* q,
                                          const void* k_prefix, const void* v_prefix,
                                          const int32_t* prefix_offsets, const void* k_cache,
                                          const void* v_cache, const int32_t* cache_len, void* out,
                                          float* lse, void* ws, size_t ws_size,
                                          fvrag_stream_t stream) {
  NvtxRange nvtx_range("fvrag_decode_attn");
  using namespace attn;
  if (!d || !q || !prefix_offsets || !k_cache || !v_cache || !cache_len || !out)
    return FVRAG_ERR_INVALID_ARG;
  if (d->num_queries < 1 || d->num_drafts < 1 || d->cache_cap < 1 || d->hq < 1 || d->hkv < 1 ||
      d->max_prefix < 0 || d->total_prefix < 0 || d->flags != 0 || !(d->softmax_scale >= 0.f) ||
      d->softmax_scale == INFINITY)
    return FVRAG_ERR_INVALID_ARG;
  if (d->total_prefix > 0 && (!k_prefix || !v_prefix)) return FVRAG_ERR_INVALID_ARG;
  const Problem pr = decode_problem(d, cache_len);
  const fvrag_status cs = check_problem(pr);
  if (cs != FVRAG_OK) return cs;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out) ||
      (k_prefix && !aligned16(k_prefix)) || (v_prefix && !aligned16(v_prefix)))
    return FVRAG_ERR_MISALIGNED;
  return run(pr, device_sms(), q, k_prefix, v_prefix, prefix_offsets, k_cache, v_cache, out, lse,
             ws, ws_size, reinterpret_cast<cudaStream_t>(stream));
}
