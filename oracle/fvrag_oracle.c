/*
 * fvrag oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, fp64 CPU statement of what the verifier hot path of
 * VideoSpeculateRAG computes.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this library; the product path
 * (libfvrag, its CUDA kernels and its Python binding) never touches it, and the
 * two share no code: inputs arrive as raw bf16/fp16 bit patterns and are decoded
 * here, exactly, by this file's own routines.
 *
 * Every floating-point sum runs in fp64 over a fixed index order, so the result
 * does not depend on the number of OpenMP threads (threads only split
 * independent output rows).
 *
 * Functions and the passages they follow:
 *   oracle_verify_attn    -- the verifier forward of Eq. 6 (Section 3.1) and
 *                            Eq. 11 (Section 3.2, "Two-Stage Verification")
 *                            restricted to one attention layer: every
 *                            candidate token attends to
 *                            the shared prefix (Q, V, retrieved passages) and to
 *                            its own candidate's tokens up to itself.
 *   oracle_score_logprobs -- the verifier's token probabilities P(token | ...):
 *                            log-softmax of the LM-head logits, gathered at the
 *                            requested token ids (Eq. 11; "self-consistent"
 *                            likelihood, Section 4.6 "Analysis of Scoring
 *                            Mechanisms").
 *   oracle_clip_align     -- Eq. 14 (cosine of CLIP embeddings) and Eq. 15 (max
 *                            over the frames), plus the keep/drop threshold.
 *   oracle_select         -- selection: length-normalised likelihood masked by
 *                            keep (mode 0), or Algorithm 1's two stages:
 *                            Eq. 12 reliability, Eq. 13 high-reliability set,
 *                            argmax alignment over it (mode 1), and the
 *                            other strategies of Sections 4.5-4.6 (modes 2-6).
 *                            Parity unpinned against the paper on two readings
 *                            only: the mean (not the sum) of the token log-probs
 *                            in mode 0, and which token ids stand for "Yes" and
 *                            "No" (the caller's targets); the function itself is
 *                            pinned by the tests.
 *   oracle_decode_attn    -- one decode step of the K drafts (Eq. 5, Eq. 8-10):
 *                            each draft's newest token over the shared prefix
 *                            and its own tokens.
 *   oracle_frame_topk     -- Eq. 2: each keyframe's most similar corpus texts.
 *   oracle_aggregate_topk -- Eq. 3: the union of a query's per-keyframe lists
 *                            and its K best texts.
 *   oracle_keyframes      -- Eq. 1: colour-histogram similarity of consecutive
 *                            frames and the keyframe set.
 * Readings where the paper is silent are stated beside each function.
 *
 * Build: gcc -O2 -fopenmp -shared -fPIC fvrag_oracle.c -o libfvrag_oracle.so -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* ---- exact decoding of the 16-bit formats (IEEE 754 binary16; bfloat16 =
 * the top half of an IEEE binary32) ---------------------------------------- */
static double dec_bf16(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

static double dec_f16(uint16_t h) {
  int sign = (h >> 15) & 1;
  int ex = (h >> 10) & 0x1F;
  int man = h & 0x3FF;
  double v;
  if (ex == 0) {
    v = ldexp((double)man, -24); /* subnormal: man * 2^-24 */
  } else if (ex == 31) {
    v = man ? NAN : INFINITY;
  } else {
    v = ldexp((double)(man + 1024), ex - 25); /* (1 + man/1024) * 2^(ex-15) */
  }
  return sign ? -v : v;
}

void oracle_decode_bf16(const uint16_t* in, double* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = dec_bf16(in[i]);
}

void oracle_decode_f16(const uint16_t* in, double* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = dec_f16(in[i]);
}

/*
 * Attention of one verifier layer over the shared prefix and each candidate's
 * own tokens.
 *
 *   q       [Qn][K][L][Hq][D]   bf16     query of token l of candidate k
 *   k_pre   [sum P][Hkv][D]     bf16     prefix keys; query qi owns rows
 *   v_pre   [sum P][Hkv][D]     bf16       offs[qi] .. offs[qi+1]-1
 *   offs    [Qn+1]              int32
 *   k_tail  [Qn][K][L][Hkv][D]  bf16     keys / values of the candidate tokens
 *   v_tail  [Qn][K][L][Hkv][D]  bf16
 *   row_sel [Qn*K*L*Hq] or NULL          compute only rows with row_sel != 0
 *   out     [Qn][K][L][Hq][D]   fp64
 *   lse     [Qn][K][L][Hq]      fp64 or NULL (natural log of the softmax denominator
 *                                             including the max shift)
 *
 * For query qi, candidate k, token l, head h with kv head g = h / (Hq / Hkv):
 *   keys  S = { prefix j : 0 <= j < P_qi }  U  { tail (k, t) : 0 <= t <= l }
 *   s_j   = scale * <q, K_j[g]>
 *   out   = sum_j softmax(s)_j * V_j[g],   lse = max s + ln sum_j exp(s_j - max s)
 * Readings: candidates do not see one another (Eq. 6 scores each a_i on its own);
 * consecutive query heads share a KV head; scale = 1/sqrt(D) unless given.
 * Returns 0, or -1 on bad arguments.
 */
int oracle_verify_attn(int Qn, int K, int L, int Hq, int Hkv, int D, double scale,
                       const uint16_t* q, const uint16_t* k_pre, const uint16_t* v_pre,
                       const int32_t* offs, const uint16_t* k_tail, const uint16_t* v_tail,
                       const uint8_t* row_sel, double* out, double* lse) {
  if (Qn <= 0 || K <= 0 || L <= 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || Hq % Hkv) return -1;
  if (!q || !offs || !k_tail || !v_tail || !out) return -1;
  if (scale == 0.0) scale = 1.0 / sqrt((double)D);
  const int grp = Hq / Hkv;
  int maxP = 0;
  for (int qi = 0; qi < Qn; ++qi) {
    int p = offs[qi + 1] - offs[qi];
    if (p < 0) return -1;
    if (p > maxP) maxP = p;
  }
  if (maxP > 0 && (!k_pre || !v_pre)) return -1;
  const int64_t nrows = (int64_t)Qn * K * L * Hq;
  int bad = 0;
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)(maxP + L));
    double* qv = (double*)malloc(sizeof(double) * (size_t)D);
    double* acc = (double*)malloc(sizeof(double) * (size_t)D);
    if (!s || !qv || !acc) {
#pragma omp atomic write
      bad = 1;
    }
#pragma omp for schedule(dynamic, 4)
    for (int64_t r = 0; r < nrows; ++r) {
      if (bad) continue;
      if (row_sel && !row_sel[r]) continue;
      const int h = (int)(r % Hq);
      const int64_t tok = r / Hq; /* ((qi*K + k)*L + l) */
      const int l = (int)(tok % L);
      const int k = (int)((tok / L) % K);
      const int qi = (int)(tok / ((int64_t)L * K));
      const int g = h / grp;
      const int P = offs[qi + 1] - offs[qi];
      for (int d = 0; d < D; ++d) qv[d] = dec_bf16(q[r * D + d]);
      int n = 0;
      for (int j = 0; j < P; ++j) {
        const uint16_t* kr = k_pre + ((int64_t)(offs[qi] + j) * Hkv + g) * D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d) dot += qv[d] * dec_bf16(kr[d]);
        s[n++] = scale * dot;
      }
      for (int t = 0; t <= l; ++t) {
        const uint16_t* kr = k_tail + ((((int64_t)qi * K + k) * L + t) * Hkv + g) * D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d) dot += qv[d] * dec_bf16(kr[d]);
        s[n++] = scale * dot;
      }
      double m = -INFINITY;
      for (int j = 0; j < n; ++j) if (s[j] > m) m = s[j];
      double Z = 0.0;
      for (int j = 0; j < n; ++j) Z += exp(s[j] - m);
      for (int d = 0; d < D; ++d) acc[d] = 0.0;
      int j = 0;
      for (; j < P; ++j) {
        const double p = exp(s[j] - m) / Z;
        const uint16_t* vr = v_pre + ((int64_t)(offs[qi] + j) * Hkv + g) * D;
        for (int d = 0; d < D; ++d) acc[d] += p * dec_bf16(vr[d]);
      }
      for (int t = 0; t <= l; ++t, ++j) {
        const double p = exp(s[j] - m) / Z;
        const uint16_t* vr = v_tail + ((((int64_t)qi * K + k) * L + t) * Hkv + g) * D;
        for (int d = 0; d < D; ++d) acc[d] += p * dec_bf16(vr[d]);
      }
      for (int d = 0; d < D; ++d) out[r * D + d] = acc[d];
      if (lse) lse[r] = m + log(Z);
    }
    free(s);
    free(qv);
    free(acc);
  }
  return bad ? -1 : 0;
}

/*
 * One decode step of the drafter (Eq. 5; the generation of e_i, r_i and a_i in
 * Eq. 8-10): the K drafts of a query are generated in parallel, each from the
 * shared prefix (video tokens and question) followed by its own tokens (its
 * retrieved text t_i and what it has generated so far).  Each draft's newest
 * token attends to the whole prefix and to its own tokens up to itself.
 *
 *   q        [Qn][K][Hq][D]     bf16   query of each draft's newest token
 *   k_pre    [sum P][Hkv][D]    bf16   shared prefix keys / values; query qi owns
 *   v_pre    [sum P][Hkv][D]    bf16     rows offs[qi] .. offs[qi+1]-1
 *   offs     [Qn+1]             int32
 *   k_cache  [Qn][K][C][Hkv][D] bf16   each draft's own keys / values; the newest
 *   v_cache  [Qn][K][C][Hkv][D] bf16     token is at position n_k - 1
 *   cache_len[Qn][K]            int32  n_k, 1 <= n_k <= C
 *   out      [Qn][K][Hq][D]     fp64
 *   lse      [Qn][K][Hq]        fp64 or NULL
 * For query qi, draft k, head h with kv head g = h / (Hq / Hkv):
 *   keys  S = { prefix j : 0 <= j < P_qi }  U  { own (k, t) : 0 <= t < n_k }
 *   out   = softmax(scale * q K_S^T) V_S,  lse as in oracle_verify_attn.
 * Readings: drafts never see one another's tokens (each a_i is drafted from its own
 * t_i, Eq. 5); cache positions at or past n_k are not read.
 * Returns 0, or -1 on bad arguments (including n_k outside [1, C]).
 */
int oracle_decode_attn(int Qn, int K, int C, int Hq, int Hkv, int D, double scale,
                       const uint16_t* q, const uint16_t* k_pre, const uint16_t* v_pre,
                       const int32_t* offs, const uint16_t* k_cache, const uint16_t* v_cache,
                       const int32_t* cache_len, double* out, double* lse) {
  if (Qn <= 0 || K <= 0 || C <= 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || Hq % Hkv) return -1;
  if (!q || !offs || !k_cache || !v_cache || !cache_len || !out) return -1;
  if (scale == 0.0) scale = 1.0 / sqrt((double)D);
  const int grp = Hq / Hkv;
  int maxP = 0;
  for (int qi = 0; qi < Qn; ++qi) {
    const int p = offs[qi + 1] - offs[qi];
    if (p < 0) return -1;
    if (p > maxP) maxP = p;
  }
  for (int64_t i = 0; i < (int64_t)Qn * K; ++i)
    if (cache_len[i] < 1 || cache_len[i] > C) return -1;
  if (maxP > 0 && (!k_pre || !v_pre)) return -1;
  const int64_t nrows = (int64_t)Qn * K * Hq;
  int bad = 0;
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)(maxP + C));
    double* qv = (double*)malloc(sizeof(double) * (size_t)D);
    double* acc = (double*)malloc(sizeof(double) * (size_t)D);
    if (!s || !qv || !acc) {
#pragma omp atomic write
      bad = 1;
    }
#pragma omp for schedule(dynamic, 4)
    for (int64_t r = 0; r < nrows; ++r) {
      if (bad) continue;
      const int h = (int)(r % Hq);
      const int64_t qk = r / Hq; /* qi*K + k */
      const int qi = (int)(qk / K);
      const int g = h / grp;
      const int P = offs[qi + 1] - offs[qi];
      const int n_own = cache_len[qk];
      for (int d = 0; d < D; ++d) qv[d] = dec_bf16(q[r * D + d]);
      int n = 0;
      for (int j = 0; j < P; ++j) {
        const uint16_t* kr = k_pre + ((int64_t)(offs[qi] + j) * Hkv + g) * D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d) dot += qv[d] * dec_bf16(kr[d]);
        s[n++] = scale * dot;
      }
      for (int t = 0; t < n_own; ++t) {
        const uint16_t* kr = k_cache + ((qk * C + t) * Hkv + g) * D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d) dot += qv[d] * dec_bf16(kr[d]);
        s[n++] = scale * dot;
      }
      double m = -INFINITY;
      for (int j = 0; j < n; ++j) if (s[j] > m) m = s[j];
      double Z = 0.0;
      for (int j = 0; j < n; ++j) Z += exp(s[j] - m);
      for (int d = 0; d < D; ++d) acc[d] = 0.0;
      int j = 0;
      for (; j < P; ++j) {
        const double p = exp(s[j] - m) / Z;
        const uint16_t* vr = v_pre + ((int64_t)(offs[qi] + j) * Hkv + g) * D;
        for (int d = 0; d < D; ++d) acc[d] += p * dec_bf16(vr[d]);
      }
      for (int t = 0; t < n_own; ++t, ++j) {
        const double p = exp(s[j] - m) / Z;
        const uint16_t* vr = v_cache + ((qk * C + t) * Hkv + g) * D;
        for (int d = 0; d < D; ++d) acc[d] += p * dec_bf16(vr[d]);
      }
      for (int d = 0; d < D; ++d) out[r * D + d] = acc[d];
      if (lse) lse[r] = m + log(Z);
    }
    free(s);
    free(qv);
    free(acc);
  }
  return bad ? -1 : 0;
}

/*
 * Verifier token log-probabilities at the candidate positions.
 *
 *   hidden  [M][H] bf16   final hidden state of each candidate row
 *   weight  [V][H] bf16   LM-head projection (one row per vocabulary entry)
 *   targets [M][G] int32  token ids whose log-probability is wanted
 *   logprob [M][G] fp64   z[m][t] - lse[m]; NaN when t is outside [0, V)
 *   lse     [M]    fp64 or NULL
 * z[m][v] = sum_h hidden[m][h] * weight[v][h]  (no bias, norm or temperature);
 * lse[m]  = max_v z + ln sum_v exp(z[m][v] - max_v z).
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int oracle_score_logprobs(int M, int H, int V, int G, const uint16_t* hidden,
                          const uint16_t* weight, const int32_t* targets, double* logprob,
                          double* lse) {
  if (M <= 0 || H <= 0 || V <= 0 || G < 0 || !hidden || !weight) return -1;
  if (G > 0 && (!targets || !logprob)) return -1;
  double* hd = (double*)malloc(sizeof(double) * (size_t)M * H);
  double* z = (double*)malloc(sizeof(double) * (size_t)M * V);
  if (!hd || !z) {
    free(hd);
    free(z);
    return -1;
  }
  for (int64_t i = 0; i < (int64_t)M * H; ++i) hd[i] = dec_bf16(hidden[i]);
  int bad = 0;
#pragma omp parallel
  {
    double* w = (double*)malloc(sizeof(double) * (size_t)H);
    if (!w) {
#pragma omp atomic write
      bad = 1;
    }
#pragma omp for schedule(static)
    for (int v = 0; v < V; ++v) {
      if (bad) continue;
      for (int h = 0; h < H; ++h) w[h] = dec_bf16(weight[(int64_t)v * H + h]);
      for (int m = 0; m < M; ++m) {
        const double* x = hd + (int64_t)m * H;
        double dot = 0.0;
        for (int h = 0; h < H; ++h) dot += x[h] * w[h];
        z[(int64_t)m * V + v] = dot;
      }
    }
    free(w);
  }
  if (!bad) {
#pragma omp parallel for schedule(static)
    for (int m = 0; m < M; ++m) {
      const double* zr = z + (int64_t)m * V;
      double mx = -INFINITY;
      for (int v = 0; v < V; ++v) if (zr[v] > mx) mx = zr[v];
      double s = 0.0;
      for (int v = 0; v < V; ++v) s += exp(zr[v] - mx);
      const double l = mx + log(s);
      if (lse) lse[m] = l;
      for (int g = 0; g < G; ++g) {
        const int32_t t = targets[(int64_t)m * G + g];
        logprob[(int64_t)m * G + g] = (t >= 0 && t < V) ? zr[t] - l : NAN;
      }
    }
  }
  free(hd);
  free(z);
  return bad ? -1 : 0;
}

/*
 * CLIP entity alignment (Eq. 14-15) with the keep threshold.
 *
 *   cand   [Qn][K][E] fp16   CLIP embedding of each candidate's entity e_k
 *   frames [Qn][F][E] fp16   CLIP embeddings of the query's keyframes
 *   cosm   [Qn][K][F] fp64 or NULL    cos(e_k, f_j)
 *   max_cos[Qn][K]    fp64            max_j cos(e_k, f_j)            (Eq. 15)
 *   argmax [Qn][K]    int32           smallest j attaining the max
 *   keep   [Qn][K]    uint8           max_cos >= tau
 * cos(a, b) = <a, b> / (|a| |b|), taken as 0 when either vector is zero.
 * Readings: the max runs over all frames given for the query (the keyframe set
 * F of Algorithm 1); ties go to the lowest frame index; keep uses >= like Eq. 13.
 */
int oracle_clip_align(int Qn, int K, int F, int E, double tau, const uint16_t* cand,
                      const uint16_t* frames, double* cosm, double* max_cos, int32_t* argmax,
                      uint8_t* keep) {
  if (Qn <= 0 || K <= 0 || F <= 0 || E <= 0 || !cand || !frames || !max_cos || !argmax || !keep)
    return -1;
#pragma omp parallel for schedule(static)
  for (int64_t qk = 0; qk < (int64_t)Qn * K; ++qk) {
    const int qi = (int)(qk / K);
    const uint16_t* e = cand + qk * E;
    double ee = 0.0;
    for (int i = 0; i < E; ++i) ee += dec_f16(e[i]) * dec_f16(e[i]);
    double best = -INFINITY;
    int besti = 0;
    for (int j = 0; j < F; ++j) {
      const uint16_t* f = frames + ((int64_t)qi * F + j) * E;
      double ef = 0.0, ff = 0.0;
      for (int i = 0; i < E; ++i) {
        ef += dec_f16(e[i]) * dec_f16(f[i]);
        ff += dec_f16(f[i]) * dec_f16(f[i]);
      }
      const double c = (ee > 0.0 && ff > 0.0) ? ef / (sqrt(ee) * sqrt(ff)) : 0.0;
      if (cosm) cosm[qk * F + j] = c;
      if (c > best) {
        best = c;
        besti = j;
      }
    }
    max_cos[qk] = best;
    argmax[qk] = besti;
    keep[qk] = best >= tau ? 1 : 0;
  }
  return 0;
}

/* SplitMix64 (Steele, Lea & Flood, OOPSLA 2014), counter form: output n of the
 * generator seeded with s is mix(s + (n+1) * 0x9E3779B97F4A7C15), mix being the
 * published finaliser.  Used for the Random selection baseline. */
static uint64_t oracle_splitmix64(uint64_t s, uint64_t n) {
  uint64_t z = s + (n + 1ULL) * 0x9E3779B97F4A7C15ULL;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/*
 * Candidate selection.
 *
 *   logprob [Qn][K][L][G] fp64   per-token log-probabilities (gather g)
 *   lengths [Qn][K] int32 or NULL  valid tokens n_k per candidate (default L)
 *   keep    [Qn][K] uint8          CLIP filter decision          (modes 0, 3)
 *   max_cos [Qn][K] fp64           alignment score of Eq. 15     (modes 1, 2, 5)
 *   score   [Qn][K] fp64           the per-candidate score of the mode
 *   selected[Qn]    int32          chosen candidate, or -1
 *
 * r_k = p_Y / (p_Y + p_N) = 1 / (1 + exp(lp_N - lp_Y)) is the reliability of Eq. 12,
 * with lp_Y = logprob[k][n_k-1][0] and lp_N = logprob[k][n_k-1][1] (the first
 * generated token after the candidate); a_k = max_cos[k] is the alignment of Eq. 15.
 * mode 0 (masked mean log-prob): score_k = (sum_{l < n_k} logprob[k][l][0]) / n_k,
 *   the verifier's own likelihood normalised by length (Section 4.6
 *   "self-consistent"); argmax over candidates with keep = 1, -1 if none.
 * mode 1 (Algorithm 1): score_k = r_k; Eq. 13 keeps A_H = { k : r_k >= max_j r_j - delta };
 *   the answer is the k in A_H with the largest a_k.
 * mode 2 (Section 4.6 "addition"): score_k = r_k + a_k, argmax over all.
 * mode 3 (Section 4.6 "invert"): filter by alignment (keep = 1), rank by reliability:
 *   score_k = r_k, argmax over kept, -1 if none.
 * mode 4 (Section 4.5 ablation "w/o ett"): score_k = r_k, argmax over all.
 * mode 5 (ablation "w/o rel"): score_k = a_k, argmax over all.
 * mode 6 (ablation "Random"): selected = floor(((x >> 32) * K) / 2^32) with x the q-th
 *   SplitMix64 output of `seed`; score_k = 0.
 * Ties go to the lowest index.  A candidate whose n_k is outside [1, L] or whose
 * score is NaN is never selected (modes 0-5).  In mode 1 a NaN a_k ranks below
 * every number (as -inf) when the best-aligned member of A_H is chosen.
 */
int oracle_select(int Qn, int K, int L, int G, int mode, double delta, const double* logprob,
                  const int32_t* lengths, const uint8_t* keep, const double* max_cos,
                  double* score, int32_t* selected, uint64_t seed) {
  if (Qn <= 0 || K <= 0 || L <= 0 || G <= 0 || !logprob || !score || !selected) return -1;
  if (mode < 0 || mode > 6) return -1;
  if ((mode == 0 || mode == 3) && !keep) return -1;
  if ((mode == 1 || mode == 2 || mode == 5) && !max_cos) return -1;
  if ((mode >= 1 && mode <= 4) && G < 2) return -1;
  for (int qi = 0; qi < Qn; ++qi) {
    for (int k = 0; k < K; ++k) {
      const int64_t qk = (int64_t)qi * K + k;
      const int n = lengths ? lengths[qk] : L;
      double sc = NAN;
      if (mode == 6) {
        sc = 0.0;
      } else if (n >= 1 && n <= L) {
        if (mode == 0) {
          double s = 0.0;
          for (int l = 0; l < n; ++l) s += logprob[(qk * L + l) * G + 0];
          sc = s / (double)n;
        } else if (mode == 5) {
          sc = max_cos[qk];
        } else {
          const double lpY = logprob[(qk * L + (n - 1)) * G + 0];
          const double lpN = logprob[(qk * L + (n - 1)) * G + 1];
          sc = 1.0 / (1.0 + exp(lpN - lpY));
          if (mode == 2) sc += max_cos[qk];
        }
      }
      score[qk] = sc;
    }
    int sel = -1;
    if (mode == 6) {
      const uint64_t x = oracle_splitmix64(seed, (uint64_t)qi);
      sel = (int)(((x >> 32) * (uint64_t)K) >> 32);
    } else if (mode == 1) {
      double top = -INFINITY;
      for (int k = 0; k < K; ++k) {
        const double s = score[(int64_t)qi * K + k];
        if (!isnan(s) && s > top) top = s;
      }
      double best = -INFINITY;
      for (int k = 0; k < K; ++k) {
        const int64_t qk = (int64_t)qi * K + k;
        const double s = score[qk];
        if (isnan(s) || !(s >= top - delta)) continue; /* Eq. 13 */
        /* a NaN alignment has no order: it ranks below every number */
        const double a = isnan(max_cos[qk]) ? -INFINITY : max_cos[qk];
        if (sel < 0 || a > best) {
          best = a;
          sel = k;
        }
      }
    } else {
      double best = -INFINITY;
      for (int k = 0; k < K; ++k) {
        const int64_t qk = (int64_t)qi * K + k;
        if (isnan(score[qk])) continue;
        if ((mode == 0 || mode == 3) && !keep[qk]) continue;
        if (sel < 0 || score[qk] > best) {
          best = score[qk];
          sel = k;
        }
      }
    }
    selected[qi] = sel;
  }
  return 0;
}

/*
 * Video-to-text retrieval, per keyframe (Eq. 2 and the retrieval loop of
 * Algorithm 1): for every keyframe f, the kf corpus texts t of largest
 * sim(f, t) = cos(CLIP(f), CLIP(t)).
 *
 *   frames  [Fr][E] fp16     CLIP image embeddings of the keyframes
 *   texts   [Nt][E] fp16     CLIP text embeddings of the document corpus
 *   top_idx [Fr][kf] int32   text ids, best first; -1 past the Nt-th entry
 *   top_sim [Fr][kf] fp64    their similarities; -inf where the id is -1
 * Order: larger similarity first, the smaller text id first among equal
 * similarities.  cos is 0 when either vector is zero.
 * Reading: the paper fixes K = 3 retrieved documents per query (Section 4.3)
 * but not the per-keyframe list length; kf is a parameter.
 */
int oracle_frame_topk(int Fr, int Nt, int E, int kf, const uint16_t* frames,
                      const uint16_t* texts, int32_t* top_idx, double* top_sim) {
  if (Fr < 0 || Nt <= 0 || E <= 0 || kf <= 0 || (Fr > 0 && (!frames || !top_idx || !top_sim)) ||
      !texts)
    return -1;
  double* tnorm = (double*)malloc(sizeof(double) * (size_t)Nt);
  if (!tnorm) return -2;
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < Nt; ++t) {
    double s = 0.0;
    for (int i = 0; i < E; ++i) s += dec_f16(texts[t * E + i]) * dec_f16(texts[t * E + i]);
    tnorm[t] = sqrt(s);
  }
  int err = 0;
#pragma omp parallel
  {
    double* sim = (double*)malloc(sizeof(double) * (size_t)Nt);
    if (!sim) {
#pragma omp atomic write
      err = -2;
    }
#pragma omp for schedule(dynamic, 1)
    for (int f = 0; f < Fr; ++f) {
      if (!sim) continue;
      const uint16_t* x = frames + (int64_t)f * E;
      double xx = 0.0;
      for (int i = 0; i < E; ++i) xx += dec_f16(x[i]) * dec_f16(x[i]);
      const double xn = sqrt(xx);
      for (int64_t t = 0; t < Nt; ++t) {
        const uint16_t* y = texts + t * E;
        double d = 0.0;
        for (int i = 0; i < E; ++i) d += dec_f16(x[i]) * dec_f16(y[i]);
        sim[t] = (xn > 0.0 && tnorm[t] > 0.0) ? d / (xn * tnorm[t]) : 0.0;
      }
      /* kf rounds of "best not yet taken"; scanning ids upwards with a strict >
       * keeps the smallest id among equal similarities */
      for (int r = 0; r < kf; ++r) {
        int32_t best = -1;
        for (int64_t t = 0; t < Nt; ++t) {
          int taken = 0;
          for (int p = 0; p < r; ++p)
            if (top_idx[(int64_t)f * kf + p] == (int32_t)t) taken = 1;
          if (taken) continue;
          if (best < 0 || sim[t] > sim[best]) best = (int32_t)t;
        }
        top_idx[(int64_t)f * kf + r] = best;
        top_sim[(int64_t)f * kf + r] = best >= 0 ? sim[best] : -INFINITY;
      }
    }
    free(sim);
  }
  free(tnorm);
  return err;
}

/*
 * Video-to-text retrieval, per query (Eq. 3): the texts the query's keyframes
 * retrieved form the set T; each text of T is scored by the largest similarity
 * with which one of those keyframes retrieved it, and the Kq best texts of T are
 * the query's external knowledge T*.
 *
 *   frame_offsets [Qn+1]  keyframes of query q: rows frame_offsets[q] .. frame_offsets[q+1]-1
 *   top_idx, top_sim [Fr][kf]  per-keyframe lists (oracle_frame_topk's layout;
 *                         entries with id -1 are ignored)
 *   out_idx [Qn][Kq] int32, out_sim [Qn][Kq] fp64: best first, the smaller id
 *                         first among equal scores; -1 / -inf past |T|
 * Reading: Eq. 3 writes sim(f, t) with f free; the f taken is the keyframe
 * that retrieved t (the best such keyframe when several did).
 */
int oracle_aggregate_topk(int Qn, int kf, int Kq, const int32_t* frame_offsets,
                          const int32_t* top_idx, const double* top_sim, int32_t* out_idx,
                          double* out_sim) {
  if (Qn <= 0 || kf <= 0 || Kq <= 0 || !frame_offsets || !out_idx || !out_sim) return -1;
  for (int q = 0; q < Qn; ++q)
    if (frame_offsets[q] < 0 || frame_offsets[q + 1] < frame_offsets[q]) return -1;
  for (int q = 0; q < Qn; ++q) {
    const int64_t e0 = (int64_t)frame_offsets[q] * kf, e1 = (int64_t)frame_offsets[q + 1] * kf;
    for (int r = 0; r < Kq; ++r) {
      int64_t best = -1;
      for (int64_t e = e0; e < e1; ++e) {
        const int32_t t = top_idx[e];
        if (t < 0) continue;
        int taken = 0;
        for (int p = 0; p < r; ++p)
          if (out_idx[(int64_t)q * Kq + p] == t) taken = 1;
        if (taken) continue;
        if (best < 0 || top_sim[e] > top_sim[best] ||
            (top_sim[e] == top_sim[best] && t < top_idx[best]))
          best = e;
      }
      out_idx[(int64_t)q * Kq + r] = best >= 0 ? top_idx[best] : -1;
      out_sim[(int64_t)q * Kq + r] = best >= 0 ? top_sim[best] : -INFINITY;
    }
  }
  return 0;
}

/*
 * Keyframe extraction (Eq. 1 and the first loop of Algorithm 1), with colour
 * histograms as the inter-frame similarity (Section 3.1).
 *
 *   pixels  [T][npix][3] uint8   RGB frames of Nv videos stored back to back
 *   video_offsets [Nv+1]         frames of video v: video_offsets[v] .. video_offsets[v+1]-1
 *   hist    [T][512] int32 or NULL  joint colour histogram with 8 levels per
 *                                channel: bin = 64 * (r / 32) + 8 * (g / 32) + b / 32
 *   sim     [T] fp64             sim(f_i, f_{i-1}) = sum_b min(h_i[b], h_{i-1}[b]) / npix
 *   is_key  [T] uint8            sim < theta (Eq. 1)
 *   key_index [T] int32          ids of the keyframes in frame order, video by video
 *   key_offsets [Nv+1] int32     keyframes of video v: key_index[key_offsets[v] ..]
 * Readings: the histogram is the joint RGB histogram above and the similarity is
 * its normalised intersection (1 for equal colour distributions, 0 for disjoint
 * ones); the previous frame of a video's first frame is empty, so its
 * similarity is 0 and it is always a keyframe (theta > 0); the comparison is
 * the strict < of Eq. 1, taken on the fp64 quotient.
 */
int oracle_keyframes(int Nv, int64_t npix, double theta, const int32_t* video_offsets,
                     const uint8_t* pixels, int32_t* hist, double* sim, uint8_t* is_key,
                     int32_t* key_index, int32_t* key_offsets) {
  if (Nv <= 0 || npix <= 0 || !video_offsets || !pixels || !sim || !is_key || !key_index ||
      !key_offsets || !(theta > 0.0))
    return -1;
  for (int v = 0; v < Nv; ++v)
    if (video_offsets[v] < 0 || video_offsets[v + 1] < video_offsets[v]) return -1;
  const int T = video_offsets[Nv];
  int32_t* h = hist ? hist : (int32_t*)malloc(sizeof(int32_t) * 512 * (size_t)(T > 0 ? T : 1));
  if (!h) return -2;
#pragma omp parallel for schedule(static)
  for (int i = 0; i < T; ++i) {
    int32_t* hi = h + (int64_t)i * 512;
    for (int b = 0; b < 512; ++b) hi[b] = 0;
    const uint8_t* p = pixels + (int64_t)i * npix * 3;
    for (int64_t x = 0; x < npix; ++x) {
      const int r = p[3 * x] / 32, g = p[3 * x + 1] / 32, b = p[3 * x + 2] / 32;
      hi[64 * r + 8 * g + b] += 1;
    }
  }
  int32_t nk = 0;
  for (int v = 0; v < Nv; ++v) {
    key_offsets[v] = nk;
    for (int i = video_offsets[v]; i < video_offsets[v + 1]; ++i) {
      int64_t inter = 0;
      if (i > video_offsets[v])
        for (int b = 0; b < 512; ++b) {
          const int32_t a = h[(int64_t)i * 512 + b], c = h[(int64_t)(i - 1) * 512 + b];
          inter += a < c ? a : c;
        }
      sim[i] = (double)inter / (double)npix;
      is_key[i] = sim[i] < theta ? 1 : 0;
      if (is_key[i]) key_index[nk++] = i;
    }
  }
  key_offsets[Nv] = nk;
  if (!hist) free(h);
  return 0;
}
