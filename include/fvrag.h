/*
 * libfvrag -- the verifier hot path of VideoSpeculateRAG (arXiv 2601.01513) on
 * one GB300 (sm_103a).
 *
 * The verifier of the paper scores K draft candidates that share one long
 * prefix (video tokens, question, retrieved passages) in a single forward pass
 * (Section 3.1, Eq. 6; Section 3.2 "Two-Stage Verification", Eq. 11), then
 * checks each candidate's entity against the video's keyframes with CLIP
 * (Eq. 14-15) and picks the answer (Eq. 7, Eq. 12-13, Algorithm 1).  This
 * library implements the data-parallel core of that step as four calls:
 *
 *   fvrag_verify_attn       one attention layer of the verifier forward over
 *                           all K x L candidate rows: the shared prefix is read
 *                           once for all candidates (split over the key axis),
 *                           plus each candidate's own causal tail;
 *   fvrag_score_logprobs    the LM head: hidden @ W^T fused with an online
 *                           log-sum-exp and a gather of the target ids, so the
 *                           [rows x vocab] logits never reach memory;
 *   fvrag_clip_align        cosine of each candidate-entity embedding with every
 *                           frame embedding, max/argmax over frames, keep flag;
 *   fvrag_select_candidate  the per-query selection reduction.
 *
 * the drafts' own decode step (Eq. 5, Eq. 8-10):
 *
 *   fvrag_decode_attn       each draft's newest token over the shared prefix and
 *                           its own cached tokens (the same kernel as above);
 *
 * and the two data-parallel steps before the drafts (Section 3.1, "Multimodal
 * Retrieval"; Algorithm 1's first two loops):
 *
 *   fvrag_keyframes         colour histograms of the video frames, similarity
 *                           with the previous frame, keyframe set (Eq. 1);
 *   fvrag_retrieve          CLIP cosine of every keyframe with every corpus text,
 *                           per-keyframe top-k and per-query top-K (Eq. 2-3).
 *
 * Conventions shared by every call
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     never allocates, frees or synchronises (except fvrag_read_status), and
 *     keeps no state between calls other than read-only driver entry points.
 *   - Every call validates its arguments on the host and returns an error
 *     before launching anything; on success it has only enqueued work on
 *     `stream` (NULL = the legacy default stream).
 *   - Layouts are dense row-major, leading index first, as written beside each
 *     argument.  bf16 / fp16 tensors are passed as `const void*`.
 *   - Workspaces: the first 256 bytes hold a 32-bit status word that kernels
 *     only ever OR error bits into (FVRAG_ERR_TIMEOUT when a bounded wait ran
 *     out).  Zero it once (fvrag_clear_status or a memset) before first use;
 *     read it with fvrag_read_status.  The rest is scratch owned by the call
 *     while it runs; calls that share a workspace must not overlap in time.
 *   - Alignment: every tensor pointer must be 16-byte aligned
 *     (FVRAG_ERR_MISALIGNED otherwise).
 *   - SM budgets (fvrag_attn_desc.sm_budget, fvrag_lm_desc.sm_budget): each of
 *     these kernels needs a whole SM per CTA (shared and tensor memory), so two
 *     of them share the GPU only when their grids together fit its SMs.  In a
 *     verify step whose LM head streams its weight from HBM (M <= 128 rows) the
 *     attention, which is bound by the tensor cores, can run on a few SMs beside
 *     it: give the LM head budget S - A and the attention budget A, and enqueue
 *     them on two streams.  A budget changes the grid and the key split, hence the
 *     rounding order of partial sums, never the operation computed; the workspace
 *     size depends on it (pass the same descriptor to the *_workspace call).
 *   - Tracing: with FVRAG_NVTX set in the environment (not "0"; read once, at the
 *     first call) every compute entry point wraps its work in an NVTX range named
 *     after it, so that Nsight Systems or ncu's NVTX filters group the kernels a
 *     call enqueues.  Without a profiler attached the ranges cost nothing.
 *   - fvrag_launch_count() counts the kernel launches the library has enqueued
 *     in this process (a launch captured into a CUDA graph counts once, at
 *     capture), so a caller can tell how many kernels one call or one captured
 *     step runs.
 */
#ifndef FVRAG_H
#define FVRAG_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define FVRAG_ABI_VERSION 6

/* cudaStream_t without including the CUDA headers. */
typedef struct CUstream_st* fvrag_stream_t;

typedef enum {
  FVRAG_OK = 0,
  FVRAG_ERR_INVALID_ARG = 1, /* null required pointer, non-positive size, bad mode */
  FVRAG_ERR_UNSUPPORTED = 2, /* shape outside what the kernels handle (see each call) */
  FVRAG_ERR_MISALIGNED = 3,  /* pointer not 16-byte aligned, row pitch not a multiple of 16 B */
  FVRAG_ERR_WORKSPACE = 4,   /* workspace pointer null or smaller than the *_workspace() size */
  FVRAG_ERR_CUDA = 5,        /* a CUDA runtime/driver call or a launch failed */
  FVRAG_ERR_TIMEOUT = 6      /* device status: a bounded wait inside a kernel ran out */
} fvrag_status;

/* FVRAG_ABI_VERSION of the loaded library. */
int fvrag_abi_version(void);

/* Kernel launches this library has enqueued since it was loaded (all devices and
 * threads; a launch into a capturing stream counts once, when it is captured). */
uint64_t fvrag_launch_count(void);

/* Static, never NULL, human-readable name of a status code. */
const char* fvrag_status_string(int status);

/* ------------------------------------------------------------------------ *
 * 1. Shared-prefix attention (verifier forward, Eq. 6 and Eq. 11)
 *
 * For query q, candidate k, candidate token l and query head h, with KV head
 * g = h / (hq / hkv) (consecutive query heads share a KV head):
 *   keys   = the P_q prefix tokens of query q, then tokens 0..l of candidate k
 *            (candidates never see one another; causal inside a candidate)
 *   out    = softmax(scale * q . K^T) V over those keys,   scale = softmax_scale
 *            or 1/sqrt(head_dim) when softmax_scale == 0
 *   lse    = natural-log log-sum-exp of the scaled scores (optional output)
 * ------------------------------------------------------------------------ */
typedef struct fvrag_attn_desc {
  int32_t num_queries;  /* Qn >= 1 */
  int32_t num_cand;     /* K >= 1 */
  int32_t cand_len;     /* L, 1..64 */
  int32_t hq;           /* query heads, multiple of hkv */
  int32_t hkv;          /* KV heads >= 1 */
  int32_t head_dim;     /* D: 64 or 128 */
  int32_t max_prefix;   /* upper bound on every P_q (plans the key split); >= 0 */
  int32_t total_prefix; /* sum over queries of P_q = rows of k_prefix / v_prefix */
  float softmax_scale;  /* > 0, or 0 => 1/sqrt(head_dim); negative / NaN / inf rejected */
  uint32_t flags;       /* 0 (the library picks the key split), or one FVRAG_ATTN_SPLIT_* */
  int32_t sm_budget;    /* SMs the key split is planned for: 0 = every SM of the current
                           device, else 1 .. that count (more: FVRAG_ERR_INVALID_ARG).  A
                           budget below the device's count leaves the other SMs to a call
                           running beside this one on another stream (see "SM budgets") */
} fvrag_attn_desc;

/* fvrag_attn_desc.flags: how the keys of every row tile (a group of candidate tokens x the
 * query heads of one KV head) are split over CTAs.  Every split gives the same result up to
 * the order of floating-point additions; with flags = 0 the library picks one by its cost
 * model.  Any other value: FVRAG_ERR_INVALID_ARG. */
#define FVRAG_ATTN_SPLIT_STATIC 1u  /* each tile's key list cut into equal runs, one CTA per run */
#define FVRAG_ATTN_SPLIT_STREAM 2u  /* one CTA per SM (of the budget), each an equal share of all
                                       tiles' key lists in tile order; needs num_queries <= 64,
                                       at most 64 tiles per KV head and query, and every P_q <=
                                       max_prefix, else FVRAG_ERR_UNSUPPORTED (and a workspace
                                       size of 0) */

/* Bytes of workspace fvrag_verify_attn needs for `d` (0 if `d` is invalid). */
size_t fvrag_verify_attn_workspace(const fvrag_attn_desc* d);

/*
 *   q              [Qn][K][L][hq][D]     bf16
 *   k_prefix       [total_prefix][hkv][D] bf16   query q owns rows
 *   v_prefix       [total_prefix][hkv][D] bf16     prefix_offsets[q] .. prefix_offsets[q+1]-1
 *   prefix_offsets [Qn+1]                int32  device; non-decreasing, offsets[0] = 0,
 *                                               offsets[Qn] = total_prefix, every
 *                                               P_q <= max_prefix (not checked on device)
 *   k_tail, v_tail [Qn][K][L][hkv][D]    bf16   the candidates' own tokens
 *   out            [Qn][K][L][hq][D]     bf16   written
 *   lse            [Qn][K][L][hq]        fp32   written when not NULL
 *   ws / ws_bytes  workspace of at least fvrag_verify_attn_workspace(d) bytes
 * k_prefix / v_prefix may be NULL when total_prefix == 0.
 */
fvrag_status fvrag_verify_attn(const fvrag_attn_desc* d, const void* q, const void* k_prefix,
                               const void* v_prefix, const int32_t* prefix_offsets,
                               const void* k_tail, const void* v_tail, void* out, float* lse,
                               void* ws, size_t ws_bytes, fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 1b. Drafter decode step (Eq. 5; the generation of e_i, r_i, a_i in Eq. 8-10)
 *
 * The K drafts of a query are generated in parallel from the shared prefix
 * (video tokens and question) followed by each draft's own tokens (its retrieved
 * text t_i, then what it has generated so far).  One call is one decode step:
 * for query q, draft k and query head h (KV head g = h / (hq / hkv)),
 *   keys   = the P_q prefix tokens of query q, then own slots 0 .. n_k - 1 of draft k
 *            (the newest token, whose K/V is already in slot n_k - 1, included;
 *            drafts never see one another's tokens)
 *   out    = softmax(scale * q . K^T) V,  lse as in fvrag_verify_attn.
 * Same kernel as fvrag_verify_attn: the prefix is read once for all drafts.
 * ------------------------------------------------------------------------ */
typedef struct fvrag_decode_desc {
  int32_t num_queries;  /* Qn >= 1 */
  int32_t num_drafts;   /* K >= 1 */
  int32_t cache_cap;    /* C >= 1: own-token slots per draft */
  int32_t hq;           /* query heads, multiple of hkv, hq / hkv <= 128 */
  int32_t hkv;          /* KV heads >= 1 */
  int32_t head_dim;     /* D: 64 or 128 */
  int32_t max_prefix;   /* upper bound on every P_q; >= 0 */
  int32_t total_prefix; /* sum over queries of P_q */
  float softmax_scale;  /* > 0, or 0 => 1/sqrt(head_dim) */
  uint32_t flags;       /* must be 0 */
} fvrag_decode_desc;

size_t fvrag_decode_attn_workspace(const fvrag_decode_desc* d);

/*
 *   q              [Qn][K][hq][D]        bf16   the newest token of each draft
 *   k_prefix, v_prefix, prefix_offsets   as in fvrag_verify_attn
 *   k_cache        [Qn][K][C][hkv][D]    bf16   each draft's own keys / values
 *   v_cache        [Qn][K][C][hkv][D]    bf16
 *   cache_len      [Qn][K]               int32  device; n_k in [1, C] (values outside are
 *                                               clamped to [0, C], not reported)
 *   out            [Qn][K][hq][D]        bf16   written
 *   lse            [Qn][K][hq]           fp32   written when not NULL
 *   ws / ws_bytes  workspace of at least fvrag_decode_attn_workspace(d) bytes
 * Slots at or past n_k are never read into the result (they may hold anything).
 */
fvrag_status fvrag_decode_attn(const fvrag_decode_desc* d, const void* q, const void* k_prefix,
                               const void* v_prefix, const int32_t* prefix_offsets,
                               const void* k_cache, const void* v_cache, const int32_t* cache_len,
                               void* out, float* lse, void* ws, size_t ws_bytes,
                               fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 2. LM-head log-probabilities (Eq. 11; the verifier likelihood of Section 4.6)
 *
 *   z[m][v]        = sum_h hidden[m][h] * weight[v][h]   (bf16 x bf16, fp32 accumulate)
 *   lse[m]         = log sum_v exp(z[m][v])              (natural log)
 *   logprob[m][g]  = z[m][targets[m][g]] - lse[m], NaN when the id is outside [0, V)
 * The [rows x vocab] logits are never written to memory.
 * ------------------------------------------------------------------------ */
typedef struct fvrag_lm_desc {
  int32_t rows;    /* M >= 1 (candidate token rows, (q, k, l) order) */
  int32_t hidden;  /* H >= 8, multiple of 8 (16-byte row pitch) */
  int32_t vocab;   /* V >= 1 */
  int32_t gathers; /* G: target ids per row, 1..8 (1: likelihood; 2: "Yes"/"No") */
  uint32_t flags;  /* must be 0 */
  int32_t sm_budget; /* most SMs the call's persistent grid occupies: 0 = every SM of the
                        current device, else 1 .. that count (more: FVRAG_ERR_INVALID_ARG);
                        see "SM budgets" */
} fvrag_lm_desc;

size_t fvrag_score_logprobs_workspace(const fvrag_lm_desc* d);

/*
 *   hidden  [M][H] bf16
 *   weight  [V][H] bf16   (nn.Linear layout: one row per vocabulary entry)
 *   targets [M][G] int32
 *   logprob [M][G] fp32   written
 *   lse     [M]    fp32   written when not NULL
 */
fvrag_status fvrag_score_logprobs(const fvrag_lm_desc* d, const void* hidden, const void* weight,
                                  const int32_t* targets, float* logprob, float* lse, void* ws,
                                  size_t ws_bytes, fvrag_stream_t stream);

/*
 * Allocation-free form of fvrag_score_logprobs (the paper has no counterpart:
 * this is a deployment aid).  For callers that cannot call cudaMalloc -- for
 * example a serving runtime whose device memory is owned by another allocator,
 * or code that must not allocate once it is running -- the scratch that the
 * workspace argument would hold lives instead in a fixed static device array
 * inside the library: 2,130,176 bytes per GPU that loads the library, held
 * until the process exits.  Same arguments, layouts and results as
 * fvrag_score_logprobs without ws / ws_bytes.
 *   - rows must be <= 1024 (gathers <= 8): larger shapes return
 *     FVRAG_ERR_UNSUPPORTED without enqueuing anything.
 *   - The first call on a device looks up the array's device address (with
 *     that device current) and caches it with the CUDA context it belongs to;
 *     make that first call before any stream capture.  After cudaDeviceReset
 *     (a new context) the next call looks the address up again.  No call
 *     allocates or frees memory.
 *   - Every call shares the one array and leaves its contents behind; each call
 *     clears the array's status word before its kernels run.  Calls that
 *     overlap on the GPU (other streams, other threads) race on the array:
 *     serialise them.
 *   - The return value reports host-side checks and launches only.  A device-side
 *     error (a bounded wait that ran out: FVRAG_ERR_TIMEOUT) lands in the array's
 *     status word; read it with fvrag_score_logprobs_noalloc_status before the
 *     next call clears it.
 */
fvrag_status fvrag_score_logprobs_noalloc(const fvrag_lm_desc* d, const void* hidden,
                                          const void* weight, const int32_t* targets,
                                          float* logprob, float* lse, fvrag_stream_t stream);

/*
 * Device-side status of the most recent fvrag_score_logprobs_noalloc call on the
 * current device (the counterpart of fvrag_read_status for the static array,
 * whose address the caller never sees).  Synchronises `stream`, then reads the
 * status word: FVRAG_OK, or FVRAG_ERR_TIMEOUT when a bounded wait ran out.
 * Allocates nothing.
 */
fvrag_status fvrag_score_logprobs_noalloc_status(fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 3. CLIP entity alignment (Eq. 14-15) with the keep/drop threshold
 *
 *   cos[q][k][f]  = <e_qk, f_qf> / (|e_qk| |f_qf|)   (0 when either vector is 0)
 *   max_cos[q][k] = max_f cos[q][k][f]                (Eq. 15)
 *   argmax[q][k]  = lowest f attaining the max
 *   keep[q][k]    = max_cos >= threshold
 * ------------------------------------------------------------------------ */
typedef struct fvrag_clip_desc {
  int32_t num_queries; /* Qn >= 1 */
  int32_t num_cand;    /* K >= 1 */
  int32_t num_frames;  /* F >= 1 */
  int32_t dim;         /* E: multiple of 8, 8..4096 */
  float threshold;     /* tau */
  uint32_t flags;      /* must be 0 */
} fvrag_clip_desc;

/*
 *   cand_emb  [Qn][K][E] fp16
 *   frame_emb [Qn][F][E] fp16
 *   cos       [Qn][K][F] fp32  written when not NULL
 *   max_cos   [Qn][K]    fp32  written
 *   argmax    [Qn][K]    int32 written
 *   keep      [Qn][K]    uint8 written
 */
fvrag_status fvrag_clip_align(const fvrag_clip_desc* d, const void* cand_emb,
                              const void* frame_emb, float* cos, float* max_cos, int32_t* argmax,
                              uint8_t* keep, fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 4. Candidate selection
 *
 * FVRAG_SEL_MASKED_MEAN_LOGPROB: score_k = (sum_{l < n_k} logprob[k][l][0]) / n_k
 *   (the verifier's own length-normalised likelihood, Section 4.6); selected =
 *   argmax over candidates with keep = 1, lowest index on ties, -1 if none.
 * FVRAG_SEL_TWO_STAGE (Algorithm 1): with lpY = logprob[k][n_k-1][0] and
 *   lpN = logprob[k][n_k-1][1], score_k = 1 / (1 + exp(lpN - lpY)) = pY/(pY+pN)
 *   (Eq. 12); A_H = {k : score_k >= max_j score_j - delta} (Eq. 13); selected =
 *   the k in A_H with the largest max_cos, lowest index on ties; a NaN max_cos
 *   ranks below every number there (as -inf), so it is chosen only when every
 *   member of A_H has a NaN alignment.
 * The other strategies the paper compares share the reliability r_k of Eq. 12 (the
 * TWO_STAGE score) and the alignment a_k = max_cos of Eq. 15:
 * FVRAG_SEL_ADDITION ("addition", Section 4.6, Table 3): score_k = r_k + a_k;
 *   selected = argmax over all candidates.
 * FVRAG_SEL_INVERT ("invert", Section 4.6, Table 3): filter by alignment first
 *   (keep_k = 1), then rank by reliability: score_k = r_k, argmax over kept, -1 if none.
 * FVRAG_SEL_RELIABILITY_ONLY ("w/o ett", Section 4.5, Table 2): score_k = r_k,
 *   argmax over all candidates.
 * FVRAG_SEL_ALIGNMENT_ONLY ("w/o rel", Table 2): score_k = a_k, argmax over all.
 * FVRAG_SEL_RANDOM ("Random", Table 2): selected[q] = floor(u_q * K) with
 *   u_q = (x_q >> 32) / 2^32 and x_q the q-th output of SplitMix64 seeded with
 *   `seed` (x_q = mix(seed + (q + 1) * 0x9E3779B97F4A7C15)); score_k = 0.
 * n_k = lengths[q][k] (or L when lengths is NULL); a candidate with n_k outside
 * [1, L] or a NaN score gets score NaN and is never selected.  Sums and the
 * comparisons run in fp64; score is rounded to fp32 on output.
 * ------------------------------------------------------------------------ */
typedef enum {
  FVRAG_SEL_MASKED_MEAN_LOGPROB = 0,
  FVRAG_SEL_TWO_STAGE = 1,
  FVRAG_SEL_ADDITION = 2,
  FVRAG_SEL_INVERT = 3,
  FVRAG_SEL_RELIABILITY_ONLY = 4,
  FVRAG_SEL_ALIGNMENT_ONLY = 5,
  FVRAG_SEL_RANDOM = 6
} fvrag_sel_mode;

typedef struct fvrag_select_desc {
  int32_t num_queries; /* Qn >= 1 */
  int32_t num_cand;    /* K, 1..1024 */
  int32_t cand_len;    /* L >= 1 */
  int32_t gathers;     /* G: innermost extent of logprob (>= 2 for the reliability modes) */
  int32_t mode;        /* fvrag_sel_mode */
  float delta;         /* Eq. 13 margin (the paper uses 0.05) */
  uint32_t flags;      /* must be 0 */
  uint64_t seed;       /* FVRAG_SEL_RANDOM only */
} fvrag_select_desc;

/*
 *   logprob  [Qn][K][L][G] fp32
 *   lengths  [Qn][K] int32, or NULL
 *   keep     [Qn][K] uint8  (required for MASKED_MEAN_LOGPROB and INVERT)
 *   max_cos  [Qn][K] fp32   (required for TWO_STAGE, ADDITION, ALIGNMENT_ONLY)
 *   score    [Qn][K] fp32   written
 *   selected [Qn]    int32  written
 */
fvrag_status fvrag_select_candidate(const fvrag_select_desc* d, const float* logprob,
                                    const int32_t* lengths, const uint8_t* keep,
                                    const float* max_cos, float* score, int32_t* selected,
                                    fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 5. Video-to-text retrieval (Eq. 2-3; the retrieval loop of Algorithm 1)
 *
 *   sim(f, t)        = <f, t> / (|f| |t|)   CLIP cosine (Eq. 2), 0 when either is 0
 *   frame list of f  = the k_frame texts of largest sim(f, t), best first, the
 *                      smaller text id first among equal similarities
 *   T_q              = the texts in the lists of query q's keyframes, each scored by
 *                      the largest similarity with which one of them retrieved it
 *   query list of q  = the k_query best texts of T_q (Eq. 3), same order; id -1 and
 *                      similarity -inf past |T_q|
 * The [keyframes x texts] similarity matrix is never written to memory.
 * ------------------------------------------------------------------------ */
typedef struct fvrag_retrieve_desc {
  int32_t num_queries;   /* Qn >= 1 */
  int32_t num_keyframes; /* Fr = frame_offsets[Qn], 0..2048, with
                            ceil(Fr / 128) * 128 * k_frame <= 4096 */
  int32_t num_texts;     /* Nt >= 1 */
  int32_t dim;           /* E >= 8, multiple of 8 (16-byte rows) */
  int32_t k_frame;       /* texts kept per keyframe, 1..8 */
  int32_t k_query;       /* texts kept per query, 1..64 (the paper retrieves 3) */
  uint32_t flags;        /* must be 0 */
} fvrag_retrieve_desc;

size_t fvrag_retrieve_workspace(const fvrag_retrieve_desc* d);

/*
 * inv_norm[r] = 1 / |x_r| (0 for a zero row) for an fp16 matrix x [rows][dim]
 * (dim a multiple of 8).  Computing the corpus norms is an index-build step: run
 * it once per corpus and pass the result to every fvrag_retrieve call.
 */
fvrag_status fvrag_embed_inv_norms(const void* x, int32_t rows, int32_t dim, float* inv_norm,
                                   fvrag_stream_t stream);

/*
 *   frame_emb      [Fr][E] fp16   keyframe CLIP image embeddings, query by query
 *   frame_offsets  [Qn+1]  int32  device; keyframes of query q are rows
 *                                 frame_offsets[q] .. frame_offsets[q+1]-1 (non-decreasing,
 *                                 offsets[0] = 0, offsets[Qn] = Fr; a query whose offsets
 *                                 fall outside [0, Fr] is treated as empty)
 *   text_emb       [Nt][E] fp16   corpus CLIP text embeddings
 *   text_inv_norm  [Nt]    fp32   from fvrag_embed_inv_norms, or NULL (then computed
 *                                 in the workspace on every call: one more corpus pass)
 *   frame_topk     [Fr][k_frame] int32, frame_topk_sim [Fr][k_frame] fp32: the
 *                                 per-keyframe lists, written when not NULL
 *   out_idx        [Qn][k_query] int32, out_sim [Qn][k_query] fp32: written
 * Similarities are fp32 from an fp32-accumulated fp16 dot product.
 */
fvrag_status fvrag_retrieve(const fvrag_retrieve_desc* d, const void* frame_emb,
                            const int32_t* frame_offsets, const void* text_emb,
                            const float* text_inv_norm, int32_t* frame_topk,
                            float* frame_topk_sim, int32_t* out_idx, float* out_sim, void* ws,
                            size_t ws_bytes, fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * 6. Keyframe extraction (Eq. 1; the first loop of Algorithm 1)
 *
 *   hist[i][b] = number of pixels of frame i in bin b of the joint RGB histogram
 *                with 8 levels per channel: b = 64 (r / 32) + 8 (g / 32) + b / 32
 *   sim[i]     = sum_b min(hist[i][b], hist[i-1][b]) / (height * width)
 *                (histogram intersection with the previous frame of the same video;
 *                0 for a video's first frame, which has no previous frame)
 *   is_key[i]  = sim[i] < theta (Eq. 1), the quotient and the comparison in fp64
 *   key_index  = ids of the frames with is_key = 1 in increasing order; the keyframes
 *                of video v are key_index[key_offsets[v] .. key_offsets[v+1]-1]
 * ------------------------------------------------------------------------ */
typedef struct fvrag_keyframe_desc {
  int32_t num_videos;   /* Nv >= 1 */
  int32_t total_frames; /* T = video_offsets[Nv] >= 0 */
  int32_t height;       /* >= 1 */
  int32_t width;        /* >= 1; height * width a multiple of 16 (frames start on 16 B) */
  double theta;         /* > 0 */
  uint32_t flags;       /* must be 0 */
} fvrag_keyframe_desc;

size_t fvrag_keyframes_workspace(const fvrag_keyframe_desc* d);

/*
 *   pixels        [T][height][width][3] uint8  RGB, videos back to back
 *   video_offsets [Nv+1] int32  device; frames of video v are video_offsets[v] ..
 *                               video_offsets[v+1]-1 (non-decreasing, offsets[0] = 0,
 *                               offsets[Nv] = T; not checked on the device)
 *   hist          [T][512] int32  written when not NULL (else kept in the workspace)
 *   sim           [T] fp32   written (the fp64 quotient rounded to fp32)
 *   is_key        [T] uint8  written
 *   key_index     [T] int32  the first key_offsets[Nv] entries written
 *   key_offsets   [Nv+1] int32  written
 */
fvrag_status fvrag_keyframes(const fvrag_keyframe_desc* d, const uint8_t* pixels,
                             const int32_t* video_offsets, int32_t* hist, float* sim,
                             uint8_t* is_key, int32_t* key_index, int32_t* key_offsets, void* ws,
                             size_t ws_bytes, fvrag_stream_t stream);

/* ------------------------------------------------------------------------ *
 * Device status (failure detection without faulting the GPU)
 * ------------------------------------------------------------------------ */

/* Synchronises `stream`, then returns the status word stored in `ws`
 * (FVRAG_OK, or the error a kernel recorded), or FVRAG_ERR_CUDA if the copy failed. */
fvrag_status fvrag_read_status(const void* ws, fvrag_stream_t stream);

/* Enqueues a reset of the status word in `ws` to FVRAG_OK. */
fvrag_status fvrag_clear_status(void* ws, fvrag_stream_t stream);

/* Limit, in nanoseconds, of every bounded wait inside the kernels launched
 * after this call (default 1e9 = one second; clamped to >= 1000). */
void fvrag_set_wait_limit_ns(uint64_t ns);
uint64_t fvrag_get_wait_limit_ns(void);

/* Diagnostic: launches one CTA that waits, with the bounded wait every kernel
 * uses, on a shared-memory barrier that nothing ever completes.  The wait runs
 * out after the current wait limit and records FVRAG_ERR_TIMEOUT in `ws`'s
 * status word; the kernel then returns normally and the context stays usable. */
fvrag_status fvrag_selftest_wait_timeout(void* ws, fvrag_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* FVRAG_H */
