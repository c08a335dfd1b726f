"""Seeded synthetic workloads for the verifier hot path (input construction only).

The random numbers come from ``synth.c`` (counter-based SplitMix64 -> Box-Muller,
see its header for the exact definition).  This module only arranges them into
the tensors one verify step consumes; it contains none of the arithmetic of the
method (no attention, no log-softmax, no cosine filter, no selection), so the
CUDA path and the fp64 oracle can both take their inputs from here without
sharing any code of the computation.

Layouts (row-major, leading index first):
  q        [Qn][K][L][Hq][D]  bf16   ~N(0,1)
  k_prefix [sum P_q][Hkv][D]  bf16   ~N(0,1), ragged over queries via prefix_offsets
  v_prefix [sum P_q][Hkv][D]  bf16   ~N(0,1)
  prefix_offsets [Qn+1]       int32
  k_tail   [Qn][K][L][Hkv][D] bf16   ~N(0,1)
  v_tail   [Qn][K][L][Hkv][D] bf16   ~N(0,1)
  hidden   [M][H]             bf16   ~N(0,1),   M = Qn*K*L in (q, k, l) order
  weight   [V][H]             bf16   ~N(0, w_std)
  targets  [M][G]             int32  ~U[0, V)
  cand_emb [Qn][K][E]         fp16
  frame_emb[Qn][F][E]         fp16
bf16/fp16 tensors are returned as numpy uint16 bit patterns.

CLIP embeddings: independent Gaussian E-dimensional vectors have cosines of
about N(0, 1/sqrt(E)), so their max over F frames stays near 0.1, below the
keep threshold 0.2, and every candidate would be dropped.  The recipe plants
structure: for ceil(K/2) candidates per query (chosen by a seeded permutation)
one seeded frame is replaced by  c*e_hat + sqrt(1-c^2)*n_hat  with
c ~ U(0.25, 0.6) (kept), and one more candidate gets a near miss with
c ~ U(0.10, 0.18) (dropped); n_hat is the frame's own Gaussian draw made
orthogonal to e_hat.  Unit-normalised configs are then normalised before fp16
rounding; the others are rescaled to N(0,1)-like norms (sqrt(E)).
"""
import ctypes
import math
import os

import numpy as np

from .configs import DecodeConfig, KeyframeConfig, RetrievalConfig, VerifyConfig

_HERE = os.path.dirname(os.path.abspath(__file__))
SYNTH_SO = os.path.join(_HERE, "libfvrag_synth.so")

# stream ids (one independent SplitMix64 stream per tensor)
S_Q, S_KP, S_VP, S_KT, S_VT, S_HID, S_W, S_TGT = 1, 2, 3, 4, 5, 6, 7, 8
S_CAND, S_FRAME, S_PLEN, S_PERM, S_PFRAME, S_PC = 9, 10, 11, 12, 13, 14
S_LOGPROB, S_KEEP, S_MAXCOS, S_LEN = 20, 21, 22, 23
S_RT_NKF, S_RT_TEXT, S_RT_FRAME, S_RT_REL, S_RT_PICK, S_RT_C = 30, 31, 32, 33, 34, 35
S_DC_Q, S_DC_KP, S_DC_VP, S_DC_KC, S_DC_VC, S_DC_LEN, S_DC_PLEN = 50, 51, 52, 53, 54, 55, 56
S_KF_LEN, S_KF_SCENE, S_KF_CUT, S_KF_FADE, S_KF_PARAM, S_KF_NOISE = 40, 41, 42, 43, 44, 45

_lib = None


def build_synth(force: bool = False) -> str:
    """Compile synth.c into libfvrag_synth.so next to it (gcc, OpenMP)."""
    src = os.path.join(_HERE, "synth.c")
    if force or not os.path.exists(SYNTH_SO) or os.path.getmtime(SYNTH_SO) < os.path.getmtime(src):
        import subprocess
        tmp = SYNTH_SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=gnu11",
                               src, "-o", tmp, "-lm"])
        os.replace(tmp, SYNTH_SO)
    return SYNTH_SO


def _L():
    global _lib
    if _lib is None:
        build_synth()
        lib = ctypes.CDLL(SYNTH_SO)
        u64, i64, vp, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p, ctypes.c_double
        lib.synth_stream_key.restype = u64
        lib.synth_stream_key.argtypes = [u64, u64]
        lib.synth_raw.restype = u64
        lib.synth_raw.argtypes = [u64, u64]
        lib.synth_normal.restype = dbl
        lib.synth_normal.argtypes = [u64, u64]
        for name in ("synth_fill_normal_f64", "synth_fill_normal_bf16"):
            getattr(lib, name).argtypes = [vp, i64, u64, dbl, dbl]
            getattr(lib, name).restype = None
        lib.synth_fill_uniform_f64.argtypes = [vp, i64, u64, dbl, dbl]
        lib.synth_fill_uniform_f64.restype = None
        lib.synth_fill_uniform_i32.argtypes = [vp, i64, u64, i64, i64]
        lib.synth_fill_uniform_i32.restype = None
        lib.synth_round_f16.argtypes = [vp, vp, i64]
        lib.synth_round_f16.restype = None
        lib.synth_round_bf16.argtypes = [vp, vp, i64]
        lib.synth_round_bf16.restype = None
        lib.synth_fill_unit_rows_f16.argtypes = [vp, i64, ctypes.c_int, u64]
        lib.synth_fill_unit_rows_f16.restype = None
        lib.synth_video_frames.argtypes = [vp] + [ctypes.c_int] * 3 + [u64] + [vp] * 5
        lib.synth_video_frames.restype = None
        _lib = lib
    return _lib


def stream_key(seed: int, stream: int) -> int:
    return _L().synth_stream_key(seed & (2**64 - 1), stream)


def normal_bf16(shape, seed, stream, mean=0.0, std=1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    _L().synth_fill_normal_bf16(out.ctypes.data, out.size, stream_key(seed, stream), mean, std)
    return out


def normal_f64(shape, seed, stream, mean=0.0, std=1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    _L().synth_fill_normal_f64(out.ctypes.data, out.size, stream_key(seed, stream), mean, std)
    return out


def uniform_f64(shape, seed, stream, a=0.0, b=1.0) -> np.ndarray:
    out = np.empty(shape, dtype=np.float64)
    _L().synth_fill_uniform_f64(out.ctypes.data, out.size, stream_key(seed, stream), a, b)
    return out


def uniform_i32(shape, seed, stream, lo, hi) -> np.ndarray:
    """Integers uniform in [lo, hi)."""
    out = np.empty(shape, dtype=np.int32)
    _L().synth_fill_uniform_i32(out.ctypes.data, out.size, stream_key(seed, stream), lo, hi)
    return out


def round_f16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    _L().synth_round_f16(x.ctypes.data, out.ctypes.data, x.size)
    return out


def round_bf16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    _L().synth_round_bf16(x.ctypes.data, out.ctypes.data, x.size)
    return out


def prefix_lengths(cfg: VerifyConfig, seed=None) -> np.ndarray:
    seed = cfg.seed if seed is None else seed
    if cfg.prefix_range is None:
        return np.full(cfg.num_queries, cfg.prefix_len, dtype=np.int32)
    lo, hi = cfg.prefix_range
    return uniform_i32((cfg.num_queries,), seed, S_PLEN, lo, hi + 1)


def clip_embeddings(cfg: VerifyConfig, seed=None):
    """Candidate-entity and frame embeddings with the planted structure described above."""
    seed = cfg.seed if seed is None else seed
    Qn, K, F, E = cfg.num_queries, cfg.num_cand, cfg.num_frames, cfg.clip_dim
    cand = normal_f64((Qn, K, E), seed, S_CAND)
    frames = normal_f64((Qn, F, E), seed, S_FRAME)
    perm_keys = uniform_f64((Qn, K), seed, S_PERM)
    pframe = uniform_i32((Qn, K), seed, S_PFRAME, 0, F)
    pc = uniform_f64((Qn, K), seed, S_PC)
    n_strong = (K + 1) // 2
    for qi in range(Qn):
        order = np.argsort(perm_keys[qi], kind="stable")
        used = set()
        for rank, k in enumerate(order):
            if rank < n_strong:
                c = 0.25 + 0.35 * pc[qi, k]
            elif rank == n_strong:
                c = 0.10 + 0.08 * pc[qi, k]
            else:
                continue
            j = int(pframe[qi, k])
            while j in used:                      # one planted frame per candidate
                j = (j + 1) % F
                if len(used) >= F:
                    break
            if len(used) >= F:
                break
            used.add(j)
            e_hat = cand[qi, k] / np.linalg.norm(cand[qi, k])
            n = frames[qi, j] - np.dot(frames[qi, j], e_hat) * e_hat
            n_hat = n / np.linalg.norm(n)
            frames[qi, j] = (c * e_hat + math.sqrt(1.0 - c * c) * n_hat) * np.linalg.norm(frames[qi, j])
    if cfg.clip_unit:
        cand = cand / np.linalg.norm(cand, axis=-1, keepdims=True)
        frames = frames / np.linalg.norm(frames, axis=-1, keepdims=True)
    return round_f16(cand), round_f16(frames)


def make_inputs(cfg: VerifyConfig, seed=None, parts=("attn", "lm", "clip")) -> dict:
    """All tensors of one verify step, as numpy arrays (bf16/fp16 as uint16 bits)."""
    seed = cfg.seed if seed is None else seed
    Qn, K, L = cfg.num_queries, cfg.num_cand, cfg.cand_len
    Hq, Hkv, D = cfg.hq, cfg.hkv, cfg.head_dim
    out = {}
    if "attn" in parts:
        plen = prefix_lengths(cfg, seed)
        offs = np.zeros(Qn + 1, dtype=np.int32)
        offs[1:] = np.cumsum(plen)
        total = int(offs[-1])
        out["prefix_offsets"] = offs
        out["q"] = normal_bf16((Qn, K, L, Hq, D), seed, S_Q)
        out["k_prefix"] = normal_bf16((total, Hkv, D), seed, S_KP)
        out["v_prefix"] = normal_bf16((total, Hkv, D), seed, S_VP)
        out["k_tail"] = normal_bf16((Qn, K, L, Hkv, D), seed, S_KT)
        out["v_tail"] = normal_bf16((Qn, K, L, Hkv, D), seed, S_VT)
    if "lm" in parts:
        M = cfg.rows
        out["hidden"] = normal_bf16((M, cfg.hidden), seed, S_HID)
        out["weight"] = normal_bf16((cfg.vocab, cfg.hidden), seed, S_W, 0.0, cfg.w_std)
        out["targets"] = uniform_i32((M, cfg.gathers), seed, S_TGT, 0, cfg.vocab)
    if "clip" in parts:
        out["cand_emb"], out["frame_emb"] = clip_embeddings(cfg, seed)
    return out


def selection_inputs(num_queries, num_cand, cand_len, gathers, seed, std=1.0):
    """Synthetic per-token log-probs / keep / max_cos for the selection step alone.

    Log-probs are -|N(0, std)| - 1 rounded to fp32 (so they are <= 0 like real
    log-probabilities); keep is a seeded coin flip; max_cos ~ U(-0.2, 0.8) in fp32.
    """
    lp = -np.abs(normal_f64((num_queries, num_cand, cand_len, gathers), seed, S_LOGPROB, 0.0, std)) - 1.0
    keep = (uniform_f64((num_queries, num_cand), seed, S_KEEP) < 0.6).astype(np.uint8)
    mc = uniform_f64((num_queries, num_cand), seed, S_MAXCOS, -0.2, 0.8)
    return lp.astype(np.float32), keep, mc.astype(np.float32)


def decode_inputs(cfg: DecodeConfig, seed=None) -> dict:
    """One drafter decode step: q [Qn][K][hq][D], prefix K/V [sum P][hkv][D] with
    prefix_offsets [Qn+1], own caches [Qn][K][C][hkv][D] (all N(0,1) bf16) and
    cache_len [Qn][K] ~ U[cache_range]."""
    seed = cfg.seed if seed is None else seed
    Qn, K, C = cfg.num_queries, cfg.num_drafts, cfg.cache_cap
    if cfg.prefix_range is None:
        plen = np.full(Qn, cfg.prefix_len, dtype=np.int32)
    else:
        plen = uniform_i32((Qn,), seed, S_DC_PLEN, cfg.prefix_range[0], cfg.prefix_range[1] + 1)
    offs = np.zeros(Qn + 1, dtype=np.int32)
    offs[1:] = np.cumsum(plen)
    tot = int(offs[-1])
    lo, hi = cfg.cache_range
    return {
        "q": normal_bf16((Qn, K, cfg.hq, cfg.head_dim), seed, S_DC_Q),
        "k_prefix": normal_bf16((tot, cfg.hkv, cfg.head_dim), seed, S_DC_KP),
        "v_prefix": normal_bf16((tot, cfg.hkv, cfg.head_dim), seed, S_DC_VP),
        "prefix_offsets": offs,
        "k_cache": normal_bf16((Qn, K, C, cfg.hkv, cfg.head_dim), seed, S_DC_KC),
        "v_cache": normal_bf16((Qn, K, C, cfg.hkv, cfg.head_dim), seed, S_DC_VC),
        "cache_len": uniform_i32((Qn, K), seed, S_DC_LEN, lo, hi + 1),
    }


def unit_rows_f16(rows, dim, seed, stream) -> np.ndarray:
    """[rows][dim] fp16 bit patterns of unit-length Gaussian directions."""
    out = np.empty((rows, dim), dtype=np.uint16)
    _L().synth_fill_unit_rows_f16(out.ctypes.data, rows, dim, stream_key(seed, stream))
    return out


def retrieval_inputs(cfg: RetrievalConfig, seed=None) -> dict:
    """Keyframe and corpus embeddings for video-to-text retrieval (Eq. 2-3).

    texts [Nt][E] fp16 unit vectors; frames [Fr][E] fp16 unit vectors with
    frame_offsets [Qn+1].  Each query gets ``cfg.relevant`` relevant text ids; each
    of its keyframes, with probability 1/2, is replaced by
    c*t_hat + sqrt(1-c^2)*n_hat with t_hat one of those texts (decoded from fp16),
    c ~ U(0.25, 0.5) and n_hat the keyframe's own draw made orthogonal to t_hat.
    Unplanted pairs have cosines of about N(0, 1/sqrt(E)), so a keyframe's best
    background text over a million sits near 0.18.
    """
    seed = cfg.seed if seed is None else seed
    Qn, E = cfg.num_queries, cfg.dim
    lo, hi = cfg.keyframes_range
    nkf = uniform_i32((Qn,), seed, S_RT_NKF, lo, hi + 1)
    offs = np.zeros(Qn + 1, dtype=np.int32)
    offs[1:] = np.cumsum(nkf)
    Fr = int(offs[-1])
    texts = unit_rows_f16(cfg.num_texts, E, seed, S_RT_TEXT)
    frames = normal_f64((Fr, E), seed, S_RT_FRAME)
    rel = uniform_i32((Qn, cfg.relevant), seed, S_RT_REL, 0, cfg.num_texts)
    pick = uniform_f64((Fr,), seed, S_RT_PICK)
    cs = uniform_f64((Fr,), seed, S_RT_C, 0.25, 0.5)
    for q in range(Qn):
        for f in range(int(offs[q]), int(offs[q + 1])):
            if pick[f] >= 0.5:
                continue
            t = int(rel[q, int(pick[f] * 2 * cfg.relevant) % cfg.relevant])
            t_hat = texts[t].view(np.float16).astype(np.float64)
            t_hat = t_hat / np.linalg.norm(t_hat)
            n = frames[f] - np.dot(frames[f], t_hat) * t_hat
            c = cs[f]
            frames[f] = c * t_hat + math.sqrt(1.0 - c * c) * n / np.linalg.norm(n)
    frames = frames / np.linalg.norm(frames, axis=-1, keepdims=True)
    return {"frames": round_f16(frames), "frame_offsets": offs, "texts": texts, "relevant": rel}


def video_timeline(cfg: KeyframeConfig, seed=None):
    """Per-frame scene schedule of ``cfg.num_videos`` videos.

    Returns (video_offsets [Nv+1], fa [T], fb [T], fw [T], ftau [T], scenes [S][17]).
    Scene lengths are max(8, round(-scene_mean * ln u)); at each scene change a
    fade of 8-15 frames (with probability fade_prob) blends the old scene into the
    new one linearly, otherwise the cut is hard.
    """
    seed = cfg.seed if seed is None else seed
    lo, hi = cfg.frames_range
    nfr = uniform_i32((cfg.num_videos,), seed, S_KF_LEN, lo, hi + 1)
    voffs = np.zeros(cfg.num_videos + 1, dtype=np.int32)
    voffs[1:] = np.cumsum(nfr)
    T = int(voffs[-1])
    ucut = uniform_f64((T + 1,), seed, S_KF_CUT)
    ufade = uniform_f64((T + 1, 2), seed, S_KF_FADE)
    fa = np.zeros(T, np.int32)
    fb = np.zeros(T, np.int32)
    fw = np.zeros(T, np.float64)
    ftau = np.zeros(T, np.float64)
    scene = -1
    draws = 0
    for v in range(cfg.num_videos):
        t = int(voffs[v])
        end = int(voffs[v + 1])
        prev = -1
        while t < end:
            scene += 1
            n = max(8, int(round(-cfg.scene_mean * math.log(max(ucut[draws], 1e-300)))))
            fade = prev >= 0 and ufade[draws, 0] < cfg.fade_prob
            nf = 8 + int(ufade[draws, 1] * 8) if fade else 0
            draws += 1
            for i in range(n):
                if t >= end:
                    break
                fa[t], ftau[t] = scene, float(i)
                if i < nf:
                    # fade from the previous scene (continuing its clock) into this one
                    fa[t], fb[t], fw[t] = prev, scene, (i + 1) / (nf + 1)
                    ftau[t] = float(i)
                t += 1
            prev = scene
    S = scene + 1
    u = uniform_f64((S, 17), seed, S_KF_PARAM)
    scenes = np.empty((S, 17), np.float64)
    scenes[:, 0:9] = u[:, 0:9] * 255.0                       # c0, c1, c2
    scenes[:, 9] = u[:, 9] * 2.0 * math.pi                   # gradient angle
    scenes[:, 10] = (u[:, 10] - 0.5) * 0.02                  # drift, cycles per frame
    scenes[:, 11:13] = u[:, 11:13]                           # disc centre
    scenes[:, 13:15] = (u[:, 13:15] - 0.5) * 0.01            # disc velocity per frame
    scenes[:, 15] = 0.05 + 0.2 * u[:, 15]                    # disc radius (fraction of height)
    scenes[:, 16] = 2.0 + 8.0 * u[:, 16]                     # noise amplitude
    return voffs, fa, fb, fw, ftau, scenes


def video_frames(cfg: KeyframeConfig, seed=None, out=None):
    """RGB frames [T][H][W][3] uint8 of the videos of ``video_timeline`` and the offsets."""
    seed = cfg.seed if seed is None else seed
    voffs, fa, fb, fw, ftau, scenes = video_timeline(cfg, seed)
    T = int(voffs[-1])
    if out is None:
        out = np.empty((T, cfg.height, cfg.width, 3), dtype=np.uint8)
    assert out.shape == (T, cfg.height, cfg.width, 3) and out.dtype == np.uint8 and out.flags.c_contiguous
    _L().synth_video_frames(out.ctypes.data, T, cfg.height, cfg.width, stream_key(seed, S_KF_NOISE),
                            fa.ctypes.data, fb.ctypes.data, fw.ctypes.data, ftau.ctypes.data,
                            np.ascontiguousarray(scenes).ctypes.data)
    return out, voffs


def bf16_bits_to_f32(x: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to fp32 (for test-side printing)."""
    return (x.astype(np.uint32) << 16).view(np.float32)


def f16_bits_to_f32(x: np.ndarray) -> np.ndarray:
    return x.view(np.float16).astype(np.float32)
