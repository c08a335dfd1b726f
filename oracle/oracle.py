"""Python handle on the fp64 oracle (``fvrag_oracle.c``) -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` use this module.  It imports nothing from the product package; it
receives plain numpy arrays (bf16/fp16 as uint16 bit patterns) and returns fp64
results.  See the C file for the definitions and the passages they follow.
"""
import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(_HERE, "fvrag_oracle.c")
SO = os.path.join(_HERE, "libfvrag_oracle.so")
_lib = None

SEL_MASKED_MEAN_LOGPROB = 0
SEL_TWO_STAGE = 1
SEL_ADDITION = 2
SEL_INVERT = 3
SEL_RELIABILITY_ONLY = 4
SEL_ALIGNMENT_ONLY = 5
SEL_RANDOM = 6


def build(force: bool = False) -> str:
    if force or not os.path.exists(SO) or os.path.getmtime(SO) < os.path.getmtime(SRC):
        tmp = SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-std=gnu11",
                               SRC, "-o", tmp, "-lm"])
        os.replace(tmp, SO)
    return SO


def _L():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(SO)
        vp, ci, cd = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
        lib.oracle_max_threads.restype = ci
        lib.oracle_set_threads.argtypes = [ci]
        lib.oracle_verify_attn.argtypes = [ci] * 6 + [cd] + [vp] * 9
        lib.oracle_verify_attn.restype = ci
        lib.oracle_score_logprobs.argtypes = [ci] * 4 + [vp] * 5
        lib.oracle_score_logprobs.restype = ci
        lib.oracle_clip_align.argtypes = [ci] * 4 + [cd] + [vp] * 6
        lib.oracle_clip_align.restype = ci
        lib.oracle_select.argtypes = [ci] * 5 + [cd] + [vp] * 6 + [ctypes.c_uint64]
        lib.oracle_select.restype = ci
        lib.oracle_decode_attn.argtypes = [ci] * 6 + [cd] + [vp] * 9
        lib.oracle_decode_attn.restype = ci
        lib.oracle_frame_topk.argtypes = [ci] * 4 + [vp] * 4
        lib.oracle_frame_topk.restype = ci
        lib.oracle_aggregate_topk.argtypes = [ci] * 3 + [vp] * 5
        lib.oracle_aggregate_topk.restype = ci
        lib.oracle_keyframes.argtypes = [ci, ctypes.c_int64, cd] + [vp] * 7
        lib.oracle_keyframes.restype = ci
        lib.oracle_decode_bf16.argtypes = [vp, vp, ctypes.c_int64]
        lib.oracle_decode_f16.argtypes = [vp, vp, ctypes.c_int64]
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data


def _c(a, dt):
    return None if a is None else np.ascontiguousarray(a, dtype=dt)


def max_threads() -> int:
    return _L().oracle_max_threads()


def set_threads(n: int) -> None:
    _L().oracle_set_threads(n)


def decode_bf16(bits: np.ndarray) -> np.ndarray:
    bits = _c(bits, np.uint16)
    out = np.empty(bits.shape, np.float64)
    _L().oracle_decode_bf16(_p(bits), _p(out), bits.size)
    return out


def decode_f16(bits: np.ndarray) -> np.ndarray:
    bits = _c(bits, np.uint16)
    out = np.empty(bits.shape, np.float64)
    _L().oracle_decode_f16(_p(bits), _p(out), bits.size)
    return out


def verify_attn(q, k_prefix, v_prefix, prefix_offsets, k_tail, v_tail, scale=0.0, row_sel=None):
    """Attention over shared prefix + own causal tail.  q: [Qn][K][L][Hq][D] uint16 (bf16 bits).

    Returns (out [Qn][K][L][Hq][D] fp64, lse [Qn][K][L][Hq] fp64); rows not selected
    by ``row_sel`` ([Qn][K][L][Hq] bool) are left as NaN.
    """
    Qn, K, L, Hq, D = q.shape
    Hkv = k_tail.shape[3]
    q, kt, vt = _c(q, np.uint16), _c(k_tail, np.uint16), _c(v_tail, np.uint16)
    kp, vp_ = _c(k_prefix, np.uint16), _c(v_prefix, np.uint16)
    offs = _c(prefix_offsets, np.int32)
    sel = None if row_sel is None else _c(row_sel, np.uint8)
    out = np.full(q.shape, np.nan)
    lse = np.full(q.shape[:-1], np.nan)
    rc = _L().oracle_verify_attn(Qn, K, L, Hq, Hkv, D, float(scale), _p(q),
                                 _p(kp) if kp is not None and kp.size else None,
                                 _p(vp_) if vp_ is not None and vp_.size else None,
                                 _p(offs), _p(kt), _p(vt), _p(sel), _p(out), _p(lse))
    if rc != 0:
        raise ValueError("oracle_verify_attn: bad arguments")
    return out, lse


def decode_attn(q, k_prefix, v_prefix, prefix_offsets, k_cache, v_cache, cache_len, scale=0.0):
    """One drafter decode step.  q [Qn][K][Hq][D]; caches [Qn][K][C][Hkv][D] (bf16 bits);
    cache_len [Qn][K].  Returns (out [Qn][K][Hq][D] fp64, lse [Qn][K][Hq] fp64)."""
    Qn, K, Hq, D = q.shape
    C, Hkv = k_cache.shape[2], k_cache.shape[3]
    q, kc, vc = _c(q, np.uint16), _c(k_cache, np.uint16), _c(v_cache, np.uint16)
    kp, vp_ = _c(k_prefix, np.uint16), _c(v_prefix, np.uint16)
    offs, n = _c(prefix_offsets, np.int32), _c(cache_len, np.int32)
    out = np.full(q.shape, np.nan)
    lse = np.full(q.shape[:-1], np.nan)
    rc = _L().oracle_decode_attn(Qn, K, C, Hq, Hkv, D, float(scale), _p(q),
                                 _p(kp) if kp is not None and kp.size else None,
                                 _p(vp_) if vp_ is not None and vp_.size else None,
                                 _p(offs), _p(kc), _p(vc), _p(n), _p(out), _p(lse))
    if rc != 0:
        raise ValueError("oracle_decode_attn: bad arguments")
    return out, lse


def score_logprobs(hidden, weight, targets):
    """Log-softmax of hidden @ weight.T gathered at targets.  Returns (logprob [M][G], lse [M])."""
    M, H = hidden.shape
    V = weight.shape[0]
    targets = _c(targets, np.int32)
    if targets.ndim == 1:
        targets = targets[:, None]
    G = targets.shape[1]
    hidden, weight = _c(hidden, np.uint16), _c(weight, np.uint16)
    lp = np.empty((M, G), np.float64)
    lse = np.empty(M, np.float64)
    rc = _L().oracle_score_logprobs(M, H, V, G, _p(hidden), _p(weight), _p(targets), _p(lp), _p(lse))
    if rc != 0:
        raise ValueError("oracle_score_logprobs: bad arguments or out of memory")
    return lp, lse


def clip_align(cand, frames, tau):
    """Returns (cos [Qn][K][F], max_cos [Qn][K], argmax [Qn][K] int32, keep [Qn][K] uint8)."""
    Qn, K, E = cand.shape
    F = frames.shape[1]
    cand, frames = _c(cand, np.uint16), _c(frames, np.uint16)
    cosm = np.empty((Qn, K, F), np.float64)
    mc = np.empty((Qn, K), np.float64)
    am = np.empty((Qn, K), np.int32)
    keep = np.empty((Qn, K), np.uint8)
    rc = _L().oracle_clip_align(Qn, K, F, E, float(tau), _p(cand), _p(frames), _p(cosm), _p(mc),
                                _p(am), _p(keep))
    if rc != 0:
        raise ValueError("oracle_clip_align: bad arguments")
    return cosm, mc, am, keep


def select(logprob, mode=SEL_MASKED_MEAN_LOGPROB, lengths=None, keep=None, max_cos=None, delta=0.05,
           seed=0):
    """logprob [Qn][K][L][G] (any float dtype, widened exactly to fp64).  Returns (score, selected)."""
    lp = _c(logprob, np.float64)
    Qn, K, L, G = lp.shape
    lengths = _c(lengths, np.int32)
    keep = _c(keep, np.uint8)
    max_cos = _c(max_cos, np.float64)
    score = np.empty((Qn, K), np.float64)
    sel = np.empty(Qn, np.int32)
    rc = _L().oracle_select(Qn, K, L, G, int(mode), float(delta), _p(lp), _p(lengths), _p(keep),
                            _p(max_cos), _p(score), _p(sel), int(seed) & (2**64 - 1))
    if rc != 0:
        raise ValueError("oracle_select: bad arguments")
    return score, sel


def frame_topk(frames, texts, kf):
    """Eq. 2 per keyframe: returns (top_idx [Fr][kf] int32, top_sim [Fr][kf] fp64)."""
    frames, texts = _c(frames, np.uint16), _c(texts, np.uint16)
    Fr, E = frames.shape
    Nt = texts.shape[0]
    idx = np.empty((Fr, kf), np.int32)
    sim = np.empty((Fr, kf), np.float64)
    rc = _L().oracle_frame_topk(Fr, Nt, E, kf, _p(frames), _p(texts), _p(idx), _p(sim))
    if rc != 0:
        raise ValueError("oracle_frame_topk: bad arguments or out of memory")
    return idx, sim


def aggregate_topk(frame_offsets, top_idx, top_sim, Kq):
    """Eq. 3 per query: returns (idx [Qn][Kq] int32, sim [Qn][Kq] fp64)."""
    offs = _c(frame_offsets, np.int32)
    top_idx, top_sim = _c(top_idx, np.int32), _c(top_sim, np.float64)
    Qn = offs.shape[0] - 1
    kf = top_idx.shape[1]
    idx = np.empty((Qn, Kq), np.int32)
    sim = np.empty((Qn, Kq), np.float64)
    rc = _L().oracle_aggregate_topk(Qn, kf, Kq, _p(offs), _p(top_idx), _p(top_sim), _p(idx), _p(sim))
    if rc != 0:
        raise ValueError("oracle_aggregate_topk: bad arguments")
    return idx, sim


def retrieve(frames, frame_offsets, texts, kf, Kq):
    """Eq. 2-3 end to end: (frame lists, query lists) as (idx, sim) pairs."""
    fi, fs = frame_topk(frames, texts, kf)
    qi, qs = aggregate_topk(frame_offsets, fi, fs, Kq)
    return fi, fs, qi, qs


def keyframes(pixels, video_offsets, theta):
    """Eq. 1.  pixels [T][npix][3] (or [T][H][W][3]) uint8.

    Returns (hist [T][512] int32, sim [T] fp64, is_key [T] uint8, key_index [n] int32,
    key_offsets [Nv+1] int32)."""
    px = _c(pixels, np.uint8)
    T = px.shape[0]
    npix = px[0].size // 3 if T > 0 else 1
    offs = _c(video_offsets, np.int32)
    Nv = offs.shape[0] - 1
    hist = np.empty((T, 512), np.int32)
    sim = np.empty(T, np.float64)
    key = np.empty(T, np.uint8)
    kidx = np.empty(max(T, 1), np.int32)
    koffs = np.empty(Nv + 1, np.int32)
    rc = _L().oracle_keyframes(Nv, npix, float(theta), _p(offs), _p(px), _p(hist), _p(sim), _p(key),
                               _p(kidx), _p(koffs))
    if rc != 0:
        raise ValueError("oracle_keyframes: bad arguments")
    return hist, sim, key, kidx[:koffs[-1]].copy(), koffs
