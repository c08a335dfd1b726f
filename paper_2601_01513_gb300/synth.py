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

from .configs import VerifyConfig

_HERE = os.path.dirname(os.path.abspath(__file__))
SYNTH_SO = os.path.join(_HERE, "libfvrag_synth.so")

# stream ids (one independent SplitMix64 stream per tensor)
S_Q, S_KP, S_VP, S_KT, S_VT, S_HID, S_W, S_TGT = 1, 2, 3, 4, 5, 6, 7, 8
S_CAND, S_FRAME, S_PLEN, S_PERM, S_PFRAME, S_PC = 9, 10, 11, 12, 13, 14
S_LOGPROB, S_KEEP, S_MAXCOS, S_LEN = 20, 21, 22, 23

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


def bf16_bits_to_f32(x: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to fp32 (for test-side printing)."""
    return (x.astype(np.uint32) << 16).view(np.float32)


def f16_bits_to_f32(x: np.ndarray) -> np.ndarray:
    return x.view(np.float16).astype(np.float32)
