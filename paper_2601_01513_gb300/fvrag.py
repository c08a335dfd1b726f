"""Thin Python binding of libfvrag (``include/fvrag.h``): argument marshalling only.

Every function here fills the C descriptor from tensor shapes, passes raw
device pointers and the current CUDA stream, and raises ``FvragError`` on a
non-OK status.  All arithmetic runs in the library's CUDA kernels; there is no
fallback of any kind -- if ``libfvrag.so`` is missing, loading raises.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfvrag.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_MISALIGNED, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT = range(7)
# fvrag_attn_desc.flags: the key split of the verification attention (0: the library's choice)
ATTN_SPLIT_STATIC, ATTN_SPLIT_STREAM = 1, 2
SEL_MASKED_MEAN_LOGPROB = 0
SEL_TWO_STAGE = 1
SEL_ADDITION = 2
SEL_INVERT = 3
SEL_RELIABILITY_ONLY = 4
SEL_ALIGNMENT_ONLY = 5
SEL_RANDOM = 6
WS_HEADER_BYTES = 256

EXPORTED = (
    "fvrag_abi_version", "fvrag_status_string", "fvrag_launch_count",
    "fvrag_verify_attn_workspace", "fvrag_verify_attn",
    "fvrag_decode_attn_workspace", "fvrag_decode_attn",
    "fvrag_score_logprobs_workspace", "fvrag_score_logprobs", "fvrag_score_logprobs_noalloc",
    "fvrag_score_logprobs_noalloc_status",
    "fvrag_clip_align", "fvrag_select_candidate",
    "fvrag_embed_inv_norms", "fvrag_retrieve_workspace", "fvrag_retrieve",
    "fvrag_keyframes_workspace", "fvrag_keyframes",
    "fvrag_read_status", "fvrag_clear_status",
    "fvrag_set_wait_limit_ns", "fvrag_get_wait_limit_ns", "fvrag_selftest_wait_timeout",
)


class FvragError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__("%s: %s (status %d)" % (where, status_string(status), status))


class AttnDesc(ctypes.Structure):
    _fields_ = [("num_queries", ctypes.c_int32), ("num_cand", ctypes.c_int32),
                ("cand_len", ctypes.c_int32), ("hq", ctypes.c_int32), ("hkv", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("max_prefix", ctypes.c_int32),
                ("total_prefix", ctypes.c_int32), ("softmax_scale", ctypes.c_float),
                ("flags", ctypes.c_uint32), ("sm_budget", ctypes.c_int32)]


class DecodeDesc(ctypes.Structure):
    _fields_ = [("num_queries", ctypes.c_int32), ("num_drafts", ctypes.c_int32),
                ("cache_cap", ctypes.c_int32), ("hq", ctypes.c_int32), ("hkv", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("max_prefix", ctypes.c_int32),
                ("total_prefix", ctypes.c_int32), ("softmax_scale", ctypes.c_float),
                ("flags", ctypes.c_uint32)]


class LmDesc(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int32), ("hidden", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("gathers", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("sm_budget", ctypes.c_int32)]


class ClipDesc(ctypes.Structure):
    _fields_ = [("num_queries", ctypes.c_int32), ("num_cand", ctypes.c_int32),
                ("num_frames", ctypes.c_int32), ("dim", ctypes.c_int32),
                ("threshold", ctypes.c_float), ("flags", ctypes.c_uint32)]


class SelectDesc(ctypes.Structure):
    _fields_ = [("num_queries", ctypes.c_int32), ("num_cand", ctypes.c_int32),
                ("cand_len", ctypes.c_int32), ("gathers", ctypes.c_int32),
                ("mode", ctypes.c_int32), ("delta", ctypes.c_float), ("flags", ctypes.c_uint32),
                ("seed", ctypes.c_uint64)]


class RetrieveDesc(ctypes.Structure):
    _fields_ = [("num_queries", ctypes.c_int32), ("num_keyframes", ctypes.c_int32),
                ("num_texts", ctypes.c_int32), ("dim", ctypes.c_int32), ("k_frame", ctypes.c_int32),
                ("k_query", ctypes.c_int32), ("flags", ctypes.c_uint32)]


class KeyframeDesc(ctypes.Structure):
    _fields_ = [("num_videos", ctypes.c_int32), ("total_frames", ctypes.c_int32),
                ("height", ctypes.c_int32), ("width", ctypes.c_int32), ("theta", ctypes.c_double),
                ("flags", ctypes.c_uint32)]


_lib = None


def lib():
    """The loaded libfvrag.so (raises OSError if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise OSError("libfvrag.so not built: run `python -m paper_2601_01513_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        vp, sz, i32, u64 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_uint64
        L.fvrag_abi_version.restype = i32
        L.fvrag_launch_count.restype = u64
        L.fvrag_status_string.restype = ctypes.c_char_p
        L.fvrag_status_string.argtypes = [i32]
        L.fvrag_verify_attn_workspace.restype = sz
        L.fvrag_verify_attn_workspace.argtypes = [ctypes.POINTER(AttnDesc)]
        L.fvrag_verify_attn.restype = i32
        L.fvrag_verify_attn.argtypes = [ctypes.POINTER(AttnDesc)] + [vp] * 8 + [vp, sz, vp]
        L.fvrag_decode_attn_workspace.restype = sz
        L.fvrag_decode_attn_workspace.argtypes = [ctypes.POINTER(DecodeDesc)]
        L.fvrag_decode_attn.restype = i32
        L.fvrag_decode_attn.argtypes = [ctypes.POINTER(DecodeDesc)] + [vp] * 9 + [vp, sz, vp]
        L.fvrag_score_logprobs_workspace.restype = sz
        L.fvrag_score_logprobs_workspace.argtypes = [ctypes.POINTER(LmDesc)]
        L.fvrag_score_logprobs.restype = i32
        L.fvrag_score_logprobs.argtypes = [ctypes.POINTER(LmDesc)] + [vp] * 5 + [vp, sz, vp]
        L.fvrag_score_logprobs_noalloc.restype = i32
        L.fvrag_score_logprobs_noalloc.argtypes = [ctypes.POINTER(LmDesc)] + [vp] * 5 + [vp]
        L.fvrag_score_logprobs_noalloc_status.restype = i32
        L.fvrag_score_logprobs_noalloc_status.argtypes = [vp]
        L.fvrag_clip_align.restype = i32
        L.fvrag_clip_align.argtypes = [ctypes.POINTER(ClipDesc)] + [vp] * 6 + [vp]
        L.fvrag_select_candidate.restype = i32
        L.fvrag_select_candidate.argtypes = [ctypes.POINTER(SelectDesc)] + [vp] * 6 + [vp]
        L.fvrag_embed_inv_norms.restype = i32
        L.fvrag_embed_inv_norms.argtypes = [vp, ctypes.c_int32, ctypes.c_int32, vp, vp]
        L.fvrag_retrieve_workspace.restype = sz
        L.fvrag_retrieve_workspace.argtypes = [ctypes.POINTER(RetrieveDesc)]
        L.fvrag_retrieve.restype = i32
        L.fvrag_retrieve.argtypes = [ctypes.POINTER(RetrieveDesc)] + [vp] * 9 + [sz, vp]
        L.fvrag_keyframes_workspace.restype = sz
        L.fvrag_keyframes_workspace.argtypes = [ctypes.POINTER(KeyframeDesc)]
        L.fvrag_keyframes.restype = i32
        L.fvrag_keyframes.argtypes = [ctypes.POINTER(KeyframeDesc)] + [vp] * 8 + [sz, vp]
        L.fvrag_read_status.restype = i32
        L.fvrag_read_status.argtypes = [vp, vp]
        L.fvrag_clear_status.restype = i32
        L.fvrag_clear_status.argtypes = [vp, vp]
        L.fvrag_set_wait_limit_ns.restype = None
        L.fvrag_set_wait_limit_ns.argtypes = [u64]
        L.fvrag_get_wait_limit_ns.restype = u64
        L.fvrag_selftest_wait_timeout.restype = i32
        L.fvrag_selftest_wait_timeout.argtypes = [vp, vp]
        _lib = L
    return _lib


def status_string(s: int) -> str:
    return lib().fvrag_status_string(int(s)).decode()


def _check(s, where):
    if s != OK:
        raise FvragError(s, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


# --------------------------------------------------------------------- descriptors
def lm_desc(hidden, weight, targets, sm_budget=0) -> LmDesc:
    G = 1 if targets.dim() == 1 else int(targets.shape[1])
    return LmDesc(int(hidden.shape[0]), int(hidden.shape[1]), int(weight.shape[0]), G, 0,
                  int(sm_budget))


def attn_workspace_bytes(desc: AttnDesc) -> int:
    return int(lib().fvrag_verify_attn_workspace(ctypes.byref(desc)))


def lm_workspace_bytes(desc: LmDesc) -> int:
    return int(lib().fvrag_score_logprobs_workspace(ctypes.byref(desc)))


# --------------------------------------------------------------------- the four calls
def verify_attn(q, k_prefix, v_prefix, prefix_offsets, k_tail, v_tail, out, ws, max_prefix,
                lse=None, softmax_scale=0.0, stream=None, sm_budget=0, split=0):
    """q [Qn][K][L][hq][D] bf16; k/v_prefix [sum P][hkv][D]; prefix_offsets [Qn+1] int32 (device);
    k/v_tail [Qn][K][L][hkv][D]; out like q; lse [Qn][K][L][hq] fp32 or None; ws uint8 device;
    sm_budget: SMs the key split is planned for (0: all); split: 0 (library's choice),
    ATTN_SPLIT_STATIC or ATTN_SPLIT_STREAM."""
    d = AttnDesc(q.shape[0], q.shape[1], q.shape[2], q.shape[3], k_tail.shape[3], q.shape[4],
                 int(max_prefix), 0 if k_prefix is None else int(k_prefix.shape[0]),
                 float(softmax_scale), int(split), int(sm_budget))
    s = lib().fvrag_verify_attn(ctypes.byref(d), _ptr(q), _ptr(k_prefix), _ptr(v_prefix),
                                _ptr(prefix_offsets), _ptr(k_tail), _ptr(v_tail), _ptr(out),
                                _ptr(lse), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream))
    _check(s, "fvrag_verify_attn")


def decode_desc(q, k_prefix, k_cache, max_prefix, softmax_scale=0.0) -> DecodeDesc:
    return DecodeDesc(int(q.shape[0]), int(q.shape[1]), int(k_cache.shape[2]), int(q.shape[2]),
                      int(k_cache.shape[3]), int(q.shape[3]), int(max_prefix),
                      0 if k_prefix is None else int(k_prefix.shape[0]), float(softmax_scale), 0)


def decode_workspace_bytes(desc: DecodeDesc) -> int:
    return int(lib().fvrag_decode_attn_workspace(ctypes.byref(desc)))


def decode_attn(q, k_prefix, v_prefix, prefix_offsets, k_cache, v_cache, cache_len, out, ws,
                max_prefix, lse=None, softmax_scale=0.0, stream=None):
    """q [Qn][K][hq][D] bf16; k/v_prefix [sum P][hkv][D]; prefix_offsets [Qn+1] int32 (device);
    k/v_cache [Qn][K][C][hkv][D]; cache_len [Qn][K] int32 (device); out like q;
    lse [Qn][K][hq] fp32 or None."""
    d = decode_desc(q, k_prefix, k_cache, max_prefix, softmax_scale)
    s = lib().fvrag_decode_attn(ctypes.byref(d), _ptr(q), _ptr(k_prefix), _ptr(v_prefix),
                                _ptr(prefix_offsets), _ptr(k_cache), _ptr(v_cache), _ptr(cache_len),
                                _ptr(out), _ptr(lse), _ptr(ws), ws.numel() * ws.element_size(),
                                _stream(stream))
    _check(s, "fvrag_decode_attn")


def score_logprobs(hidden, weight, targets, logprob, ws, lse=None, stream=None, sm_budget=0):
    """hidden [M][H] bf16, weight [V][H] bf16, targets [M][G] int32 -> logprob [M][G] fp32;
    sm_budget: the most SMs the persistent grid occupies (0: all)."""
    d = lm_desc(hidden, weight, targets, sm_budget)
    s = lib().fvrag_score_logprobs(ctypes.byref(d), _ptr(hidden), _ptr(weight), _ptr(targets),
                                   _ptr(logprob), _ptr(lse), _ptr(ws), ws.numel() * ws.element_size(),
                                   _stream(stream))
    _check(s, "fvrag_score_logprobs")


def score_logprobs_noalloc(hidden, weight, targets, logprob, lse=None, stream=None):
    """As score_logprobs, with the scratch in the library's static device array (no workspace)."""
    d = lm_desc(hidden, weight, targets)
    s = lib().fvrag_score_logprobs_noalloc(ctypes.byref(d), _ptr(hidden), _ptr(weight), _ptr(targets),
                                           _ptr(logprob), _ptr(lse), _stream(stream))
    _check(s, "fvrag_score_logprobs_noalloc")


def noalloc_status(stream=None) -> int:
    """Device-side status of the last score_logprobs_noalloc call (synchronises `stream`)."""
    return lib().fvrag_score_logprobs_noalloc_status(_stream(stream))


def clip_align(cand_emb, frame_emb, threshold, max_cos, argmax, keep, cos=None, stream=None):
    """cand_emb [Qn][K][E] fp16, frame_emb [Qn][F][E] fp16 -> max_cos, argmax, keep [Qn][K]."""
    Qn, K, E = cand_emb.shape
    d = ClipDesc(Qn, K, int(frame_emb.shape[1]), E, float(threshold), 0)
    s = lib().fvrag_clip_align(ctypes.byref(d), _ptr(cand_emb), _ptr(frame_emb), _ptr(cos),
                               _ptr(max_cos), _ptr(argmax), _ptr(keep), _stream(stream))
    _check(s, "fvrag_clip_align")


def select_candidate(logprob, score, selected, mode=SEL_MASKED_MEAN_LOGPROB, keep=None, max_cos=None,
                     lengths=None, delta=0.05, seed=0, stream=None):
    """logprob [Qn][K][L][G] fp32 -> score [Qn][K] fp32, selected [Qn] int32."""
    Qn, K, L, G = logprob.shape
    d = SelectDesc(Qn, K, L, G, int(mode), float(delta), 0, int(seed) & (2**64 - 1))
    s = lib().fvrag_select_candidate(ctypes.byref(d), _ptr(logprob), _ptr(lengths), _ptr(keep),
                                     _ptr(max_cos), _ptr(score), _ptr(selected), _stream(stream))
    _check(s, "fvrag_select_candidate")


def embed_inv_norms(x, inv_norm, stream=None):
    """x [rows][dim] fp16 -> inv_norm [rows] fp32 (1/|row|, 0 for a zero row)."""
    s = lib().fvrag_embed_inv_norms(_ptr(x), int(x.shape[0]), int(x.shape[1]), _ptr(inv_norm),
                                    _stream(stream))
    _check(s, "fvrag_embed_inv_norms")


def retrieve_desc(num_queries, frame_emb, text_emb, k_frame, k_query) -> RetrieveDesc:
    return RetrieveDesc(int(num_queries), int(frame_emb.shape[0]), int(text_emb.shape[0]),
                        int(text_emb.shape[1]), int(k_frame), int(k_query), 0)


def retrieve_workspace_bytes(desc: RetrieveDesc) -> int:
    return int(lib().fvrag_retrieve_workspace(ctypes.byref(desc)))


def retrieve(frame_emb, frame_offsets, text_emb, k_frame, out_idx, out_sim, ws, text_inv_norm=None,
             frame_topk=None, frame_topk_sim=None, stream=None):
    """frame_emb [Fr][E] fp16, frame_offsets [Qn+1] int32 (device), text_emb [Nt][E] fp16 ->
    out_idx [Qn][Kq] int32, out_sim [Qn][Kq] fp32; frame_topk / frame_topk_sim [Fr][k_frame]
    are written when given; text_inv_norm [Nt] fp32 from embed_inv_norms, or None."""
    Qn, Kq = out_idx.shape
    d = retrieve_desc(Qn, frame_emb, text_emb, k_frame, Kq)
    s = lib().fvrag_retrieve(ctypes.byref(d), _ptr(frame_emb), _ptr(frame_offsets), _ptr(text_emb),
                             _ptr(text_inv_norm), _ptr(frame_topk), _ptr(frame_topk_sim),
                             _ptr(out_idx), _ptr(out_sim), _ptr(ws), ws.numel() * ws.element_size(),
                             _stream(stream))
    _check(s, "fvrag_retrieve")


def keyframe_desc(num_videos, pixels, theta) -> KeyframeDesc:
    return KeyframeDesc(int(num_videos), int(pixels.shape[0]), int(pixels.shape[1]),
                        int(pixels.shape[2]), float(theta), 0)


def keyframes_workspace_bytes(desc: KeyframeDesc) -> int:
    return int(lib().fvrag_keyframes_workspace(ctypes.byref(desc)))


def keyframes(pixels, video_offsets, theta, sim, is_key, key_index, key_offsets, ws, hist=None,
              stream=None):
    """pixels [T][H][W][3] uint8, video_offsets [Nv+1] int32 (device) -> sim [T] fp32,
    is_key [T] uint8, key_index [T] int32, key_offsets [Nv+1] int32 (and hist [T][512])."""
    d = keyframe_desc(int(video_offsets.shape[0]) - 1, pixels, theta)
    s = lib().fvrag_keyframes(ctypes.byref(d), _ptr(pixels), _ptr(video_offsets), _ptr(hist),
                              _ptr(sim), _ptr(is_key), _ptr(key_index), _ptr(key_offsets), _ptr(ws),
                              ws.numel() * ws.element_size(), _stream(stream))
    _check(s, "fvrag_keyframes")


# --------------------------------------------------------------------- status
def launch_count() -> int:
    """Kernel launches the library has enqueued in this process (captures count once)."""
    return int(lib().fvrag_launch_count())


def read_status(ws, stream=None) -> int:
    return int(lib().fvrag_read_status(_ptr(ws), _stream(stream)))


def clear_status(ws, stream=None) -> None:
    _check(lib().fvrag_clear_status(_ptr(ws), _stream(stream)), "fvrag_clear_status")


def set_wait_limit_ns(ns: int) -> None:
    lib().fvrag_set_wait_limit_ns(int(ns))


def get_wait_limit_ns() -> int:
    return int(lib().fvrag_get_wait_limit_ns())


def selftest_wait_timeout(ws, stream=None) -> None:
    _check(lib().fvrag_selftest_wait_timeout(_ptr(ws), _stream(stream)), "fvrag_selftest_wait_timeout")
