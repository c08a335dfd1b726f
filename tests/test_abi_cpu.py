"""The C ABI without a GPU: the library loads, exports every symbol that
include/fvrag.h declares, and rejects bad arguments on the host before any
CUDA call (fake, never-dereferenced pointer values are enough for that)."""
import ctypes
import os
import re

import pytest

from paper_2601_01513_gb300 import build, fvrag

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fvrag.h")

P = ctypes.c_void_p(0x10000)      # aligned fake pointer (never dereferenced: calls fail first)
PMIS = ctypes.c_void_p(0x10008)   # 8-byte aligned only


@pytest.fixture(scope="module")
def L():
    build.build_lib()
    return fvrag.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fvrag_[a-z_0-9]+)\s*\(", text)))


def test_exports_every_declared_symbol(L):
    names = declared_functions()
    assert len(names) >= 13
    assert set(names) == set(fvrag.EXPORTED)
    for n in names:
        assert hasattr(L, n), n


def test_version_and_strings(L):
    assert L.fvrag_abi_version() == 6
    for s in range(7):
        assert fvrag.status_string(s)
    assert fvrag.status_string(99) == "unknown status"


def test_wait_limit_roundtrip(L):
    old = fvrag.get_wait_limit_ns()
    fvrag.set_wait_limit_ns(5)
    assert fvrag.get_wait_limit_ns() == 1000    # clamped
    fvrag.set_wait_limit_ns(old)
    assert fvrag.get_wait_limit_ns() == old


def _attn(L, d, ws_bytes=1 << 30, q=P, kp=P, vp=P, offs=P, kt=P, vt=P, out=P, ws=P):
    return L.fvrag_verify_attn(ctypes.byref(d), q, kp, vp, offs, kt, vt, out, None, ws, ws_bytes, None)


def test_attn_validation(L):
    good = fvrag.AttnDesc(1, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 0)
    ws = L.fvrag_verify_attn_workspace(ctypes.byref(good))
    assert ws > 256
    assert _attn(L, fvrag.AttnDesc(0, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _attn(L, good, q=None) == fvrag.ERR_INVALID_ARG
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 3)) == fvrag.ERR_INVALID_ARG
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 4)) == fvrag.ERR_INVALID_ARG
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 5, 128, 8192, 8192, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 4, 96, 8192, 8192, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _attn(L, fvrag.AttnDesc(1, 5, 65, 28, 4, 128, 8192, 8192, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 4, 128, 8192, 8192, -1.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _attn(L, fvrag.AttnDesc(1, 5, 16, 28, 4, 128, 8192, 8192, float("nan"), 0)) == fvrag.ERR_INVALID_ARG
    assert _attn(L, good, q=PMIS) == fvrag.ERR_MISALIGNED
    assert _attn(L, good, ws_bytes=ws - 1) == fvrag.ERR_WORKSPACE
    assert _attn(L, good, ws=None) == fvrag.ERR_WORKSPACE
    assert _attn(L, good, kp=None) == fvrag.ERR_INVALID_ARG
    # no prefix at all: prefix pointers may be NULL, workspace is just the header
    nop = fvrag.AttnDesc(1, 2, 3, 4, 2, 64, 0, 0, 0.0, 0)
    assert L.fvrag_verify_attn_workspace(ctypes.byref(nop)) == 256


def test_attn_split_flags(L):
    """flags selects the key split: 0 (the library's choice), static, or streamed.  The
    streamed plan needs <= 64 queries (and <= 64 row tiles per KV head): beyond, both the
    workspace query (0) and the call (UNSUPPORTED) refuse it; the other plans serve it."""
    base = (1, 5, 16, 28, 4, 128, 8192, 8192, 0.0)
    for f in (0, fvrag.ATTN_SPLIT_STATIC, fvrag.ATTN_SPLIT_STREAM):
        assert L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*base, f))) >= 256
    many = (65, 2, 4, 8, 8, 64, 1000, 65000, 0.0)
    assert L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*many, fvrag.ATTN_SPLIT_STREAM))) == 0
    assert _attn(L, fvrag.AttnDesc(*many, fvrag.ATTN_SPLIT_STREAM)) == fvrag.ERR_UNSUPPORTED
    assert L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*many, fvrag.ATTN_SPLIT_STATIC))) >= 256
    assert L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*many, 0))) >= 256


def test_attn_sm_budget(L):
    # the budget is the last field; a negative one is rejected by both the call and the
    # workspace query, and a small one plans a coarser split (no partials for 20 SMs and
    # 20 row tiles: each tile's whole key list runs on one CTA)
    assert ctypes.sizeof(fvrag.AttnDesc) == 44
    assert fvrag.AttnDesc.sm_budget.offset == 40
    base = (1, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 0)
    bad = fvrag.AttnDesc(*base, -1)
    assert L.fvrag_verify_attn_workspace(ctypes.byref(bad)) == 0
    assert _attn(L, bad) == fvrag.ERR_INVALID_ARG
    full = L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*base, 0)))
    b20 = L.fvrag_verify_attn_workspace(ctypes.byref(fvrag.AttnDesc(*base, 20)))
    assert b20 == 256 < full
    # the budget only plans the split: validation and the workspace check still apply
    assert _attn(L, fvrag.AttnDesc(*base, 20), ws_bytes=255) == fvrag.ERR_WORKSPACE


def test_launch_count_ignores_rejected_calls(L):
    n0 = fvrag.launch_count()
    assert n0 >= 0
    assert _attn(L, fvrag.AttnDesc(0, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 0)) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_score_logprobs(ctypes.byref(fvrag.LmDesc(0, 8, 8, 1, 0)), P, P, P, P, None, P,
                                  1 << 20, None) == fvrag.ERR_INVALID_ARG
    assert fvrag.launch_count() == n0


def test_lm_validation(L):
    d = fvrag.LmDesc(80, 3584, 152064, 1, 0)
    need = L.fvrag_score_logprobs_workspace(ctypes.byref(d))
    assert need >= 256 + 2 * 256 * 80 * 4 + 80 * 4

    def call(desc, h=P, w=P, t=P, lp=P, ws=P, wsb=need):
        return L.fvrag_score_logprobs(ctypes.byref(desc), h, w, t, lp, None, ws, wsb, None)

    assert call(d, h=None) == fvrag.ERR_INVALID_ARG
    assert call(fvrag.LmDesc(0, 3584, 152064, 1, 0)) == fvrag.ERR_INVALID_ARG
    assert call(fvrag.LmDesc(80, 3584, 152064, 9, 0)) == fvrag.ERR_UNSUPPORTED
    assert call(fvrag.LmDesc(4096, 3584, 152064, 1, 0)) == fvrag.ERR_UNSUPPORTED
    assert call(fvrag.LmDesc(80, 3583, 152064, 1, 0)) == fvrag.ERR_MISALIGNED
    assert call(d, w=PMIS) == fvrag.ERR_MISALIGNED
    assert call(d, wsb=need - 4) == fvrag.ERR_WORKSPACE
    assert L.fvrag_score_logprobs_workspace(ctypes.byref(fvrag.LmDesc(0, 8, 8, 1, 0))) == 0
    # SM budget: the last field; negative budgets are rejected before anything is enqueued
    assert ctypes.sizeof(fvrag.LmDesc) == 24 and fvrag.LmDesc.sm_budget.offset == 20
    neg = fvrag.LmDesc(80, 3584, 152064, 1, 0, -1)
    assert call(neg) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_score_logprobs_workspace(ctypes.byref(neg)) == 0
    assert L.fvrag_score_logprobs_noalloc(ctypes.byref(neg), P, P, P, P, None, None) == \
        fvrag.ERR_INVALID_ARG
    # the workspace does not depend on the budget (partials are sized for the largest grid)
    assert L.fvrag_score_logprobs_workspace(ctypes.byref(fvrag.LmDesc(80, 3584, 152064, 1, 0, 64))) == need


def test_clip_and_select_validation(L):
    d = fvrag.ClipDesc(1, 5, 64, 768, 0.2, 0)
    assert L.fvrag_clip_align(ctypes.byref(d), None, P, None, P, P, P, None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_clip_align(ctypes.byref(fvrag.ClipDesc(1, 5, 64, 770, 0.2, 0)), P, P, None, P, P, P,
                              None) == fvrag.ERR_UNSUPPORTED
    assert L.fvrag_clip_align(ctypes.byref(fvrag.ClipDesc(1, 5, 0, 768, 0.2, 0)), P, P, None, P, P, P,
                              None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_clip_align(ctypes.byref(d), PMIS, P, None, P, P, P, None) == fvrag.ERR_MISALIGNED
    s = fvrag.SelectDesc(1, 5, 16, 1, fvrag.SEL_MASKED_MEAN_LOGPROB, 0.05, 0)
    assert L.fvrag_select_candidate(ctypes.byref(s), P, None, None, None, P, P, None) == fvrag.ERR_INVALID_ARG
    s2 = fvrag.SelectDesc(1, 5, 16, 1, fvrag.SEL_TWO_STAGE, 0.05, 0)
    assert L.fvrag_select_candidate(ctypes.byref(s2), P, None, None, P, P, P, None) == fvrag.ERR_INVALID_ARG
    s3 = fvrag.SelectDesc(1, 5, 16, 2, 7, 0.05, 0)
    assert L.fvrag_select_candidate(ctypes.byref(s3), P, None, P, P, P, P, None) == fvrag.ERR_INVALID_ARG
    s4 = fvrag.SelectDesc(1, 2000, 16, 1, 0, 0.05, 0)
    assert L.fvrag_select_candidate(ctypes.byref(s4), P, None, P, P, P, P, None) == fvrag.ERR_UNSUPPORTED
    sel = lambda mode, G, keep, mc: L.fvrag_select_candidate(
        ctypes.byref(fvrag.SelectDesc(1, 5, 16, G, mode, 0.05, 0, 7)), P, None, keep, mc, P, P, None)
    assert sel(fvrag.SEL_INVERT, 2, None, P) == fvrag.ERR_INVALID_ARG        # needs keep
    assert sel(fvrag.SEL_ADDITION, 2, P, None) == fvrag.ERR_INVALID_ARG      # needs max_cos
    assert sel(fvrag.SEL_ADDITION, 1, P, P) == fvrag.ERR_INVALID_ARG        # needs Yes/No gathers
    assert sel(fvrag.SEL_ALIGNMENT_ONLY, 1, None, None) == fvrag.ERR_INVALID_ARG
    assert sel(fvrag.SEL_RANDOM + 1, 2, P, P) == fvrag.ERR_INVALID_ARG       # unknown mode
    assert ctypes.sizeof(fvrag.SelectDesc) == 40


def test_status_calls_reject_null(L):
    assert L.fvrag_read_status(None, None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_clear_status(None, None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_selftest_wait_timeout(None, None) == fvrag.ERR_INVALID_ARG


def test_binding_raises_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(fvrag, "_lib", None)
    monkeypatch.setattr(fvrag, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(OSError):
        fvrag.lib()


def _rt(L, d, ws_bytes=1 << 30, fe=P, fo=P, te=P, inv=P, oi=P, os_=P, ws=P):
    return L.fvrag_retrieve(ctypes.byref(d), fe, fo, te, inv, None, None, oi, os_, ws, ws_bytes, None)


def test_retrieve_validation(L):
    assert ctypes.sizeof(fvrag.RetrieveDesc) == 28
    good = fvrag.RetrieveDesc(16, 300, 1 << 20, 768, 3, 3, 0)
    ws = L.fvrag_retrieve_workspace(ctypes.byref(good))
    assert ws >= 256 + 2 * 256 * 300 * 3 * 4 + (1 << 20) * 4
    assert _rt(L, fvrag.RetrieveDesc(0, 300, 1 << 20, 768, 3, 3, 0)) == fvrag.ERR_INVALID_ARG
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 0, 768, 3, 3, 0)) == fvrag.ERR_INVALID_ARG
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 1 << 20, 768, 0, 3, 0)) == fvrag.ERR_INVALID_ARG
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 1 << 20, 768, 3, 3, 2)) == fvrag.ERR_INVALID_ARG
    assert _rt(L, good, te=None) == fvrag.ERR_INVALID_ARG
    assert _rt(L, good, fe=None) == fvrag.ERR_INVALID_ARG
    assert _rt(L, good, oi=None) == fvrag.ERR_INVALID_ARG
    assert _rt(L, fvrag.RetrieveDesc(16, 2049, 1 << 20, 768, 1, 3, 0)) == fvrag.ERR_UNSUPPORTED
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 1 << 20, 768, 9, 3, 0)) == fvrag.ERR_UNSUPPORTED
    assert _rt(L, fvrag.RetrieveDesc(16, 1281, 1 << 20, 768, 3, 3, 0)) == fvrag.ERR_UNSUPPORTED
    assert _rt(L, fvrag.RetrieveDesc(16, 513, 1 << 20, 768, 8, 3, 0)) == fvrag.ERR_UNSUPPORTED
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 1 << 20, 768, 3, 65, 0)) == fvrag.ERR_UNSUPPORTED
    assert _rt(L, fvrag.RetrieveDesc(16, 300, 1 << 20, 764, 3, 3, 0)) == fvrag.ERR_MISALIGNED
    assert _rt(L, good, te=PMIS) == fvrag.ERR_MISALIGNED
    assert _rt(L, good, inv=PMIS) == fvrag.ERR_MISALIGNED
    assert _rt(L, good, ws_bytes=ws - 1) == fvrag.ERR_WORKSPACE
    assert L.fvrag_embed_inv_norms(None, 10, 768, P, None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_embed_inv_norms(P, 0, 768, P, None) == fvrag.ERR_INVALID_ARG
    assert L.fvrag_embed_inv_norms(P, 10, 764, P, None) == fvrag.ERR_MISALIGNED
    assert L.fvrag_embed_inv_norms(PMIS, 10, 768, P, None) == fvrag.ERR_MISALIGNED


def _kf(L, d, ws_bytes=1 << 30, px=P, vo=P, sim=P, key=P, ki=P, ko=P, ws=P):
    return L.fvrag_keyframes(ctypes.byref(d), px, vo, None, sim, key, ki, ko, ws, ws_bytes, None)


def test_keyframes_validation(L):
    assert ctypes.sizeof(fvrag.KeyframeDesc) == 32
    good = fvrag.KeyframeDesc(8, 5000, 720, 1280, 0.6, 0)
    ws = L.fvrag_keyframes_workspace(ctypes.byref(good))
    assert ws == 256 + 5000 * 512 * 4
    assert _kf(L, fvrag.KeyframeDesc(0, 5000, 720, 1280, 0.6, 0)) == fvrag.ERR_INVALID_ARG
    assert _kf(L, fvrag.KeyframeDesc(8, -1, 720, 1280, 0.6, 0)) == fvrag.ERR_INVALID_ARG
    assert _kf(L, fvrag.KeyframeDesc(8, 5000, 720, 1280, 0.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _kf(L, fvrag.KeyframeDesc(8, 5000, 720, 1280, float("nan"), 0)) == fvrag.ERR_INVALID_ARG
    assert _kf(L, fvrag.KeyframeDesc(8, 5000, 720, 1280, 0.6, 1)) == fvrag.ERR_INVALID_ARG
    assert _kf(L, good, px=None) == fvrag.ERR_INVALID_ARG
    assert _kf(L, good, vo=None) == fvrag.ERR_INVALID_ARG
    assert _kf(L, good, ki=None) == fvrag.ERR_INVALID_ARG
    assert _kf(L, fvrag.KeyframeDesc(8, 5000, 3, 5, 0.6, 0)) == fvrag.ERR_MISALIGNED
    assert _kf(L, good, px=PMIS) == fvrag.ERR_MISALIGNED
    assert _kf(L, good, ws_bytes=ws - 1) == fvrag.ERR_WORKSPACE
    assert _kf(L, good, ws=None) == fvrag.ERR_WORKSPACE


def _dec(L, d, ws_bytes=1 << 30, q=P, kp=P, vp=P, offs=P, kc=P, vc=P, n=P, out=P, ws=P):
    return L.fvrag_decode_attn(ctypes.byref(d), q, kp, vp, offs, kc, vc, n, out, None, ws, ws_bytes, None)


def test_decode_validation(L):
    assert ctypes.sizeof(fvrag.DecodeDesc) == 40
    good = fvrag.DecodeDesc(16, 5, 1024, 16, 2, 128, 16384, 160000, 0.0, 0)
    ws = L.fvrag_decode_attn_workspace(ctypes.byref(good))
    assert ws >= 256
    assert _dec(L, fvrag.DecodeDesc(0, 5, 1024, 16, 2, 128, 16384, 160000, 0.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _dec(L, fvrag.DecodeDesc(16, 5, 0, 16, 2, 128, 16384, 160000, 0.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _dec(L, fvrag.DecodeDesc(16, 5, 1024, 16, 2, 128, 16384, 160000, -1.0, 0)) == fvrag.ERR_INVALID_ARG
    assert _dec(L, fvrag.DecodeDesc(16, 5, 1024, 16, 2, 128, 16384, 160000, 0.0, 4)) == fvrag.ERR_INVALID_ARG
    assert _dec(L, good, n=None) == fvrag.ERR_INVALID_ARG
    assert _dec(L, good, kc=None) == fvrag.ERR_INVALID_ARG
    assert _dec(L, good, kp=None) == fvrag.ERR_INVALID_ARG
    assert _dec(L, fvrag.DecodeDesc(16, 5, 1024, 16, 3, 128, 16384, 160000, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _dec(L, fvrag.DecodeDesc(16, 5, 1024, 16, 2, 96, 16384, 160000, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _dec(L, fvrag.DecodeDesc(1 << 16, 64, 1024, 16, 2, 128, 0, 0, 0.0, 0)) == fvrag.ERR_UNSUPPORTED
    assert _dec(L, good, q=PMIS) == fvrag.ERR_MISALIGNED
    assert _dec(L, good, kc=PMIS) == fvrag.ERR_MISALIGNED
    assert _dec(L, good, ws_bytes=ws - 1) == fvrag.ERR_WORKSPACE


def test_nvtx_ranges_switch_on_without_a_profiler():
    """FVRAG_NVTX=1 makes every public call push and pop an NVTX range; with no profiler
    attached that is a no-op, so validation still returns the same status (run in a child
    process, since the switch is read once)."""
    import subprocess
    import sys
    import os
    code = (
        "import ctypes, sys; sys.path.insert(0, %r)\n"
        "from paper_2601_01513_gb300 import fvrag\n"
        "L = fvrag.lib()\n"
        "d = fvrag.AttnDesc(0, 5, 16, 28, 4, 128, 8192, 8192, 0.0, 0)\n"
        "p = ctypes.c_void_p(1 << 20)\n"
        "st = L.fvrag_verify_attn(ctypes.byref(d), p, p, p, p, p, p, p, None, p, 1 << 30, None)\n"
        "print(st)\n" % os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    env = dict(os.environ, FVRAG_NVTX="1")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=120)
    assert r.returncode == 0, r.stderr
    assert int(r.stdout.strip().splitlines()[-1]) == fvrag.ERR_INVALID_ARG
