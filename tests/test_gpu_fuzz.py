"""Seeded random shapes within each call's supported ranges, through the C ABI, against
the fp64 oracle element by element: ragged prefixes (including none), odd tail lengths and
head counts, GQA ratios from 1 to 16, both head dimensions; odd row counts, hidden sizes,
vocabularies and gather counts for the LM head; odd candidate, frame and dimension counts
for CLIP; ragged prefixes and cache fills for the decode step; keyframe and corpus counts,
dimensions, k_frame and k_query for retrieval; frame sizes, video lengths and thresholds
for keyframe extraction.  The shapes are drawn once from fixed seeds, so every run checks
the same cases."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import configs, fvrag, synth

from gpu_helpers import (ATTN_ATOL, ATTN_LSE_ATOL, COS_ATOL, LOGPROB_ATOL, check_argmax_with_margin,
                         check_keep_with_margin, ensure_built, run_attn, run_clip, run_decode, run_lm)

pytestmark = pytest.mark.gpu

N_CASES = 8


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return ensure_built()


def _heads(rng):
    grp = int(rng.choice([1, 2, 4, 7, 8, 16]))
    hkv = int(rng.integers(1, 5))
    return grp * hkv, hkv


def _attn_cases():
    rng = np.random.default_rng(20261202)
    out = []
    for _ in range(N_CASES):
        hq, hkv = _heads(rng)
        Qn, K, L = int(rng.integers(1, 4)), int(rng.integers(1, 7)), int(rng.integers(1, 65))
        D = int(rng.choice([64, 128]))
        plens = [int(p) if rng.random() > 0.15 else 0 for p in rng.integers(0, 2500, Qn)]
        out.append((Qn, K, L, hq, hkv, D, tuple(plens)))
    return out


@pytest.mark.parametrize("case", _attn_cases(), ids=lambda c: "x".join(map(str, c[:6])) + "_P" + "-".join(map(str, c[6])))
def test_attn_random_shapes(case):
    Qn, K, L, Hq, Hkv, D, plens = case
    seed = 5000 + sum(plens) + 7 * L + Hq
    offs = np.zeros(Qn + 1, np.int32)
    offs[1:] = np.cumsum(plens)
    tot = int(offs[-1])
    q = synth.normal_bf16((Qn, K, L, Hq, D), seed, 1)
    kp, vp = synth.normal_bf16((tot, Hkv, D), seed, 2), synth.normal_bf16((tot, Hkv, D), seed, 3)
    kt, vt = synth.normal_bf16((Qn, K, L, Hkv, D), seed, 4), synth.normal_bf16((Qn, K, L, Hkv, D), seed, 5)
    out, lse, st = run_attn(q, kp, vp, offs, kt, vt)
    assert st == fvrag.OK
    ref, ref_lse = oracle.verify_attn(q, kp, vp, offs, kt, vt)
    assert np.all(np.isfinite(out))
    assert np.max(np.abs(out - ref)) <= ATTN_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= ATTN_LSE_ATOL


def _lm_cases():
    rng = np.random.default_rng(20261203)
    return [(int(rng.integers(1, 700)), 8 * int(rng.integers(1, 41)), int(rng.integers(1, 20000)),
             int(rng.integers(1, 9))) for _ in range(N_CASES)]


@pytest.mark.parametrize("case", _lm_cases(), ids=lambda c: "M%d_H%d_V%d_G%d" % c)
def test_lm_random_shapes(case):
    M, H, V, G = case
    seed = 6000 + M + V
    hid = synth.normal_bf16((M, H), seed, 1)
    W = synth.normal_bf16((V, H), seed, 2, 0.0, 0.2)
    tgt = synth.uniform_i32((M, G), seed, 3, 0, V)
    lp, lse, st = run_lm(hid, W, tgt)
    assert st == fvrag.OK
    ref, ref_lse = oracle.score_logprobs(hid, W, tgt)
    assert np.max(np.abs(lp - ref)) <= LOGPROB_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= LOGPROB_ATOL


def _clip_cases():
    rng = np.random.default_rng(20261204)
    return [(int(rng.integers(1, 4)), int(rng.integers(1, 41)), int(rng.integers(1, 700)),
             8 * int(rng.integers(1, 129))) for _ in range(N_CASES)]


@pytest.mark.parametrize("case", _clip_cases(), ids=lambda c: "Q%dK%dF%dE%d" % c)
def test_clip_random_shapes(case):
    Qn, K, F, E = case
    seed = 7000 + K * F + E
    cand = synth.round_f16(synth.normal_f64((Qn, K, E), seed, 1))
    frames = synth.round_f16(synth.normal_f64((Qn, F, E), seed, 2))
    # plant a matching frame for the first candidate of every query, so keep is exercised
    frames[:, F // 2] = cand[:, 0]
    tau = 0.2
    cos, mc, am, keep = run_clip(cand, frames, tau)
    rcos, rmc, _, _ = oracle.clip_align(cand, frames, tau)
    assert np.max(np.abs(cos - rcos)) <= COS_ATOL
    assert np.max(np.abs(mc - rmc)) <= COS_ATOL
    check_argmax_with_margin(am, rcos)
    check_keep_with_margin(keep, rmc, tau)


def _decode_cases():
    rng = np.random.default_rng(20261205)
    out = []
    for _ in range(N_CASES):
        hq, hkv = _heads(rng)
        cap = int(rng.integers(1, 400))
        lo = int(rng.integers(0, 2500))
        out.append((int(rng.integers(1, 4)), int(rng.integers(1, 9)), hq, hkv, int(rng.choice([64, 128])),
                    (lo, lo + int(rng.integers(0, 800))), cap, (1, cap)))
    return out


@pytest.mark.parametrize("case", _decode_cases(), ids=lambda c: "x".join(map(str, c[:5])) + "_P%d-%d_C%d" % (c[5] + (c[6],)))
def test_decode_random_shapes(case):
    Qn, K, hq, hkv, D, pr, C, cr = case
    cfg = configs.DEC_TINY.with_(num_queries=Qn, num_drafts=K, hq=hq, hkv=hkv, head_dim=D,
                                 prefix_range=pr, cache_cap=C, cache_range=cr, seed=8000 + C + K)
    x = synth.decode_inputs(cfg)
    out, lse, st = run_decode(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_cache"],
                              x["v_cache"], x["cache_len"])
    assert st == fvrag.OK
    ro, rl = oracle.decode_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                x["k_cache"], x["v_cache"], x["cache_len"])
    assert np.max(np.abs(out - ro)) <= ATTN_ATOL
    assert np.max(np.abs(lse - rl)) <= ATTN_LSE_ATOL


def _retrieve_cases():
    rng = np.random.default_rng(20261206)
    out = []
    for _ in range(N_CASES):
        nq, kf = int(rng.integers(1, 5)), int(rng.integers(1, 9))
        # the per-keyframe lists: ceil(keyframes / 128) * 128 * k_frame <= 4096
        cap = (4096 // (128 * kf)) * 128
        nkf = [int(n) if rng.random() > 0.1 else 0 for n in rng.integers(0, cap // nq + 1, nq)]
        out.append((tuple(nkf), int(rng.integers(1, 6000)), 8 * int(rng.integers(8, 97)), kf,
                    int(rng.integers(1, 65))))
    return out


@pytest.mark.parametrize("case", _retrieve_cases(),
                         ids=lambda c: "kf" + "-".join(map(str, c[0])) + "_N%d_E%d_k%d_K%d" % c[1:])
def test_retrieve_random_shapes(case):
    from test_gpu_retrieval import _check_retrieve
    nkf, Nt, E, kf, Kq = case
    offs = np.zeros(len(nkf) + 1, np.int32)
    offs[1:] = np.cumsum(nkf)
    frames = synth.round_f16(synth.normal_f64((int(offs[-1]), E), 9000 + Nt, 1))
    texts = synth.unit_rows_f16(Nt, E, 9000 + Nt, 2)
    _check_retrieve(frames, offs, texts, kf, Kq)


def _keyframe_cases():
    rng = np.random.default_rng(20261207)
    # frames start on 16-byte boundaries: width a multiple of 16 pixels
    return [(int(rng.integers(1, 97)), 16 * int(rng.integers(1, 7)),
             tuple(int(n) for n in rng.integers(0, 40, int(rng.integers(1, 5)))), float(rng.uniform(0.3, 0.9)))
            for _ in range(N_CASES)]


@pytest.mark.parametrize("case", _keyframe_cases(),
                         ids=lambda c: "%dx%d_" % c[:2] + "-".join(map(str, c[2])) + "_t%.2f" % c[3])
def test_keyframes_random_shapes(case):
    from test_gpu_retrieval import _check_keyframes
    h, w, lens, theta = case
    cfg = configs.KF_TINY.with_(height=h, width=w, num_videos=1, frames_range=(1, 1), scene_mean=4.0)
    voffs = np.zeros(len(lens) + 1, np.int32)
    voffs[1:] = np.cumsum(lens)
    T = int(voffs[-1])
    px, _ = synth.video_frames(cfg.with_(frames_range=(max(T, 1), max(T, 1))))
    _check_keyframes(px[:T], voffs, theta)
