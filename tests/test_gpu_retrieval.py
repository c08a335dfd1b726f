"""GPU parity of keyframe extraction (Eq. 1) and video-to-text retrieval (Eq. 2-3)
against the fp64 oracle, through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import configs, fvrag, synth

from gpu_helpers import COS_ATOL, check_frame_lists, dev_f16, ensure_built, run_keyframes, run_retrieve

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_built()


# --------------------------------------------------------------------------- keyframes

def _check_keyframes(px, voffs, theta, with_hist=True):
    h, s, k, ki, ko, st = run_keyframes(px, voffs, theta, with_hist)
    assert st == fvrag.OK
    oh, osim, okey, oki, oko = oracle.keyframes(px, voffs, theta)
    if with_hist:
        assert np.array_equal(h, oh)
    assert np.array_equal(s, osim.astype(np.float32))     # same fp64 quotient, rounded once
    assert np.array_equal(k, okey)
    assert np.array_equal(ki, oki) and np.array_equal(ko, oko)
    return okey


def test_keyframes_tiny_matches_oracle():
    cfg = configs.KF_TINY
    px, voffs = synth.video_frames(cfg)
    key = _check_keyframes(px, voffs, cfg.theta)
    assert 0 < key.sum() < len(key)
    _check_keyframes(px, voffs, cfg.theta, with_hist=False)


@pytest.mark.parametrize("h,w,lens", [
    (128, 96, [3, 1, 5]),          # 1.5 ring chunks per frame, a one-frame video
    (40, 36, [0, 4, 0, 2]),        # empty videos, a frame smaller than a chunk
    (32, 48, [200, 210]),          # more frames than SMs: CTAs take several frames
])
def test_keyframes_shapes(h, w, lens):
    cfg = configs.KF_TINY.with_(height=h, width=w, num_videos=len(lens), frames_range=(1, 1),
                                scene_mean=5.0)
    voffs = np.zeros(len(lens) + 1, np.int32)
    voffs[1:] = np.cumsum(lens)
    T = int(voffs[-1])
    big = cfg.with_(num_videos=1, frames_range=(max(T, 1), max(T, 1)))
    px, _ = synth.video_frames(big)
    _check_keyframes(px[:T], voffs, 0.6)


def test_keyframes_no_frames_and_threshold_boundary():
    h, s, k, ki, ko, st = run_keyframes(np.zeros((0, 4, 4, 3), np.uint8), [0, 0, 0], 0.5)
    assert st == fvrag.OK and ko.tolist() == [0, 0, 0] and len(ki) == 0
    rng = np.random.default_rng(1)
    a = rng.integers(0, 128, size=(16, 16, 3), dtype=np.uint8)
    b = a.copy()
    b[:8] = 200                                         # half of the pixels move: sim = 0.5 exactly
    px = np.stack([a, b, b, a])
    for theta, expect in ((0.5, [1, 0, 0, 0]), (0.5000001, [1, 1, 0, 1]), (1.0, [1, 1, 0, 1]),
                          (1.0000001, [1, 1, 1, 1])):
        key = _check_keyframes(px, [0, 4], theta)
        assert key.tolist() == expect


@pytest.mark.slow
def test_keyframes_full_size_sampled_videos():
    """All 8 videos of 1280x720 on the GPU; the oracle checks two of them on their own."""
    cfg = configs.KF_720P
    px, voffs = synth.video_frames(cfg)
    h, s, k, ki, ko, st = run_keyframes(px, voffs, cfg.theta, with_hist=True)
    assert st == fvrag.OK
    for v in (0, cfg.num_videos - 1):
        a, b = int(voffs[v]), int(voffs[v + 1])
        oh, osim, okey, oki, oko = oracle.keyframes(px[a:b], [0, b - a], cfg.theta)
        assert np.array_equal(h[a:b], oh)
        assert np.array_equal(s[a:b], osim.astype(np.float32))
        assert np.array_equal(k[a:b], okey)
        assert np.array_equal(ki[ko[v]:ko[v + 1]], oki + a)
    assert np.all(h.sum(axis=1) == cfg.npix)


# --------------------------------------------------------------------------- retrieval

def _oracle_lists(frames, texts, kf):
    oi, osim = oracle.frame_topk(frames, texts, min(kf + 1, texts.shape[0]))
    return lambda f: (oi[f], osim[f])


def _check_retrieve(frames, offs, texts, kf, Kq, precompute=True):
    fi, fs, qi, qs, st = run_retrieve(frames, offs, texts, kf, Kq, precompute)
    assert st == fvrag.OK
    if frames.shape[0] > 0:
        check_frame_lists(fi, fs, texts, frames, _oracle_lists(frames, texts, kf))
    # the per-query union and top-K is exact given the per-keyframe lists
    ei, es = oracle.aggregate_topk(offs, fi, fs.astype(np.float64), Kq)
    assert np.array_equal(qi, ei)
    assert np.array_equal(qs, es.astype(np.float32))
    return fi, fs, qi, qs


def test_retrieve_tiny_matches_oracle():
    cfg = configs.RT_TINY
    r = synth.retrieval_inputs(cfg)
    fi, fs, qi, qs = _check_retrieve(r["frames"], r["frame_offsets"], r["texts"], cfg.k_frame,
                                     cfg.k_query)
    _, _, oqi, oqs = oracle.retrieve(r["frames"], r["frame_offsets"], r["texts"], cfg.k_frame,
                                     cfg.k_query)
    np.testing.assert_allclose(qs, oqs, atol=COS_ATOL)
    assert np.array_equal(qi[:, 0], oqi[:, 0])         # planted texts win by a wide margin
    _check_retrieve(r["frames"], r["frame_offsets"], r["texts"], cfg.k_frame, cfg.k_query,
                    precompute=False)


@pytest.mark.parametrize("nkf,Nt,E,kf,Kq", [
    ([1], 5, 64, 8, 12),            # fewer texts than k_frame: padding on both levels
    ([3, 0, 2], 1000, 200, 3, 3),   # an empty query; E not a multiple of 64
    ([40, 50, 60], 4099, 96, 2, 5), # 150 keyframes: two M-tiles in one group
    ([200, 150, 120], 3001, 64, 1, 64),  # 470 keyframes: two M-tile groups; k_frame = 1
    ([100, 28], 1 << 14, 768, 8, 8),     # k_frame = 8, M = 128 exactly
    ([1024, 1024], 600, 64, 2, 16),      # the most keyframes at k_frame = 2 (16 M-tiles)
    ([300, 212], 2000, 128, 8, 64),      # the most keyframes at k_frame = 8; k_query = 64
    ([150, 130], 3001, 64, 3, 5),        # 280: a last pair-tile of 24 keyframes (M = 128 MMAs)
    ([200, 184], 5000, 96, 2, 8),        # 384: a full last M = 128 pair-tile, 64 per CTA
    ([300, 30], 4099, 200, 8, 16),       # 330: 64 + 10 keyframes in the last pair-tile
    ([600, 500], 700, 64, 2, 4),         # 1100: tail of 76 after four pair-tiles; pairs with
                                         #       no texts (700 texts over 76 pairs)
])
def test_retrieve_shapes(nkf, Nt, E, kf, Kq):
    offs = np.zeros(len(nkf) + 1, np.int32)
    offs[1:] = np.cumsum(nkf)
    frames = synth.round_f16(synth.normal_f64((int(offs[-1]), E), 7, 1))
    texts = synth.unit_rows_f16(Nt, E, 7, 2)
    _check_retrieve(frames, offs, texts, kf, Kq)


def test_retrieve_ties_zero_vectors_and_no_keyframes():
    rng = np.random.default_rng(5)
    base = rng.standard_normal((300, 64))
    texts = np.concatenate([base, base[[17, 3, 17]], np.zeros((2, 64))])  # ids 300-302 duplicate
    texts = synth.round_f16(texts)
    frames = synth.round_f16(np.stack([base[17] * 0.25, base[3], np.zeros(64)]))
    fi, fs, qi, qs = _check_retrieve(frames, np.array([0, 2, 3]), texts, 3, 4)
    assert fi[0, :2].tolist() == [17, 300] and fi[1, :1].tolist() == [3]
    assert fi[2].tolist() == [0, 1, 2] and np.all(fs[2] == 0.0)     # zero keyframe: cos 0
    fi, fs, qi, qs, st = run_retrieve(np.zeros((0, 64), np.uint16), np.array([0, 0]), texts, 3, 2)
    assert st == fvrag.OK and qi.tolist() == [[-1, -1]] and np.all(np.isneginf(qs))


def test_inv_norms_match_numpy():
    x = synth.round_f16(synth.normal_f64((777, 136), 3, 1) * 0.05)
    x[5] = 0
    tx = dev_f16(x)
    inv = torch.full((777,), float("nan"), device="cuda")
    fvrag.embed_inv_norms(tx, inv)
    ref = oracle.decode_f16(x)
    nrm = np.sqrt((ref * ref).sum(axis=1))
    got = inv.cpu().numpy()
    ok = nrm > 0
    np.testing.assert_allclose(got[ok], 1.0 / nrm[ok], rtol=2e-6)
    assert got[5] == 0.0


@pytest.mark.slow
def test_retrieve_full_size_sampled():
    """16 queries against 1,048,576 texts; the oracle scans the corpus for 6 sampled
    keyframes, and the per-query step is checked exactly for every query."""
    cfg = configs.RT_16Q_1M
    r = synth.retrieval_inputs(cfg)
    frames, offs, texts = r["frames"], r["frame_offsets"], r["texts"]
    fi, fs, qi, qs, st = run_retrieve(frames, offs, texts, cfg.k_frame, cfg.k_query)
    assert st == fvrag.OK
    Fr = frames.shape[0]
    sample = np.unique(np.linspace(0, Fr - 1, 6).astype(int))
    oi, osim = oracle.frame_topk(frames[sample], texts, cfg.k_frame + 1)
    check_frame_lists(fi[sample], fs[sample], texts, frames[sample], lambda f: (oi[f], osim[f]))
    ei, es = oracle.aggregate_topk(offs, fi, fs.astype(np.float64), cfg.k_query)
    assert np.array_equal(qi, ei) and np.array_equal(qs, es.astype(np.float32))
    for q in range(cfg.num_queries):                     # the planted relevant text is found
        assert qi[q, 0] in r["relevant"][q]
