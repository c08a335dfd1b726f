"""Pins of the retrieval (Eq. 2-3) and keyframe (Eq. 1) oracle functions (CPU only).

Each oracle function is tied to a library routine (numpy sorting, histogramdd,
torch cosine similarity), a hand-computed case, a closed form or an invariant,
chosen so that a wrong bin boundary, a dropped max, a reversed tie rule or a
comparison of the wrong direction fails at least one test.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import configs, synth


def f16(x):
    return np.asarray(x, dtype=np.float16).view(np.uint16)


# --------------------------------------------------------------------------- Eq. 2 per keyframe

def _library_topk(frames_bits, texts_bits, kf):
    """Cosine via torch, ordering via numpy's stable lexsort (similarity desc, id asc)."""
    a = torch.from_numpy(frames_bits.view(np.float16).astype(np.float64))
    b = torch.from_numpy(texts_bits.view(np.float16).astype(np.float64))
    sim = torch.nn.functional.cosine_similarity(a[:, None, :], b[None, :, :], dim=-1, eps=1e-300).numpy()
    ids = np.arange(sim.shape[1])
    out_i = np.empty((sim.shape[0], kf), np.int32)
    out_s = np.empty((sim.shape[0], kf))
    for f in range(sim.shape[0]):
        order = np.lexsort((ids, -sim[f]))[:kf]
        out_i[f] = order
        out_s[f] = sim[f, order]
    return out_i, out_s


@pytest.mark.parametrize("Fr,Nt,E,kf", [(4, 300, 64, 3), (7, 1000, 96, 5), (3, 50, 16, 1)])
def test_frame_topk_matches_library_sort(Fr, Nt, E, kf):
    frames = synth.round_f16(synth.normal_f64((Fr, E), 11, 1))
    texts = synth.round_f16(synth.normal_f64((Nt, E), 11, 2))
    gi, gs = oracle.frame_topk(frames, texts, kf)
    ri, rs = _library_topk(frames, texts, kf)
    assert np.array_equal(gi, ri)
    np.testing.assert_allclose(gs, rs, rtol=0, atol=1e-12)


def test_frame_topk_ties_go_to_the_smaller_id_and_duplicates_count_once_each():
    rng = np.random.default_rng(3)
    base = rng.standard_normal((6, 32))
    texts = np.concatenate([base, base[[4, 1]]])         # ids 6, 7 duplicate ids 4, 1
    frames = np.stack([base[4] * 0.5, base[1] * 2.0])    # exact parallel copies: cos 1
    gi, gs = oracle.frame_topk(f16(frames), f16(texts), 2)
    assert gi.tolist() == [[4, 6], [1, 7]]
    np.testing.assert_allclose(gs, 1.0, atol=1e-12)
    ri, _ = _library_topk(f16(frames), f16(texts), 2)
    assert np.array_equal(gi, ri)


def test_frame_topk_closed_forms():
    E = 8
    eye = np.eye(E)
    # orthonormal basis: keyframe j has cosine 1 with text j and 0 with all others
    gi, gs = oracle.frame_topk(f16(eye[:3]), f16(eye), 2)
    assert gi[:, 0].tolist() == [0, 1, 2]
    assert np.all(gs[:, 0] == 1.0) and np.all(gs[:, 1] == 0.0)
    # the runner-up among equal zeros is the smallest other id
    assert gi[:, 1].tolist() == [1, 0, 0]
    # a negated text has cosine -1 and comes last; a zero text has cosine 0
    texts = np.stack([-eye[0], np.zeros(E), 3.0 * eye[0]])
    gi, gs = oracle.frame_topk(f16(eye[:1]), f16(texts), 3)
    assert gi.tolist() == [[2, 1, 0]]
    assert gs.tolist() == [[1.0, 0.0, -1.0]]
    # a zero keyframe has cosine 0 with everything: ids in order
    gi, gs = oracle.frame_topk(f16(np.zeros((1, E))), f16(texts), 3)
    assert gi.tolist() == [[0, 1, 2]] and np.all(gs == 0.0)


def test_frame_topk_pads_past_the_corpus_and_is_scale_invariant():
    frames = synth.round_f16(synth.normal_f64((2, 16), 5, 1))
    texts = synth.round_f16(synth.normal_f64((3, 16), 5, 2))
    gi, gs = oracle.frame_topk(frames, texts, 5)
    assert np.all(gi[:, 3:] == -1) and np.all(np.isneginf(gs[:, 3:]))
    assert sorted(gi[0, :3].tolist()) == [0, 1, 2]
    scaled = f16(texts.view(np.float16).astype(np.float64) * 4.0)   # exact in fp16
    gi2, gs2 = oracle.frame_topk(frames, scaled, 5)
    assert np.array_equal(gi, gi2)
    np.testing.assert_allclose(gs2[:, :3], gs[:, :3], rtol=0, atol=1e-14)


# --------------------------------------------------------------------------- Eq. 3 per query

def test_aggregate_by_hand():
    # two keyframes of one query; text 5 is retrieved twice (0.9 and 0.1), text 2 twice (0.5, 0.8)
    idx = np.array([[5, 2, 7], [2, 9, 5]], np.int32)
    sim = np.array([[0.9, 0.5, 0.4], [0.8, 0.6, 0.1]])
    qi, qs = oracle.aggregate_topk(np.array([0, 2]), idx, sim, 3)
    assert qi.tolist() == [[5, 2, 9]]
    assert qs.tolist() == [[0.9, 0.8, 0.6]]
    # all of T: four distinct texts, then padding
    qi, qs = oracle.aggregate_topk(np.array([0, 2]), idx, sim, 6)
    assert qi.tolist() == [[5, 2, 9, 7, -1, -1]]
    assert qs[0, :4].tolist() == [0.9, 0.8, 0.6, 0.4] and np.all(np.isneginf(qs[0, 4:]))


def test_aggregate_ties_queries_and_empty_queries():
    idx = np.array([[8, 3], [3, 8], [1, 4], [6, -1]], np.int32)
    sim = np.array([[0.5, 0.5], [0.7, 0.2], [0.3, 0.3], [0.9, -np.inf]])
    offs = np.array([0, 2, 2, 4])          # query 1 has no keyframes
    qi, qs = oracle.aggregate_topk(offs, idx, sim, 2)
    assert qi[0].tolist() == [3, 8]        # 3 scored 0.7 (max of 0.5, 0.7); 8 scored 0.5
    assert qi[1].tolist() == [-1, -1] and np.all(np.isneginf(qs[1]))
    assert qi[2].tolist() == [6, 1]        # the -1 entry is skipped; 1 before 4 at equal 0.3
    assert qs[2].tolist() == [0.9, 0.3]


def _library_aggregate(offs, idx, sim, Kq):
    """Union with max via numpy's maximum.at, ordering via lexsort."""
    out_i = np.full((len(offs) - 1, Kq), -1, np.int32)
    out_s = np.full((len(offs) - 1, Kq), -np.inf)
    for q in range(len(offs) - 1):
        ii = idx[offs[q]:offs[q + 1]].ravel()
        ss = sim[offs[q]:offs[q + 1]].ravel()
        ok = ii >= 0
        ii, ss = ii[ok], ss[ok]
        uniq, inv = np.unique(ii, return_inverse=True)
        best = np.full(len(uniq), -np.inf)
        np.maximum.at(best, inv, ss)
        order = np.lexsort((uniq, -best))[:Kq]
        out_i[q, :len(order)] = uniq[order]
        out_s[q, :len(order)] = best[order]
    return out_i, out_s


def test_aggregate_matches_library_and_ignores_keyframe_order():
    cfg = configs.RT_TINY
    r = synth.retrieval_inputs(cfg)
    fi, fs = oracle.frame_topk(r["frames"], r["texts"], cfg.k_frame)
    for Kq in (1, 3, 8):
        qi, qs = oracle.aggregate_topk(r["frame_offsets"], fi, fs, Kq)
        li, ls = _library_aggregate(r["frame_offsets"], fi, fs, Kq)
        assert np.array_equal(qi, li)
        assert np.array_equal(qs, ls)
    qi, qs = oracle.aggregate_topk(r["frame_offsets"], fi, fs, 3)
    perm = np.arange(fi.shape[0])
    for q in range(cfg.num_queries):
        a, b = r["frame_offsets"][q], r["frame_offsets"][q + 1]
        perm[a:b] = perm[a:b][::-1]
    pi, ps = oracle.aggregate_topk(r["frame_offsets"], fi[perm], fs[perm], 3)
    assert np.array_equal(pi, qi) and np.array_equal(ps, qs)


def test_planted_texts_are_retrieved():
    """The recipe plants one of each query's relevant texts in about half of its
    keyframes at cosine >= 0.25, well above the background; the query's best
    text must be one of its relevant ones with that planted cosine."""
    cfg = configs.RT_TINY
    r = synth.retrieval_inputs(cfg)
    fi, fs, qi, qs = oracle.retrieve(r["frames"], r["frame_offsets"], r["texts"], cfg.k_frame,
                                     cfg.k_query)
    for q in range(cfg.num_queries):
        assert qi[q, 0] in r["relevant"][q]
        assert qs[q, 0] > 0.24


# --------------------------------------------------------------------------- Eq. 1 keyframes

def test_histogram_matches_histogramdd():
    px = np.random.default_rng(7).integers(0, 256, size=(5, 40, 3), dtype=np.uint8)
    px[0, :8] = [[31, 32, 255]] * 8                 # bin edges on every channel
    hist, _, _, _, _ = oracle.keyframes(px, np.array([0, 5]), 0.5)
    for t in range(5):
        ref, _ = np.histogramdd(px[t].astype(np.float64), bins=(8, 8, 8), range=[(0, 256)] * 3)
        assert np.array_equal(hist[t], ref.astype(np.int64).ravel())
        assert hist[t].sum() == 40


def test_keyframes_by_hand():
    # frame 0 bins: (0,0,0)->0 twice, (32,0,0)->64, (255,255,255)->511
    # frame 1 bins: (0,0,0)->0, (100,0,0)->192, (32,5,5)->64, (224,224,224)->511
    f0 = [(0, 0, 0), (31, 31, 31), (32, 0, 0), (255, 255, 255)]
    f1 = [(0, 0, 0), (100, 0, 0), (32, 5, 5), (224, 224, 224)]
    px = np.array([f0, f1], dtype=np.uint8)
    hist, sim, key, kidx, koffs = oracle.keyframes(px, np.array([0, 2]), 0.75)
    assert hist[0, 0] == 2 and hist[0, 64] == 1 and hist[0, 511] == 1 and hist[0].sum() == 4
    assert hist[1, 0] == 1 and hist[1, 192] == 1 and hist[1, 64] == 1 and hist[1, 511] == 1
    assert sim.tolist() == [0.0, 0.75]               # min(2,1) + min(1,1) + min(1,1) = 3 of 4
    assert key.tolist() == [1, 0]                     # strict <: 0.75 is not below 0.75
    _, _, key, kidx, koffs = oracle.keyframes(px, np.array([0, 2]), 0.7500001)
    assert key.tolist() == [1, 1] and kidx.tolist() == [0, 1] and koffs.tolist() == [0, 2]


def test_keyframes_closed_forms_and_video_boundaries():
    rng = np.random.default_rng(9)
    a = rng.integers(0, 128, size=(64, 3), dtype=np.uint8)          # every channel < 128
    b = a.copy()
    b[:32] = 200                                                     # half the pixels to bin 7,7,7
    c = np.full((64, 3), 250, np.uint8)                              # all in bin 511
    d = rng.permutation(a)                                           # same pixels, shuffled
    px = np.stack([a, a, b, d, c, a])
    hist, sim, key, kidx, koffs = oracle.keyframes(px, np.array([0, 4, 6]), 0.6)
    assert sim[1] == 1.0                 # identical frames
    assert sim[2] == 0.5                 # half of the mass moved to an unused bin
    assert sim[3] == 0.5                 # shuffling pixels changes no histogram
    assert sim[4] == 0.0                 # first frame of video 1
    assert sim[5] == 0.0                 # disjoint colours
    assert key.tolist() == [1, 0, 1, 1, 1, 1]
    assert kidx.tolist() == [0, 2, 3, 4, 5] and koffs.tolist() == [0, 3, 5]
    assert np.array_equal(hist[3], hist[0])


def test_keyframes_of_synthetic_videos_follow_the_scene_schedule():
    """Hard cuts in the recipe's videos are keyframes; frames inside a scene are not."""
    cfg = configs.KF_TINY
    voffs, fa, fb, fw, ftau, scenes = synth.video_timeline(cfg)
    px, voffs2 = synth.video_frames(cfg)
    assert np.array_equal(voffs, voffs2)
    _, sim, key, kidx, koffs = oracle.keyframes(px, voffs, cfg.theta)
    assert koffs[0] == 0 and koffs[-1] == len(kidx)
    for v in range(cfg.num_videos):
        assert key[voffs[v]] == 1
        assert np.all(np.diff(kidx[koffs[v]:koffs[v + 1]]) > 0)
    for t in range(1, len(fa)):
        if t in voffs:
            continue
        steady = fa[t] == fa[t - 1] and fw[t] == 0 and fw[t - 1] == 0
        if steady:
            assert sim[t] > 0.6, t
