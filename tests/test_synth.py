"""The seeded input generator against its published definition (CPU only)."""
import math
import struct

import numpy as np

from paper_2601_01513_gb300 import configs, synth

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def _mix(z):
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def _at(seed, n):
    return _mix((seed + (n + 1) * GAMMA) & M64)


def test_splitmix64_reference_sequence():
    # Vigna's splitmix64.c seeded with 1234567: first outputs of next()
    expected = [6457827717110365317, 3203168211198807973, 9817491932198370423]
    state = 1234567
    for e in expected:
        state = (state + GAMMA) & M64
        assert _mix(state) == e
    for n, e in enumerate(expected):
        assert synth._L().synth_raw(1234567, n) == e


def test_normal_matches_scalar_definition():
    key = synth.stream_key(42, 3)
    assert key == _at(42, 3)
    vals = synth.normal_f64((16,), 42, 3)
    for i in range(16):
        u1 = ((_at(key, 2 * i) >> 11) + 1) * 2.0 ** -53
        u2 = (_at(key, 2 * i + 1) >> 11) * 2.0 ** -53
        assert vals[i] == math.sqrt(-2.0 * math.log(u1)) * math.cos(6.283185307179586 * u2)


def test_bf16_rounding_is_rne_of_fp32():
    x = synth.normal_f64((4096,), 7, 1, 0.0, 3.0)
    bits = synth.round_bf16(x)
    for xi, b in zip(x[:512], bits[:512]):
        f = struct.unpack("<I", struct.pack("<f", float(np.float32(xi))))[0]
        r = (f + 0x7FFF + ((f >> 16) & 1)) >> 16
        assert r == b
    assert np.array_equal(synth.normal_bf16((4096,), 7, 1, 0.0, 3.0), bits)


def test_f16_rounding_single_step():
    x = synth.normal_f64((4096,), 9, 1, 0.0, 0.05)
    assert np.array_equal(synth.round_f16(x), x.astype(np.float16).view(np.uint16))


def test_distribution_and_integers():
    x = synth.normal_f64((200000,), 1, 1)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    t = synth.uniform_i32((200000,), 1, 2, 0, 152064)
    assert t.min() >= 0 and t.max() < 152064
    assert abs(t.mean() / 152064 - 0.5) < 0.01


def test_clip_planting_gives_kept_and_dropped_candidates():
    cfg = configs.V7B
    cand, frames = synth.clip_embeddings(cfg)
    c = cand.view(np.float16).astype(np.float64)
    f = frames.view(np.float16).astype(np.float64)
    cos = np.einsum("qke,qfe->qkf", c, f) / (
        np.linalg.norm(c, axis=-1)[..., None] * np.linalg.norm(f, axis=-1)[:, None, :])
    mx = cos.max(-1)
    kept = (mx >= cfg.threshold).sum()
    assert kept == (cfg.num_cand + 1) // 2
    assert np.all(np.abs(np.linalg.norm(c, axis=-1) - 1) < 1e-2)


def test_ragged_prefix_lengths():
    cfg = configs.BATCH16
    p = synth.prefix_lengths(cfg)
    assert p.shape == (16,) and p.min() >= 4096 and p.max() <= 16384
    assert len(set(p.tolist())) > 8


def test_unit_rows_and_retrieval_inputs():
    from paper_2601_01513_gb300 import configs
    rows = synth.unit_rows_f16(64, 96, 5, 31)
    norms = np.linalg.norm(rows.view(np.float16).astype(np.float64), axis=1)
    assert np.all(np.abs(norms - 1.0) < 2e-3)
    assert np.array_equal(rows, synth.unit_rows_f16(64, 96, 5, 31))
    cfg = configs.RT_TINY
    r = synth.retrieval_inputs(cfg)
    offs = r["frame_offsets"]
    nkf = np.diff(offs)
    assert offs[0] == 0 and np.all(nkf >= cfg.keyframes_range[0]) and np.all(nkf <= cfg.keyframes_range[1])
    assert r["frames"].shape == (offs[-1], cfg.dim) and r["texts"].shape == (cfg.num_texts, cfg.dim)
    r2 = synth.retrieval_inputs(cfg)
    assert all(np.array_equal(r[k], r2[k]) for k in r)


def test_video_frames_are_seeded_and_follow_the_timeline():
    from paper_2601_01513_gb300 import configs
    cfg = configs.KF_TINY
    voffs, fa, fb, fw, ftau, scenes = synth.video_timeline(cfg)
    n = np.diff(voffs)
    assert np.all(n >= cfg.frames_range[0]) and np.all(n <= cfg.frames_range[1])
    assert np.all((fw >= 0) & (fw < 1)) and scenes.shape[1] == 17
    for v in range(cfg.num_videos):                  # a video starts on a fresh scene, no fade
        assert fw[voffs[v]] == 0 and (v == 0 or fa[voffs[v]] != fa[voffs[v] - 1])
    px, vo = synth.video_frames(cfg)
    px2, _ = synth.video_frames(cfg)
    assert px.shape == (voffs[-1], cfg.height, cfg.width, 3) and np.array_equal(px, px2)
    px3, _ = synth.video_frames(cfg, seed=cfg.seed + 1)
    assert not np.array_equal(px, px3)
