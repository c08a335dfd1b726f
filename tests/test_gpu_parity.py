"""GPU parity: every libfvrag call, through the C ABI, against the fp64 oracle on the
same seeded inputs.  Small cases compare every element and span several tiles with
ragged tails; the full-size workloads compare sampled rows the oracle computes one
by one (in the launch configuration the benchmark uses) plus size-independent
properties; the whole verify step is compared on every row at every workload.
Tolerances: attention |diff| <= 2e-2, log-prob |diff| <= 1e-2,
cosine |diff| <= 1e-3; integer decisions exact unless the oracle's margin is
below the tolerance."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import configs, fvrag, synth
from paper_2601_01513_gb300.pipeline import VerifyStep

from gpu_helpers import (ATTN_ATOL, ATTN_LSE_ATOL, COS_ATOL, LOGPROB_ATOL, check_argmax_with_margin,
                         check_keep_with_margin, check_selection_masked, ensure_built, run_attn,
                         run_clip, run_lm, run_select)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return ensure_built()


# ============================================================ attention
def _attn_inputs(Qn, K, L, Hq, Hkv, D, plens, seed):
    offs = np.zeros(Qn + 1, np.int32)
    offs[1:] = np.cumsum(plens)
    tot = int(offs[-1])
    return (synth.normal_bf16((Qn, K, L, Hq, D), seed, 1), synth.normal_bf16((tot, Hkv, D), seed, 2),
            synth.normal_bf16((tot, Hkv, D), seed, 3), offs,
            synth.normal_bf16((Qn, K, L, Hkv, D), seed, 4), synth.normal_bf16((Qn, K, L, Hkv, D), seed, 5))


ATTN_CASES = [
    # Qn, K, L, Hq, Hkv, D, prefix lengths
    (1, 4, 8, 8, 8, 64, [256]),            # tiny config shape
    (1, 3, 5, 14, 2, 128, [0]),            # no prefix: tail only
    (1, 2, 1, 4, 4, 64, [1]),              # one prefix key, L = 1
    (1, 2, 3, 4, 1, 128, [63]),
    (1, 2, 3, 4, 2, 128, [64]),
    (1, 2, 3, 8, 2, 64, [65]),
    (1, 2, 33, 4, 4, 128, [257]),          # L = 33 (two lanes' worth of tail keys)
    (3, 2, 4, 12, 4, 128, [0, 130, 70]),   # ragged queries
    (1, 5, 16, 28, 4, 128, [1000]),        # 7b-style GQA: 5 row tiles of 18 tokens x 7 heads
    (2, 3, 9, 16, 2, 128, [700, 2049]),    # 8 heads per KV head, several key splits
    (1, 2, 64, 8, 8, 64, [300]),           # longest supported tail
    (1, 2, 3, 128, 1, 64, [200]),          # hq / hkv = 128: one token per row tile
    # several row tiles per KV head, D = 128
    (1, 3, 16, 16, 2, 128, [500]),         # 3 tiles of 16 tokens x 8 heads
    (2, 4, 16, 16, 2, 128, [300, 1111]),   # 4 tiles, ragged prefixes, several key splits
    (1, 2, 40, 8, 1, 128, [129]),          # 5 tiles, tiles spanning two candidates
    (1, 8, 8, 28, 4, 128, [0]),            # no prefix: own blocks only
    (3, 5, 16, 28, 4, 128, [4000, 100, 2500]),   # 7b-style GQA over three ragged queries
]


@pytest.mark.parametrize("case", ATTN_CASES, ids=lambda c: "x".join(map(str, c[:6])) + "_P" + "-".join(map(str, c[6])))
def test_attn_matches_oracle(case):
    Qn, K, L, Hq, Hkv, D, plens = case
    q, kp, vp, offs, kt, vt = _attn_inputs(Qn, K, L, Hq, Hkv, D, plens, seed=1000 + sum(plens) + L)
    out, lse, st = run_attn(q, kp, vp, offs, kt, vt)
    assert st == fvrag.OK
    ref, ref_lse = oracle.verify_attn(q, kp, vp, offs, kt, vt)
    assert np.all(np.isfinite(out))
    assert np.max(np.abs(out - ref)) <= ATTN_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= ATTN_LSE_ATOL


def test_attn_custom_scale_and_no_lse():
    q, kp, vp, offs, kt, vt = _attn_inputs(1, 2, 4, 8, 2, 128, [150], seed=5)
    out, _, st = run_attn(q, kp, vp, offs, kt, vt, with_lse=False, scale=0.05)
    ref, _ = oracle.verify_attn(q, kp, vp, offs, kt, vt, scale=0.05)
    assert st == fvrag.OK and np.max(np.abs(out - ref)) <= ATTN_ATOL


def _sample_rows(shape, n, seed):
    rng = np.random.default_rng(seed)
    sel = np.zeros(shape, bool)
    flat = rng.choice(sel.size, size=min(n, sel.size), replace=False)
    sel.reshape(-1)[flat] = True
    # always include the first and the last row (edges of the row tiling)
    sel.reshape(-1)[0] = sel.reshape(-1)[-1] = True
    return sel


def _row_tile_sel(shape, hkv, tiles):
    """Rows of whole attention row tiles: for every query and KV head, the listed tiles of
    T = 128 // (hq / hkv) candidate tokens (in (k, l) order) x the heads sharing that KV head."""
    Qn, K, L, hq = shape
    grp = hq // hkv
    T = max(1, 128 // grp)
    n_tiles = -(-(K * L) // T)
    sel = np.zeros((Qn, K * L, hq), bool)
    for t in tiles:
        t = t % n_tiles
        for g in range(hkv):
            sel[:, t * T:(t + 1) * T, g * grp:(g + 1) * grp] = True
    return sel.reshape(shape)


@pytest.mark.parametrize("name", ["7b", "long", "batch16", "72b"])
@pytest.mark.parametrize("split", [0, fvrag.ATTN_SPLIT_STATIC, fvrag.ATTN_SPLIT_STREAM],
                         ids=["auto", "static", "stream"])
def test_attn_full_size(name, split):
    """Full-size attention alone on all SMs: every row at 7b and long; at batch16 and 72b
    the first and the last (ragged) row tile of every query and KV head plus sampled rows
    (every row of those two is checked by the whole-step test)."""
    cfg = configs.PRESETS[name]
    x = synth.make_inputs(cfg, parts=("attn",))
    out, lse, st = run_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_tail"],
                            x["v_tail"], split=split)
    assert st == fvrag.OK
    assert np.all(np.isfinite(out)) and np.all(np.isfinite(lse))
    shape = x["q"].shape[:-1]
    if name in ("7b", "long"):
        sel = np.ones(shape, bool)
    else:
        sel = _row_tile_sel(shape, cfg.hkv, (0, -1)) | _sample_rows(shape, 48, seed=7)
    ref, ref_lse = oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                      x["k_tail"], x["v_tail"], row_sel=sel)
    assert np.max(np.abs(out[sel] - ref[sel])) <= ATTN_ATOL
    assert np.max(np.abs(lse[sel] - ref_lse[sel])) <= ATTN_LSE_ATOL
    # size-independent property: every output is a convex combination of V rows
    assert np.max(np.abs(out)) <= 8.0


# ============================================================ LM head
LM_CASES = [
    # M, H, V, G
    (32, 512, 4096, 1),       # tiny config shape
    (1, 64, 16, 1),           # smallest: one row, one 16-row vocabulary unit
    (33, 72, 1007, 2),        # H not a multiple of 64; V not a multiple of 16
    (128, 128, 5000, 8),      # one full M-tile, 8 gathers
    (129, 256, 4103, 1),      # two M-tiles (second with one row)
    (300, 192, 3001, 2),      # 257-384 rows: the vocabulary-major pair form (Mp = 320)
    (257, 64, 50021, 1),      # vocabulary-major, Mp = 288 (boxes of 72 rows); ~1.3 tiles per pair
    (384, 96, 10007, 8),      # vocabulary-major, Mp = 384 (two accumulator ranges sharing 256 columns)
    (320, 8192, 5000, 1),     # the 72b shape's rows and hidden size, small vocabulary
    (352, 136, 40000, 3),     # vocabulary-major, Mp = 352; H not a multiple of 64
    (290, 64, 40, 2),         # vocabulary-major with 3 pairs of 16 rows: most lanes past the range
    (320, 64, 152064, 1),     # vocabulary-major over the full vocabulary: 8 tiles per pair
    (512, 96, 7777, 3),       # four M-tiles: one pass of two CTA-pair tiles (2-SM MMAs)
    (600, 128, 50021, 2),     # three pair tiles (the last one partly empty), ragged W tiles
    (200, 64, 3000, 8),       # one pair tile, two accumulator sets; 8 gathers per row
    (400, 72, 30001, 8),      # two pair tiles per pass; 8 gathers; H not a multiple of 64
    (80, 3584, 9000, 1),      # 7b hidden size, small vocabulary
    (2048, 64, 1000, 1),      # the most rows supported: 8 pair tiles in 4 passes
]


@pytest.mark.parametrize("case", LM_CASES, ids=lambda c: "M%d_H%d_V%d_G%d" % c)
def test_lm_matches_oracle(case):
    M, H, V, G = case
    seed = 2000 + M + V
    hid = synth.normal_bf16((M, H), seed, 1)
    W = synth.normal_bf16((V, H), seed, 2, 0.0, 0.02 if H > 1000 else 0.2)
    tgt = synth.uniform_i32((M, G), seed, 3, 0, V)
    if M > 2:  # out-of-range ids give NaN
        tgt[1, 0] = -1
        tgt[2, G - 1] = V
    lp, lse, st = run_lm(hid, W, tgt)
    assert st == fvrag.OK
    ref, ref_lse = oracle.score_logprobs(hid, W, tgt)
    assert np.array_equal(np.isnan(lp), np.isnan(ref))
    ok = ~np.isnan(ref)
    assert np.max(np.abs(lp[ok] - ref[ok])) <= LOGPROB_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= LOGPROB_ATOL


@pytest.mark.parametrize("M", [3, 300])
def test_lm_all_targets_sum_to_one(M):
    """Gathering every vocabulary id of a row: sum of probabilities is 1 (any size)."""
    H, V = 128, 8
    hid = synth.normal_bf16((M, H), 5, 1)
    W = synth.normal_bf16((V, H), 5, 2, 0.0, 0.3)
    tgt = np.tile(np.arange(V, dtype=np.int32), (M, 1))
    lp, _, st = run_lm(hid, W, tgt)
    assert st == fvrag.OK
    np.testing.assert_allclose(np.exp(lp.astype(np.float64)).sum(1), 1.0, atol=1e-4)


@pytest.mark.parametrize("M", [40, 300])
def test_lm_growing_logits_match_oracle(M):
    """Logits whose scale grows along the vocabulary (W row v scaled by 1 + 6 v / V), so
    later vocabulary tiles keep passing the running maxima of earlier ones: the online
    log-sum-exp rescales (and the vocabulary-major form raises its reference max) often."""
    H, V, G = 128, 30011, 2
    hid = synth.normal_bf16((M, H), 77 + M, 1)
    W = synth.bf16_bits_to_f32(synth.normal_bf16((V, H), 77 + M, 2, 0.0, 0.3)).astype(np.float64)
    W = synth.round_bf16(W * (1.0 + 6.0 * np.arange(V, dtype=np.float64) / V)[:, None])
    tgt = synth.uniform_i32((M, G), 77 + M, 3, 0, V)
    lp, lse, st = run_lm(hid, W, tgt)
    assert st == fvrag.OK
    ref, ref_lse = oracle.score_logprobs(hid, W, tgt)
    assert np.max(np.abs(lp - ref)) <= LOGPROB_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= LOGPROB_ATOL


@pytest.mark.parametrize("name", ["7b", "long", "72b", "batch16"])
def test_lm_full_size_sampled(name):
    cfg = configs.PRESETS[name]
    x = synth.make_inputs(cfg, parts=("lm",))
    lp, lse, st = run_lm(x["hidden"], x["weight"], x["targets"])
    assert st == fvrag.OK
    assert np.all(np.isfinite(lp)) and np.all(lp <= 0)
    rows = np.unique(np.concatenate([[0, cfg.rows - 1], np.random.default_rng(3).choice(cfg.rows, 6, replace=False)]))
    ref, ref_lse = oracle.score_logprobs(x["hidden"][rows], x["weight"], x["targets"][rows])
    assert np.max(np.abs(lp[rows] - ref)) <= LOGPROB_ATOL
    assert np.max(np.abs(lse[rows] - ref_lse)) <= LOGPROB_ATOL


# ============================================================ CLIP
@pytest.mark.parametrize("name", ["tiny", "7b", "long", "batch16", "72b"])
def test_clip_configs(name):
    cfg = configs.PRESETS[name]
    cand, frames = synth.clip_embeddings(cfg)
    cos, mc, am, keep = run_clip(cand, frames, cfg.threshold)
    rcos, rmc, ram, rkeep = oracle.clip_align(cand, frames, cfg.threshold)
    assert np.max(np.abs(cos - rcos)) <= COS_ATOL
    assert np.max(np.abs(mc - rmc)) <= COS_ATOL
    check_argmax_with_margin(am, rcos)
    check_keep_with_margin(keep, rmc, cfg.threshold)
    assert keep.sum() >= 1


def test_clip_edges():
    E = 8
    eye = np.eye(E)
    cand = synth.round_f16(eye[None, :3] * 3.0)
    frames = synth.round_f16(eye[None, 3:7] * 0.5)
    frames[0, 2] = cand[0, 1]
    frames[0, 3] = cand[0, 1]          # tie: lowest index wins
    cand[0, 2] = 0                     # zero vector: cos 0
    cos, mc, am, keep = run_clip(cand, frames, 0.2)
    assert am[0, 1] == 2 and abs(mc[0, 1] - 1.0) < 1e-6 and keep[0, 1] == 1
    assert np.all(cos[0, 2] == 0.0) and keep[0, 2] == 0 and am[0, 2] == 0
    assert np.all(cos[0, 0] == 0.0)
    # one frame only, and a dimension that is not a multiple of 256
    c1 = synth.round_f16(synth.normal_f64((2, 3, 40), 9, 1))
    f1 = synth.round_f16(synth.normal_f64((2, 1, 40), 9, 2))
    cos, mc, am, keep = run_clip(c1, f1, 0.0, with_cos=True)
    rcos, rmc, _, _ = oracle.clip_align(c1, f1, 0.0)
    assert np.all(am == 0) and np.max(np.abs(mc - rmc)) <= COS_ATOL
    # without the optional cos output
    _, mc2, am2, _ = run_clip(c1, f1, 0.0, with_cos=False)
    assert np.array_equal(mc2, mc) and np.array_equal(am2, am)


@pytest.mark.parametrize("Qn,K,F,E", [
    (2, 13, 300, 64),      # two candidate groups of a CTA; frames over a cluster of 2
    (3, 8, 4096, 768),     # clusters of 8 CTAs per query
    (1, 1, 1, 8),          # one frame, the smallest dimension
    (1, 9, 2, 4096),       # the largest dimension (a 2-deep copy ring)
    (16, 10, 4096, 768),   # the CLIP bandwidth-sweep size
    (2, 16, 100, 1536),    # the largest dimension with an 8-deep ring
    (1, 5, 700, 2048),     # a 4-deep ring; frames over a cluster of 4
])
def test_clip_shapes(Qn, K, F, E):
    cand = synth.round_f16(synth.normal_f64((Qn, K, E), 31 + K, 1))
    frames = synth.round_f16(synth.normal_f64((Qn, F, E), 31 + K, 2))
    frames[:, F // 2] = cand[:, 0]                     # a planted exact match
    cos, mc, am, keep = run_clip(cand, frames, 0.2)
    rcos, rmc, ram, rkeep = oracle.clip_align(cand, frames, 0.2)
    assert np.max(np.abs(cos - rcos)) <= COS_ATOL
    assert np.max(np.abs(mc - rmc)) <= COS_ATOL
    check_argmax_with_margin(am, rcos)
    check_keep_with_margin(keep, rmc, 0.2)
    assert np.all(am[:, 0] == F // 2)


def test_clip_ties_across_a_cluster():
    """Equal cosines in frames held by different CTAs of a cluster: the lowest index wins."""
    E, F = 64, 1024
    rng = np.random.default_rng(4)
    x = synth.round_f16(rng.standard_normal(E))
    y = synth.round_f16(rng.standard_normal(E))
    cand = np.stack([x, y, 2 * x])[None]
    frames = np.repeat(x[None, None], F, axis=1)       # every frame equals candidate 0 ...
    frames[0, 700] = y                                 # ... but two equal to candidate 1,
    frames[0, 900] = y                                 # held by different CTAs
    cos, mc, am, keep = run_clip(cand, frames, 0.0, with_cos=False)
    assert am[0, 0] == 0 and am[0, 2] == 0             # all maxima equal: the first frame
    assert am[0, 1] == 700


# ============================================================ selection
ALL_MODES = [fvrag.SEL_MASKED_MEAN_LOGPROB, fvrag.SEL_TWO_STAGE, fvrag.SEL_ADDITION, fvrag.SEL_INVERT,
             fvrag.SEL_RELIABILITY_ONLY, fvrag.SEL_ALIGNMENT_ONLY, fvrag.SEL_RANDOM]


@pytest.mark.parametrize("mode", ALL_MODES)
@pytest.mark.parametrize("Qn,K,L", [(1, 1, 1), (3, 7, 5), (16, 5, 16), (2, 1000, 3), (600, 10, 2),
                                    (1, 1024, 2)])
def test_select_matches_oracle(mode, Qn, K, L):
    lp, keep, mc = synth.selection_inputs(Qn, K, L, 2, seed=Qn * 31 + K)
    lengths = synth.uniform_i32((Qn, K), 77, 1, 0, L + 2)   # includes invalid 0 and L+1
    delta = float(np.float32(0.05))
    seed = 0xD1B54A32D192ED03 + Qn
    for lens in (None, lengths):
        score, sel = run_select(lp, mode, keep=keep, max_cos=mc, lengths=lens, delta=delta, seed=seed)
        rscore, rsel = oracle.select(lp, mode=mode, lengths=lens, keep=keep, max_cos=mc, delta=delta,
                                     seed=seed)
        assert np.array_equal(np.isnan(score), np.isnan(rscore))
        ok = ~np.isnan(rscore)
        assert np.array_equal(score[ok], rscore[ok].astype(np.float32))   # fp64 on both sides
        assert np.array_equal(sel, rsel)


def test_select_two_stage_nan_alignment():
    """A NaN max_cos ranks below every number when the best-aligned member of A_H is
    chosen (Algorithm 1): same pick as the oracle, including an all-NaN A_H."""
    rel = np.array([[0.7, 0.7, 0.7, 0.1], [0.6, 0.6, 0.2, 0.6], [0.5, 0.5, 0.5, 0.5]])
    lp = np.stack([np.log(rel), np.log1p(-rel)], -1)[:, :, None, :]
    mc = np.array([[np.nan, 0.3, 0.2, 0.99], [0.1, np.nan, 0.9, -np.inf],
                   [np.nan, np.nan, np.nan, np.nan]])
    _, sel = run_select(lp, fvrag.SEL_TWO_STAGE, max_cos=mc, delta=0.05)
    _, rsel = oracle.select(lp.astype(np.float32), mode=oracle.SEL_TWO_STAGE,
                            max_cos=mc.astype(np.float32), delta=float(np.float32(0.05)))
    assert np.array_equal(sel, rsel) and list(sel) == [1, 0, 0]


def test_select_case_studies_on_gpu():
    import json, os
    here = os.path.join(os.path.dirname(__file__), "golden")
    for name in ("case_penguin.json", "case_cuttlefish.json"):
        case = json.load(open(os.path.join(here, name)))
        rel = np.array(case["reliability"])
        lp = np.stack([np.log(rel), np.log1p(-rel)], -1)[None, :, None, :]
        _, sel = run_select(lp, fvrag.SEL_TWO_STAGE, max_cos=np.array([case["max_cos"]]),
                            delta=case["delta"])
        assert sel[0] == case["expected_selected"]


# ============================================================ whole step
def _oracle_step(cfg, x):
    """The oracle's verify step on every row: attention, LM-head log-probs, CLIP and the
    masked mean selection computed from the oracle's own log-probs and keep flags."""
    out, alse = oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                   x["k_tail"], x["v_tail"])
    lp, lse = oracle.score_logprobs(x["hidden"], x["weight"], x["targets"])
    cos, mc, am, keep = oracle.clip_align(x["cand_emb"], x["frame_emb"], cfg.threshold)
    score, sel = oracle.select(lp.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.gathers),
                               keep=keep)
    return dict(out=out, alse=alse, lp=lp, lse=lse, cos=cos, mc=mc, keep=keep, score=score, sel=sel)


def _check_step_result(cfg, ref, score, selected):
    """score within the log-prob tolerance of the oracle's (a mean of values each within it);
    selected valid under some resolution of the keeps the oracle cannot decide."""
    assert np.max(np.abs(score - ref["score"])) <= LOGPROB_ATOL
    check_selection_masked(selected, ref["score"], ref["mc"], cfg.threshold)


@pytest.mark.parametrize("name", ["tiny", "7b", pytest.param("long", marks=pytest.mark.slow),
                                  pytest.param("batch16", marks=pytest.mark.slow),
                                  pytest.param("72b", marks=pytest.mark.slow)])
def test_pipeline_step_matches_oracle(name):
    """The whole verify step at every workload, in the form the benchmark times (the four
    calls captured in one CUDA graph, with the workload's own SM split or serial order),
    against the oracle on every row; then the end-to-end form from pinned host buffers
    (its own SM split) against the same oracle results."""
    cfg = configs.PRESETS[name]
    x = synth.make_inputs(cfg)
    step = VerifyStep(cfg)
    step.upload(x)
    step.capture()
    for _ in range(2):            # repeated steps reuse the workspaces
        step.replay()
    torch.cuda.synchronize()
    assert fvrag.read_status(step.lm_ws) == fvrag.OK
    assert fvrag.read_status(step.attn_ws) == fvrag.OK
    ref = _oracle_step(cfg, x)
    # LM head: every row, every gather
    lp = step.logprob.cpu().numpy()
    assert np.all(np.isfinite(lp)) and np.all(lp <= 0)
    assert np.max(np.abs(lp - ref["lp"])) <= LOGPROB_ATOL
    assert np.max(np.abs(step.lm_lse.cpu().numpy() - ref["lse"])) <= LOGPROB_ATOL
    # attention: every row of every head
    out = step.out.float().cpu().numpy()
    assert np.max(np.abs(out - ref["out"])) <= ATTN_ATOL
    assert np.max(np.abs(step.attn_lse.cpu().numpy() - ref["alse"])) <= ATTN_LSE_ATOL
    # CLIP
    assert np.max(np.abs(step.max_cos.cpu().numpy() - ref["mc"])) <= COS_ATOL
    check_argmax_with_margin(step.argmax.cpu().numpy(), ref["cos"])
    check_keep_with_margin(step.keep.cpu().numpy(), ref["mc"], cfg.threshold)
    # selection from the step's own outputs, against the oracle's scores
    _check_step_result(cfg, ref, step.score.cpu().numpy(), step.selected.cpu().numpy())
    # end to end from pinned host buffers (copies inside the step)
    host = step.host_inputs()
    for _ in range(2):
        sel, sc, _, _ = step.run_from_host(host)
        torch.cuda.synchronize()
        _check_step_result(cfg, ref, sc.numpy().copy(), sel.numpy().copy())
    assert fvrag.read_status(step.lm_ws) == fvrag.OK
    assert fvrag.read_status(step.attn_ws) == fvrag.OK


def test_pipeline_end_to_end_from_host():
    cfg = configs.TINY
    x = synth.make_inputs(cfg)
    step = VerifyStep(cfg)
    step.upload(x)
    host = step.host_inputs()
    sel, sc, h2d, d2h = step.run_from_host(host)
    torch.cuda.synchronize()
    ref_sel, ref_sc = step.selected.cpu().numpy().copy(), step.score.cpu().numpy().copy()
    assert np.array_equal(sel.numpy(), ref_sel) and np.array_equal(sc.numpy(), ref_sc)
    assert h2d >= sum(v.numel() * v.element_size() for v in host.values())
    assert d2h >= cfg.num_queries * 4 + cfg.num_queries * cfg.num_cand * 4
    # new inputs written into the host views travel with the one copy of the arena
    host["targets"].copy_((host["targets"] + 1) % cfg.vocab)
    _, sc2, _, _ = step.run_from_host(host)
    torch.cuda.synchronize()
    got = sc2.numpy().copy()
    assert not np.array_equal(got, ref_sc)
    assert torch.equal(step.t["targets"].cpu(), host["targets"])
    # the device step may split the SMs differently from the host-input path (the LM head's
    # per-CTA partials then add up in another order): equal to fp32 rounding
    step.run()
    torch.cuda.synchronize()
    np.testing.assert_allclose(step.score.cpu().numpy(), got, rtol=0, atol=1e-5)
    # the same sequence launched directly on a stream (no graph) gives the same result
    host["targets"].copy_((host["targets"] + 1) % cfg.vocab)
    _, sc3, _, _ = step.run_from_host(host, stream=torch.cuda.current_stream())
    torch.cuda.synchronize()
    got3 = sc3.numpy().copy()
    step.run()
    torch.cuda.synchronize()
    np.testing.assert_allclose(step.score.cpu().numpy(), got3, rtol=0, atol=1e-5)
    assert not np.allclose(got3, got, rtol=0, atol=1e-3)
    # a plain dict of host tensors takes the tensor-by-tensor path
    plain = {k: v.clone() for k, v in host.items()}
    _, sc4, h2d4, _ = step.run_from_host(plain)
    torch.cuda.synchronize()
    np.testing.assert_allclose(sc4.numpy(), got3, rtol=0, atol=1e-5)
    assert h2d4 == sum(v.numel() * v.element_size() for v in plain.values())


# ============================================================ failure detection
def test_bounded_wait_times_out_and_context_survives():
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    old = fvrag.get_wait_limit_ns()
    try:
        fvrag.set_wait_limit_ns(2_000_000)       # 2 ms
        fvrag.selftest_wait_timeout(ws)
        assert fvrag.read_status(ws) == fvrag.ERR_TIMEOUT
        fvrag.clear_status(ws)
        assert fvrag.read_status(ws) == fvrag.OK
    finally:
        fvrag.set_wait_limit_ns(old)
    # the context is still usable: a normal call succeeds with a clean status
    hid = synth.normal_bf16((4, 64), 1, 1)
    W = synth.normal_bf16((64, 64), 1, 2)
    tgt = synth.uniform_i32((4, 1), 1, 3, 0, 64)
    lp, _, st = run_lm(hid, W, tgt)
    assert st == fvrag.OK and np.all(np.isfinite(lp))
