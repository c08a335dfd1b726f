"""SM budgets and the side-by-side verify step, through the C ABI, against the fp64 oracle.

An SM budget changes only the grid: the attention's key split (hence which partials the
merge combines) and the LM head's vocabulary slices (hence the order of its per-CTA
log-sum-exp partials).  Every budget must give the oracle's results within the same
tolerances as the default, and the verify step run with the attention beside the LM head
(two streams, each in its budget) must select what the one-after-the-other step selects."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import configs, fvrag, synth
from paper_2601_01513_gb300.pipeline import VerifyStep, plan_sm_split
from gpu_helpers import (ATTN_ATOL, ATTN_LSE_ATOL, LOGPROB_ATOL, check_selection_masked,
                         ensure_built, run_attn, run_lm)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return ensure_built()


def _sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def _attn_inputs(Qn, K, L, Hq, Hkv, D, plens, seed):
    offs = np.zeros(Qn + 1, np.int32)
    offs[1:] = np.cumsum(plens)
    tot = int(offs[-1])
    return (synth.normal_bf16((Qn, K, L, Hq, D), seed, 1), synth.normal_bf16((tot, Hkv, D), seed, 2),
            synth.normal_bf16((tot, Hkv, D), seed, 3), offs,
            synth.normal_bf16((Qn, K, L, Hkv, D), seed, 4), synth.normal_bf16((Qn, K, L, Hkv, D), seed, 5))


@pytest.mark.parametrize("split", [0, fvrag.ATTN_SPLIT_STATIC, fvrag.ATTN_SPLIT_STREAM],
                         ids=["auto", "static", "stream"])
@pytest.mark.parametrize("budget", [1, 2, 3, 5, 7, 20, -1])
@pytest.mark.parametrize("case", [(2, 3, 9, 16, 2, 128, [700, 2049]),    # several tiles, ragged
                                  (1, 5, 16, 28, 4, 128, [1000]),        # 7b-style GQA
                                  (3, 5, 16, 28, 4, 128, [4000, 100, 2500]),   # three ragged queries
                                  (2, 2, 64, 8, 8, 64, [0, 300])],       # D = 64; a query without prefix
                         ids=["ragged2q", "gqa7", "gqa7x3q", "d64"])
def test_attn_budget_matches_oracle(case, budget, split):
    """Every key-split plan at every budget.  Under the streamed plan small budgets give each
    CTA a long share of the tiles' concatenated key lists (tiles cut between CTAs, several
    whole tiles per CTA, one CTA for all at a budget of 1); -1 means the device's own SM count
    given explicitly (the same plan as 0)."""
    b = _sms() if budget == -1 else budget
    q, kp, vp, offs, kt, vt = _attn_inputs(*case, seed=4100 + b)
    out, lse, st = run_attn(q, kp, vp, offs, kt, vt, sm_budget=b, split=split)
    assert st == fvrag.OK
    ref, ref_lse = oracle.verify_attn(q, kp, vp, offs, kt, vt)
    assert np.max(np.abs(out - ref)) <= ATTN_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= ATTN_LSE_ATOL


def test_attn_budget_above_device_rejected():
    q, kp, vp, offs, kt, vt = _attn_inputs(1, 2, 3, 4, 2, 128, [64], seed=1)
    d = fvrag.AttnDesc(1, 2, 3, 4, 2, 128, 64, 64, 0.0, 0, _sms() + 1)
    assert fvrag.attn_workspace_bytes(d) == 0
    with pytest.raises(fvrag.FvragError) as e:
        run_attn(q, kp, vp, offs, kt, vt, sm_budget=_sms() + 1)
    assert e.value.status == fvrag.ERR_INVALID_ARG


@pytest.mark.parametrize("budget", [1, 2, 33, 132])
@pytest.mark.parametrize("case", [(80, 512, 9000, 1),     # one M-tile (the HBM-bound form)
                                  (200, 64, 3000, 2),     # pair form, one pair-tile
                                  (320, 128, 5000, 2),    # vocabulary-major pair form
                                  (512, 96, 7777, 3)],    # pair form, two pair-tiles
                         ids=lambda c: "M%d_H%d_V%d_G%d" % c)
def test_lm_budget_matches_oracle(case, budget):
    """The pair forms take budget // 2 CTA pairs (at least one)."""
    M, H, V, G = case
    seed = 5200 + M + budget
    hid = synth.normal_bf16((M, H), seed, 1)
    W = synth.normal_bf16((V, H), seed, 2, 0.0, 0.2)
    tgt = synth.uniform_i32((M, G), seed, 3, 0, V)
    lp, lse, st = run_lm(hid, W, tgt, sm_budget=budget)
    assert st == fvrag.OK
    ref, ref_lse = oracle.score_logprobs(hid, W, tgt)
    assert np.max(np.abs(lp - ref)) <= LOGPROB_ATOL
    assert np.max(np.abs(lse - ref_lse)) <= LOGPROB_ATOL


def test_lm_budget_full_size_sampled():
    """The 7b LM head in the budget the side-by-side step gives it, on sampled rows."""
    cfg = configs.V7B
    split = plan_sm_split(cfg, _sms())
    assert split is not None
    x = synth.make_inputs(cfg, parts=("lm",))
    lp, lse, st = run_lm(x["hidden"], x["weight"], x["targets"], sm_budget=split[1])
    assert st == fvrag.OK
    rows = np.array([0, 17, 41, cfg.rows - 1])
    ref, ref_lse = oracle.score_logprobs(x["hidden"][rows], x["weight"], x["targets"][rows])
    assert np.max(np.abs(lp[rows] - ref)) <= LOGPROB_ATOL
    assert np.max(np.abs(lse[rows] - ref_lse)) <= LOGPROB_ATOL


def test_attn_budget_full_size_sampled():
    """The 7b attention in the budget the side-by-side step gives it, on sampled rows."""
    cfg = configs.V7B
    split = plan_sm_split(cfg, _sms())
    x = synth.make_inputs(cfg, parts=("attn",))
    out, lse, st = run_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_tail"],
                            x["v_tail"], sm_budget=split[0])
    assert st == fvrag.OK
    sel = np.zeros(x["q"].shape[:-1], bool)
    flat = np.random.default_rng(11).choice(sel.size, 40, replace=False)
    sel.reshape(-1)[flat] = True
    sel.reshape(-1)[0] = sel.reshape(-1)[-1] = True
    ref, ref_lse = oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                      x["k_tail"], x["v_tail"], row_sel=sel)
    assert np.max(np.abs(out[sel] - ref[sel])) <= ATTN_ATOL
    assert np.max(np.abs(lse[sel] - ref_lse[sel])) <= ATTN_LSE_ATOL


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_side_by_side_step_matches_serial(name):
    cfg = configs.PRESETS[name]
    x = synth.make_inputs(cfg)
    par = VerifyStep(cfg)                     # "auto": side by side at these shapes
    par.upload(x)
    assert par.sm_split is not None and sum(par.sm_split) == _sms()
    ser = VerifyStep(cfg, sm_split=None)
    ser.upload(x)
    for s in (par, ser):
        for _ in range(2):
            s.run()
    torch.cuda.synchronize()
    for s in (par, ser):
        assert fvrag.read_status(s.lm_ws) == fvrag.OK and fvrag.read_status(s.attn_ws) == fvrag.OK
    # two oracle-parity results computed with different grids: each is within its tolerance
    # of the oracle, so they agree within twice that; the CLIP results are identical
    assert torch.max(torch.abs(par.out.float() - ser.out.float())).item() <= 2 * ATTN_ATOL
    assert torch.max(torch.abs(par.logprob - ser.logprob)).item() <= 2 * LOGPROB_ATOL
    assert torch.equal(par.max_cos, ser.max_cos) and torch.equal(par.keep, ser.keep)
    _, rmc, _, rkeep = oracle.clip_align(x["cand_emb"], x["frame_emb"], cfg.threshold)
    lp = ser.logprob.cpu().numpy().astype(np.float64)
    if name == "tiny":
        ref_lp, _ = oracle.score_logprobs(x["hidden"], x["weight"], x["targets"])
        assert np.max(np.abs(par.logprob.cpu().numpy() - ref_lp)) <= LOGPROB_ATOL
        ref_out, _ = oracle.verify_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                        x["k_tail"], x["v_tail"])
        assert np.max(np.abs(par.out.float().cpu().numpy() - ref_out)) <= ATTN_ATOL
        lp = ref_lp
    rscore, _ = oracle.select(lp.reshape(cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.gathers),
                              keep=rkeep)
    check_selection_masked(par.selected.cpu().numpy(), rscore, rmc, cfg.threshold)
    # captured as one graph: the same results; end to end from host buffers (its own split,
    # see plan_sm_split(late=True)): the same up to the LM head's summation order
    s_sel, s_score = par.selected.clone(), par.score.clone()
    par.capture()
    par.replay()
    torch.cuda.synchronize()
    assert torch.equal(par.selected, s_sel) and torch.equal(par.score, s_score)
    assert par.sm_split_e2e is not None and sum(par.sm_split_e2e) == _sms()
    sel, sc, _, _ = par.run_from_host(par.host_inputs())
    torch.cuda.synchronize()
    np.testing.assert_allclose(sc.numpy(), s_score.cpu().numpy(), rtol=0, atol=1e-5)
    check_selection_masked(sel.numpy(), rscore, rmc, cfg.threshold)


def test_launch_counter_counts_a_step():
    cfg = configs.TINY
    step = VerifyStep(cfg, sm_split=None)
    step.upload(synth.make_inputs(cfg))
    n = step.launches_per_step()
    parts = sum(VerifyStep.launches_of(f) for f in (step.attention, step.lm_head, step.clip,
                                                    step.select))
    torch.cuda.synchronize()
    assert n == parts
    assert 4 <= n <= 6          # attention (+ merge), LM head + merge, CLIP, selection
