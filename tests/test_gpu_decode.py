"""GPU parity of the drafter decode step (Eq. 5, Eq. 8-10) against the fp64 oracle,
through the C ABI."""
import numpy as np
import pytest

from oracle import oracle
from paper_2601_01513_gb300 import configs, fvrag, synth

from gpu_helpers import ATTN_ATOL, ATTN_LSE_ATOL, ensure_built, run_decode

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ensure_built()


def _check(x, scale=0.0):
    out, lse, st = run_decode(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"], x["k_cache"],
                              x["v_cache"], x["cache_len"], scale=scale)
    assert st == fvrag.OK
    ro, rl = oracle.decode_attn(x["q"], x["k_prefix"], x["v_prefix"], x["prefix_offsets"],
                                x["k_cache"], x["v_cache"], x["cache_len"], scale=scale)
    assert np.max(np.abs(out - ro)) <= ATTN_ATOL
    assert np.max(np.abs(lse - rl)) <= ATTN_LSE_ATOL
    return out


def test_decode_tiny_matches_oracle():
    _check(synth.decode_inputs(configs.DEC_TINY))


@pytest.mark.parametrize("Qn,K,hq,hkv,D,pr,C,cr", [
    (1, 5, 28, 4, 128, (8192, 8192), 200, (1, 200)),     # 7B-class heads, C not a block multiple
    (2, 20, 16, 2, 128, (0, 700), 64, (64, 64)),         # two row tiles; full caches; P may be 0
    (3, 4, 8, 1, 64, (100, 900), 300, (1, 1)),           # MQA, D = 64, only the newest token
    (1, 7, 2, 2, 128, (5000, 5000), 2048, (1500, 2048)), # long caches spread over many runs
    (1, 2, 4, 1, 64, (0, 0), 8192, (8000, 8192)),        # no prefix at all, 8K caches
    (170, 2, 4, 2, 64, (0, 600), 96, (1, 96)),           # 340 row tiles: a grid of 3 waves
    (1, 1, 1, 1, 64, (300000, 300000), 64, (1, 64)),     # one tile cut into the most runs (64)
])
def test_decode_shapes(Qn, K, hq, hkv, D, pr, C, cr):
    cfg = configs.DEC_TINY.with_(num_queries=Qn, num_drafts=K, hq=hq, hkv=hkv, head_dim=D,
                                 prefix_range=pr, cache_cap=C, cache_range=cr, seed=17 + K)
    _check(synth.decode_inputs(cfg))


def test_decode_ignores_slots_past_the_cache_length_and_scale():
    x = synth.decode_inputs(configs.DEC_TINY)
    big = synth.round_bf16(np.full((1,), 3.0e4))[0]
    for qi in range(x["q"].shape[0]):
        for k in range(x["q"].shape[1]):
            n = x["cache_len"][qi, k]
            x["k_cache"][qi, k, n:] = big
            x["v_cache"][qi, k, n:] = big
    _check(x)
    _check(x, scale=0.05)


@pytest.mark.slow
def test_decode_full_size_every_query():
    """16 queries x 5 drafts of the 3B-class drafter with ragged 4K-16K prefixes, in the
    launch configuration the benchmark times (the balanced plan over all SMs): every
    draft, head and output element against the oracle."""
    cfg = configs.DEC_3B_16Q
    _check(synth.decode_inputs(cfg))
