"""The benchmark's roofline numerators on CPU: the algorithmic bytes and flops that
bench.py divides by the measured time are checked against independent counts -- the
visible (row, head, key) triples enumerated one by one, the tensor sizes added up from
the shapes -- so that a fraction of peak can only be as large as the work really done."""
import numpy as np
import pytest

import bench
from paper_2601_01513_gb300 import configs, synth


def _visible_keys(cfg):
    """(query token, head, key) triples the attention scores: every prefix key of the
    query, and the candidate's own tokens 0 .. l for its token l (enumerated)."""
    plen = synth.prefix_lengths(cfg)
    n = 0
    for q in range(cfg.num_queries):
        for _k in range(cfg.num_cand):
            for l in range(cfg.cand_len):
                n += int(plen[q]) + (l + 1)
    return n * cfg.hq


@pytest.mark.parametrize("name", ["tiny", "7b", "long", "batch16", "72b"])
def test_attention_flops_count_every_visible_key(name):
    cfg = configs.PRESETS[name]
    _, flops = bench.algorithmic(cfg)["attn"]
    # one multiply-add per element for q.k and one for p.v: 4 D flops per visible triple
    assert flops == 4.0 * cfg.head_dim * _visible_keys(cfg)


@pytest.mark.parametrize("name", ["tiny", "7b", "long", "batch16", "72b"])
def test_bytes_are_the_tensors_read_and_written_once(name):
    cfg = configs.PRESETS[name]
    a = bench.algorithmic(cfg)
    Qn, K, L, hq, hkv, D = cfg.num_queries, cfg.num_cand, cfg.cand_len, cfg.hq, cfg.hkv, cfg.head_dim
    P = int(synth.prefix_lengths(cfg).sum())
    bf16 = 2
    q = out = Qn * K * L * hq * D * bf16
    prefix_kv = 2 * P * hkv * D * bf16
    tail_kv = 2 * Qn * K * L * hkv * D * bf16
    lse = Qn * K * L * hq * 4
    assert a["attn"][0] == prefix_kv + q + out + tail_kv + lse
    M, H, V, G = cfg.rows, cfg.hidden, cfg.vocab, cfg.gathers
    weight, hidden = V * H * bf16, M * H * bf16
    targets = logprob = M * G * 4
    assert a["lm"][0] == weight + hidden + targets + logprob + M * 4
    assert a["lm"][1] == 2.0 * M * H * V
    E, F = cfg.clip_dim, cfg.num_frames
    assert a["clip"][0] == Qn * (K + F) * E * 2 + Qn * K * (4 + 4 + 1)


def test_7b_figures():
    """The 7B-class workload's work, as quoted in the design notes."""
    a = bench.algorithmic(configs.V7B)
    assert a["attn"][0] / 1e6 == pytest.approx(18.1, abs=0.05)
    assert a["attn"][1] / 1e9 == pytest.approx(9.40, abs=0.01)
    assert a["lm"][0] / 1e9 == pytest.approx(1.0906, abs=0.0005)
    assert a["lm"][1] / 1e9 == pytest.approx(87.2, abs=0.05)
    # the LM head is below the ~278 flop/B ridge of the measured peaks: HBM binds
    assert a["lm"][1] / a["lm"][0] < 100
    # and the attention above it: the tensor cores bind
    assert a["attn"][1] / a["attn"][0] > 278
