"""Host logic of the side-by-side verify step: which workloads run the attention beside
the LM head, and with which SM budgets (no GPU needed)."""
from paper_2601_01513_gb300 import configs
from paper_2601_01513_gb300.pipeline import attn_row_tiles, plan_sm_split


def test_row_tiles():
    # 7b: 5 x 16 tokens x 7 query heads per KV head -> 18 tokens per 128-row tile, 5 tiles
    assert attn_row_tiles(configs.V7B) == 4 * 5
    assert attn_row_tiles(configs.TINY) == 8          # one query head per KV head: 32 rows
    assert attn_row_tiles(configs.BATCH16) == 16 * 4 * 5


def test_split_only_where_the_lm_head_streams_hbm():
    # one M-tile of rows (HBM-bound LM head) and an attention that fits in its shadow
    assert plan_sm_split(configs.V7B, 152) == (20, 132)
    assert plan_sm_split(configs.TINY, 152) == (8, 144)
    # more than 128 rows: the LM head is on the tensor cores too -> one after the other
    for name in ("long", "batch16", "72b"):
        assert plan_sm_split(configs.PRESETS[name], 152) is None
    # end to end from host buffers the attention starts late: two CTAs per row tile
    assert plan_sm_split(configs.V7B, 152, late=True) == (40, 112)
    assert plan_sm_split(configs.TINY, 152, late=True) == (16, 136)
    assert plan_sm_split(configs.LONG, 152, late=True) is None
    # the budgets always add up to the device
    for sms in (148, 132, 160):
        a, b = plan_sm_split(configs.V7B, sms)
        assert a + b == sms and a == 20


def test_no_split_when_attention_outlasts_the_lm_head():
    import dataclasses
    long_prefix = dataclasses.replace(configs.V7B, prefix_len=131072)
    assert plan_sm_split(long_prefix, 152) is None
    # too few SMs to give the attention a quarter of them
    assert plan_sm_split(configs.V7B, 40) is None
