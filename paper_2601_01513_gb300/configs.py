"""Named verifier workloads (shapes only; no arithmetic of the method).

Each preset describes one verify step of the speculative RAG verifier
(Section 3.1 "Speculate Generation", Eq. 6 and Eq. 11): ``num_queries`` questions,
each with a shared prefix (video tokens, question, retrieved passages) of
``prefix_len`` tokens, ``num_cand`` draft candidates of ``cand_len`` tokens,
an attention layer with ``hq`` query heads, ``hkv`` KV heads of ``head_dim``,
an LM head of ``hidden`` x ``vocab``, and the CLIP entity filter of
Eq. 14-15 over ``num_frames`` frames of ``clip_dim``-dimensional embeddings.
"""
from dataclasses import dataclass, replace


@dataclass(frozen=True)
class VerifyConfig:
    name: str
    num_queries: int
    hidden: int
    hq: int
    hkv: int
    head_dim: int
    prefix_len: int                 # fixed prefix length (ignored when prefix_range is set)
    num_cand: int
    cand_len: int
    vocab: int
    num_frames: int
    clip_dim: int
    threshold: float = 0.2          # CLIP keep threshold tau
    delta: float = 0.05             # reliability margin of Eq. 13 (Section 4.3: delta = 0.05)
    gathers: int = 1                # target ids gathered per row (1: likelihood, 2: Yes/No)
    prefix_range: tuple = None      # (lo, hi) inclusive: ragged prefix lengths drawn per query
    w_std: float = 0.02
    seed: int = 20260101
    clip_unit: bool = True          # embeddings unit-normalised before fp16 rounding
    description: str = ""

    @property
    def rows(self) -> int:
        """Candidate token rows M = Qn * K * L (one LM-head row per candidate token)."""
        return self.num_queries * self.num_cand * self.cand_len

    def with_(self, **kw) -> "VerifyConfig":
        return replace(self, **kw)


TINY = VerifyConfig(
    name="tiny", num_queries=1, hidden=512, hq=8, hkv=8, head_dim=64, prefix_len=256,
    num_cand=4, cand_len=8, vocab=4096, num_frames=16, clip_dim=512, clip_unit=False,
    description="tiny verify step: 1 query, H=512, 8/8 heads of 64, P=256, K=4 x L=8, V=4096, "
                "CLIP 4x16x512")

V7B = VerifyConfig(
    name="7b", num_queries=1, hidden=3584, hq=28, hkv=4, head_dim=128, prefix_len=8192,
    num_cand=5, cand_len=16, vocab=152064, num_frames=64, clip_dim=768,
    description="7B-class GQA verifier: 1 query, H=3584, 28/4 heads of 128, P=8192, K=5 x L=16, "
                "V=152064, CLIP 5x64x768")

LONG = VerifyConfig(
    name="long", num_queries=1, hidden=3584, hq=28, hkv=4, head_dim=128, prefix_len=32768,
    num_cand=8, cand_len=32, vocab=152064, num_frames=256, clip_dim=768,
    description="long-context verifier: 1 query, H=3584, 28/4 heads of 128, P=32768, K=8 x L=32, "
                "V=152064, CLIP 8x256x768")

BATCH16 = VerifyConfig(
    name="batch16", num_queries=16, hidden=3584, hq=28, hkv=4, head_dim=128, prefix_len=0,
    prefix_range=(4096, 16384), num_cand=5, cand_len=16, vocab=152064, num_frames=128,
    clip_dim=768,
    description="batched serving: 16 queries, H=3584, 28/4 heads of 128, ragged P~U[4096,16384], "
                "K=5 x L=16, V=152064, CLIP 16x5x128x768")

V72B = VerifyConfig(
    name="72b", num_queries=1, hidden=8192, hq=64, hkv=8, head_dim=128, prefix_len=16384,
    num_cand=10, cand_len=32, vocab=152064, num_frames=256, clip_dim=1024,
    description="72B-class verifier: 1 query, H=8192, 64/8 heads of 128, P=16384, K=10 x L=32, "
                "V=152064, CLIP 10x256x1024")

PRESETS = {c.name: c for c in (TINY, V7B, LONG, BATCH16, V72B)}
