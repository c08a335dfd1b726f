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


@dataclass(frozen=True)
class RetrievalConfig:
    """Video-to-text retrieval (Section 3.1, Eq. 2-3): ``num_queries`` videos, each
    with a ragged number of keyframes drawn from ``keyframes_range``, against a
    corpus of ``num_texts`` CLIP text embeddings of ``dim``; each keyframe keeps
    its ``k_frame`` most similar texts and each query its ``k_query`` best texts
    of their union.  ``relevant`` texts per query are planted with similarity
    c ~ U(0.25, 0.5) to about half of the query's keyframes."""
    name: str
    num_queries: int
    keyframes_range: tuple          # (lo, hi) inclusive keyframes per query
    num_texts: int
    dim: int
    k_frame: int = 3
    k_query: int = 3                # Section 4.3: k = 3 documents per query
    relevant: int = 4
    seed: int = 20260102
    description: str = ""

    def with_(self, **kw) -> "RetrievalConfig":
        return replace(self, **kw)


RT_TINY = RetrievalConfig(
    name="retrieve-tiny", num_queries=3, keyframes_range=(1, 6), num_texts=2000, dim=512,
    description="3 queries x 1-6 keyframes against 2000 texts of dim 512")

RT_16Q_1M = RetrievalConfig(
    name="retrieve-16q-1m", num_queries=16, keyframes_range=(4, 32), num_texts=1 << 20, dim=768,
    description="16 queries x 4-32 keyframes against 1,048,576 CLIP ViT-L/14 text embeddings "
                "(dim 768, fp16)")

RT_16Q_256K = RT_16Q_1M.with_(
    name="retrieve-16q-256k", num_texts=1 << 18,
    description="16 queries x 4-32 keyframes against 262,144 text embeddings (dim 768, fp16; "
                "the profiling size)")

RETRIEVAL_PRESETS = {c.name: c for c in (RT_TINY, RT_16Q_1M, RT_16Q_256K)}


@dataclass(frozen=True)
class KeyframeConfig:
    """Keyframe extraction (Section 3.1, Eq. 1): ``num_videos`` RGB videos of
    ``height`` x ``width`` with a number of frames drawn from ``frames_range``;
    scenes last an exponential number of frames (mean ``scene_mean`` frames,
    at least 8), and a scene change is a fade of 8-15 frames with probability
    ``fade_prob`` (a hard cut otherwise)."""
    name: str
    num_videos: int
    frames_range: tuple             # (lo, hi) inclusive frames per video
    height: int
    width: int
    theta: float = 0.6              # keyframe threshold of Eq. 1
    scene_mean: float = 75.0        # 2.5 s at 30 frames/s
    fade_prob: float = 0.3
    seed: int = 20260103
    description: str = ""

    @property
    def npix(self) -> int:
        return self.height * self.width

    def with_(self, **kw) -> "KeyframeConfig":
        return replace(self, **kw)


KF_TINY = KeyframeConfig(
    name="keyframe-tiny", num_videos=3, frames_range=(5, 40), height=16, width=24, scene_mean=6.0,
    description="3 videos of 5-40 frames at 24x16")

KF_720P = KeyframeConfig(
    name="keyframe-8x720p", num_videos=8, frames_range=(500, 840), height=720, width=1280,
    description="8 videos of 500-840 frames (16.7-28 s at 30 frames/s, mean 22.3 s) at 1280x720 "
                "RGB uint8")

KF_720P_1V = KF_720P.with_(
    name="keyframe-1x720p", num_videos=1, frames_range=(300, 300),
    description="1 video of 300 frames at 1280x720 RGB uint8 (the profiling size)")

KEYFRAME_PRESETS = {c.name: c for c in (KF_TINY, KF_720P, KF_720P_1V)}


@dataclass(frozen=True)
class DecodeConfig:
    """One decode step of the drafter (Eq. 5, Eq. 8-10): ``num_queries`` queries,
    each with ``num_drafts`` drafts generated in parallel from one shared prefix
    (video tokens and question) of ``prefix_len`` tokens (or ragged in
    ``prefix_range``) and an own-token cache of ``cache_cap`` slots per draft, of
    which n_k ~ U[cache_range] are filled (retrieved text plus generated tokens)."""
    name: str
    num_queries: int
    num_drafts: int
    hq: int
    hkv: int
    head_dim: int
    prefix_len: int
    cache_cap: int
    cache_range: tuple              # (lo, hi) inclusive filled slots per draft
    prefix_range: tuple = None
    seed: int = 20260104
    description: str = ""

    def with_(self, **kw) -> "DecodeConfig":
        return replace(self, **kw)


DEC_TINY = DecodeConfig(
    name="decode-tiny", num_queries=2, num_drafts=3, hq=4, hkv=2, head_dim=64, prefix_len=0,
    prefix_range=(40, 300), cache_cap=150, cache_range=(1, 150),
    description="2 queries x 3 drafts, 4/2 heads of 64, ragged prefix 40-300, caches of 1-150 of 150")

DEC_3B_16Q = DecodeConfig(
    name="decode-3b-16q", num_queries=16, num_drafts=5, hq=16, hkv=2, head_dim=128, prefix_len=0,
    prefix_range=(4096, 16384), cache_cap=1024, cache_range=(256, 1024),
    description="3B-class drafter (Qwen2.5-VL-3B shapes: 16/2 heads of 128), 16 queries x 5 drafts, "
                "ragged shared prefix U[4096,16384], own caches of U[256,1024] of 1024 slots")

DECODE_PRESETS = {c.name: c for c in (DEC_TINY, DEC_3B_16Q)}
