"""Shared helpers of the GPU parity tests: device placement of seeded inputs, guarded
output buffers (sentinel regions before and after every output, checked after each
call) and the comparison rules (tolerances and margin rules for integer decisions)."""
import numpy as np
import torch

from paper_2601_01513_gb300 import build, fvrag

ATTN_ATOL = 2e-2        # attention output, max-abs (bf16 output vs fp64)
ATTN_LSE_ATOL = 2e-3    # attention log-sum-exp (fp32 scores, fp32 sums)
LOGPROB_ATOL = 1e-2     # per-token log-prob
COS_ATOL = 1e-3         # cosine / max_cos


GUARD_BYTES = 4096      # sentinel bytes before and after every output buffer


class Guarded:
    """An output tensor placed between two guard regions of sentinel bytes.  Writes past
    either end of the output (which NaN-poisoning of the output itself cannot reveal)
    change a guard; ``check`` asserts both are intact.  The output starts 4096 bytes into
    its allocation, so it keeps the allocation's alignment."""

    def __init__(self, shape, dtype, fill):
        esz = torch.empty((), dtype=dtype).element_size()
        n = int(np.prod(shape)) * esz
        self.n = n
        self.buf = torch.empty(GUARD_BYTES * 2 + n, dtype=torch.uint8, device="cuda")
        pat = (torch.arange(GUARD_BYTES, dtype=torch.int32, device="cuda") * 37 + 11) % 251
        self.pat = pat.to(torch.uint8)
        self.buf[:GUARD_BYTES].copy_(self.pat)
        self.buf[GUARD_BYTES + n:].copy_(self.pat)
        self.t = self.buf[GUARD_BYTES:GUARD_BYTES + n].view(dtype).view(shape)
        if n:
            self.t.fill_(fill)

    def check(self, what=""):
        torch.cuda.synchronize()
        lo = self.buf[:GUARD_BYTES]
        hi = self.buf[GUARD_BYTES + self.n:]
        assert torch.equal(lo, self.pat), "write before the start of output %s" % what
        assert torch.equal(hi, self.pat), "write past the end of output %s" % what


def guarded(shape, dtype, fill, pool):
    """A guarded output tensor; its guard object is appended to `pool` for ``check_all``."""
    g = Guarded(shape, dtype, fill)
    pool.append(g)
    return g.t


def check_all(pool):
    for i, g in enumerate(pool):
        g.check("#%d" % i)


def ensure_built():
    build.build_all()
    return fvrag.lib()


def dev_bf16(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()


def dev_f16(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.float16).cuda()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_attn(q, kp, vp, offs, kt, vt, with_lse=True, scale=0.0, sm_budget=0, split=0):
    """Runs fvrag_verify_attn on numpy inputs; returns (out fp32 numpy, lse numpy, status).
    split: the key-split plan requested in the descriptor's flags (0: the library's choice)."""
    Qn, K, L, Hq, D = q.shape
    tq, tkt, tvt = dev_bf16(q), dev_bf16(kt), dev_bf16(vt)
    tkp = dev_bf16(kp) if kp.shape[0] > 0 else None
    tvp = dev_bf16(vp) if vp.shape[0] > 0 else None
    toffs = dev(offs.astype(np.int32))
    maxp = int(np.max(np.diff(offs))) if len(offs) > 1 else 0
    d = fvrag.AttnDesc(Qn, K, L, Hq, kt.shape[3], D, maxp, int(kp.shape[0]), float(scale), split,
                       sm_budget)
    ws = torch.zeros(fvrag.attn_workspace_bytes(d), dtype=torch.uint8, device="cuda")
    pool = []
    out = guarded(q.shape, torch.bfloat16, float("nan"), pool)
    lse = guarded(q.shape[:-1], torch.float32, float("nan"), pool) if with_lse else None
    fvrag.verify_attn(tq, tkp, tvp, toffs, tkt, tvt, out, ws, maxp, lse=lse, softmax_scale=scale,
                      sm_budget=sm_budget, split=split)
    st = fvrag.read_status(ws)
    check_all(pool)
    return out.float().cpu().numpy(), (lse.cpu().numpy() if with_lse else None), st


def run_lm(hidden, weight, targets, sm_budget=0):
    th, tw, tt = dev_bf16(hidden), dev_bf16(weight), dev(targets.astype(np.int32))
    M = hidden.shape[0]
    G = targets.shape[1]
    d = fvrag.LmDesc(M, hidden.shape[1], weight.shape[0], G, 0)
    ws = torch.zeros(fvrag.lm_workspace_bytes(d), dtype=torch.uint8, device="cuda")
    pool = []
    lp = guarded((M, G), torch.float32, float("nan"), pool)
    lse = guarded((M,), torch.float32, float("nan"), pool)
    fvrag.score_logprobs(th, tw, tt, lp, ws, lse=lse, sm_budget=sm_budget)
    st = fvrag.read_status(ws)
    check_all(pool)
    return lp.cpu().numpy(), lse.cpu().numpy(), st


def run_clip(cand, frames, tau, with_cos=True):
    Qn, K, E = cand.shape
    F = frames.shape[1]
    tc, tf = dev_f16(cand), dev_f16(frames)
    pool = []
    mc = guarded((Qn, K), torch.float32, float("nan"), pool)
    am = guarded((Qn, K), torch.int32, -7, pool)
    keep = guarded((Qn, K), torch.uint8, 9, pool)
    cos = guarded((Qn, K, F), torch.float32, float("nan"), pool) if with_cos else None
    fvrag.clip_align(tc, tf, tau, mc, am, keep, cos=cos)
    check_all(pool)
    return ((cos.cpu().numpy() if with_cos else None), mc.cpu().numpy(), am.cpu().numpy(),
            keep.cpu().numpy())


def run_select(lp, mode, keep=None, max_cos=None, lengths=None, delta=0.05, seed=0):
    Qn, K, L, G = lp.shape
    pool = []
    score = guarded((Qn, K), torch.float32, float("nan"), pool)
    sel = guarded((Qn,), torch.int32, -7, pool)
    fvrag.select_candidate(dev(lp.astype(np.float32)), score, sel, mode=mode,
                           keep=None if keep is None else dev(keep.astype(np.uint8)),
                           max_cos=None if max_cos is None else dev(max_cos.astype(np.float32)),
                           lengths=None if lengths is None else dev(lengths.astype(np.int32)),
                           delta=delta, seed=seed)
    check_all(pool)
    return score.cpu().numpy(), sel.cpu().numpy()


def check_argmax_with_margin(gpu_idx, oracle_cos, tol=COS_ATOL):
    """GPU frame index must attain the oracle max within tol (unique when the margin is larger)."""
    Qn, K, F = oracle_cos.shape
    for q in range(Qn):
        for k in range(K):
            row = oracle_cos[q, k]
            j = int(gpu_idx[q, k])
            assert 0 <= j < F
            assert row[j] >= row.max() - tol, (q, k, j, row[j], row.max())
            srt = np.sort(row)
            if F > 1 and srt[-1] - srt[-2] > tol:
                assert j == int(np.argmax(row))


def check_keep_with_margin(gpu_keep, oracle_maxcos, tau, tol=COS_ATOL):
    exp = (oracle_maxcos >= tau).astype(np.uint8)
    ambiguous = np.abs(oracle_maxcos - tau) < tol
    assert np.all((gpu_keep == exp) | ambiguous)
    assert np.all((gpu_keep == 0) | (gpu_keep == 1))


def check_selection_masked(gpu_sel, oracle_score, oracle_maxcos, tau, tol_score=2 * LOGPROB_ATOL,
                           tol_cos=COS_ATOL):
    """The GPU pick must be a valid answer under some resolution of the ambiguous keeps, and
    within the score tolerance of the best valid candidate."""
    Qn, K = oracle_score.shape
    for q in range(Qn):
        sure = oracle_maxcos[q] >= tau + tol_cos
        maybe = oracle_maxcos[q] > tau - tol_cos
        s = int(gpu_sel[q])
        if s < 0:
            assert not sure.any()
            continue
        assert maybe[s]
        best_sure = oracle_score[q][sure].max() if sure.any() else -np.inf
        assert oracle_score[q, s] >= best_sure - tol_score


def run_keyframes(pixels, video_offsets, theta, with_hist=True):
    """fvrag_keyframes on numpy inputs; returns (hist, sim, is_key, key_index, key_offsets, status)."""
    T = pixels.shape[0]
    Nv = len(video_offsets) - 1
    px = torch.from_numpy(np.ascontiguousarray(pixels)).cuda() if T > 0 else \
        torch.empty((0,) + tuple(pixels.shape[1:]), dtype=torch.uint8, device="cuda")
    vo = dev(np.asarray(video_offsets, np.int32))
    d = fvrag.keyframe_desc(Nv, px, theta)
    ws = torch.zeros(fvrag.keyframes_workspace_bytes(d), dtype=torch.uint8, device="cuda")
    pool = []
    hist = guarded((T, 512), torch.int32, -7, pool) if with_hist else None
    sim = guarded((max(T, 1),), torch.float32, float("nan"), pool)
    key = guarded((max(T, 1),), torch.uint8, 9, pool)
    kidx = guarded((max(T, 1),), torch.int32, -7, pool)
    koffs = guarded((Nv + 1,), torch.int32, -7, pool)
    fvrag.keyframes(px, vo, theta, sim, key, kidx, koffs, ws, hist=hist)
    st = fvrag.read_status(ws)
    check_all(pool)
    ko = koffs.cpu().numpy()
    return ((hist.cpu().numpy() if with_hist else None), sim.cpu().numpy()[:T], key.cpu().numpy()[:T],
            kidx.cpu().numpy()[:ko[-1]], ko, st)


def run_retrieve(frames, frame_offsets, texts, k_frame, k_query, precompute_norms=True):
    """fvrag_retrieve on numpy inputs; returns (frame_idx, frame_sim, idx, sim, status)."""
    Fr = frames.shape[0]
    Qn = len(frame_offsets) - 1
    tf = dev_f16(frames) if Fr > 0 else torch.empty((0, texts.shape[1]), dtype=torch.float16, device="cuda")
    tt = dev_f16(texts)
    fo = dev(np.asarray(frame_offsets, np.int32))
    inv = None
    if precompute_norms:
        npool = []
        inv = guarded((texts.shape[0],), torch.float32, float("nan"), npool)
        fvrag.embed_inv_norms(tt, inv)
        check_all(npool)
    d = fvrag.retrieve_desc(Qn, tf, tt, k_frame, k_query)
    ws = torch.zeros(fvrag.retrieve_workspace_bytes(d), dtype=torch.uint8, device="cuda")
    pool = []
    fi = guarded((max(Fr, 1), k_frame), torch.int32, -7, pool)
    fs = guarded((max(Fr, 1), k_frame), torch.float32, float("nan"), pool)
    oi = guarded((Qn, k_query), torch.int32, -7, pool)
    os_ = guarded((Qn, k_query), torch.float32, float("nan"), pool)
    fvrag.retrieve(tf, fo, tt, k_frame, oi, os_, ws, text_inv_norm=inv, frame_topk=fi,
                   frame_topk_sim=fs)
    st = fvrag.read_status(ws)
    check_all(pool)
    return (fi.cpu().numpy()[:Fr], fs.cpu().numpy()[:Fr], oi.cpu().numpy(), os_.cpu().numpy(), st)


def check_frame_lists(gpu_idx, gpu_sim, texts, frames, oracle_frame_topk_all, tol=COS_ATOL):
    """Per-keyframe lists: each GPU entry is a real similarity of that text (within tol), the
    list is sorted, ids are unique, and it agrees with the oracle's full ordering: the j-th
    GPU similarity is within tol of the oracle's j-th, every text whose oracle similarity
    beats the oracle's k-th by more than tol is present, and ids match exactly wherever the
    oracle's neighbours are more than tol apart.  ``oracle_frame_topk_all(f)`` returns the
    oracle's (ids, sims) of keyframe f over the whole corpus, best first."""
    Fr, kf = gpu_idx.shape
    for f in range(Fr):
        oi, osim = oracle_frame_topk_all(f)
        n = min(kf, len(oi))
        gi, gs = gpu_idx[f], gpu_sim[f]
        assert np.all(gi[n:] == -1) and np.all(np.isneginf(gs[n:]))
        gi, gs = gi[:n], gs[:n]
        assert len(set(gi.tolist())) == n and np.all(gi >= 0)
        assert np.all(np.diff(gs) <= 0)
        sim_of = dict(zip(oi.tolist(), osim.tolist()))
        for j in range(n):
            assert abs(gs[j] - osim[j]) <= tol, (f, j, gs[j], osim[j])
            if int(gi[j]) in sim_of:
                assert abs(gs[j] - sim_of[int(gi[j])]) <= tol
        kth = osim[n - 1]
        sure = oi[osim > kth + tol]
        assert set(sure.tolist()) <= set(gi.tolist())
        for j in range(n):
            lo = osim[j - 1] - osim[j] if j > 0 else np.inf
            hi = osim[j] - osim[j + 1] if j + 1 < len(osim) else np.inf
            if lo > tol and hi > tol:
                assert gi[j] == oi[j], (f, j, gi[j], oi[j])


def run_decode(q, kp, vp, offs, kc, vc, n, with_lse=True, scale=0.0):
    """fvrag_decode_attn on numpy inputs; returns (out fp32 numpy, lse numpy, status)."""
    tq, tkc, tvc = dev_bf16(q), dev_bf16(kc), dev_bf16(vc)
    tkp = dev_bf16(kp) if kp.shape[0] > 0 else None
    tvp = dev_bf16(vp) if vp.shape[0] > 0 else None
    toffs = dev(np.asarray(offs, np.int32))
    tn = dev(np.asarray(n, np.int32))
    maxp = int(np.max(np.diff(offs))) if len(offs) > 1 else 0
    d = fvrag.decode_desc(tq, tkp, tkc, maxp, scale)
    ws = torch.zeros(fvrag.decode_workspace_bytes(d), dtype=torch.uint8, device="cuda")
    pool = []
    out = guarded(q.shape, torch.bfloat16, float("nan"), pool)
    lse = guarded(q.shape[:-1], torch.float32, float("nan"), pool) if with_lse else None
    fvrag.decode_attn(tq, tkp, tvp, toffs, tkc, tvc, tn, out, ws, maxp, lse=lse, softmax_scale=scale)
    st = fvrag.read_status(ws)
    check_all(pool)
    return out.float().cpu().numpy(), (lse.cpu().numpy() if with_lse else None), st
