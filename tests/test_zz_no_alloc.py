"""The allocation-free LM-head entry point (fvrag_score_logprobs_noalloc).

It serves callers that cannot call cudaMalloc (their device memory belongs to
another allocator, or they may not allocate once running): the scratch lives in
a static device array inside the library instead of a caller workspace.  This
test calls it through the C ABI on consecutive calls of every kernel form the LM
head has -- the largest shape first (1024 rows x 8 gathers fills the array), then
smaller ones, so contents an earlier call left in the shared array must not leak
into a later one -- and checks each against the workspace entry point and against
the oracle, and reads the array's status word after each call.  Shapes beyond the
array's limit are refused.  It lives in its own file so that it runs after every
other test, and it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2601_01513_gb300 import fvrag, synth

from gpu_helpers import LOGPROB_ATOL, dev, dev_bf16, ensure_built

pytestmark = pytest.mark.gpu

# rows, hidden, vocabulary, gathers: the kernel form each selects
CASES = [
    (1024, 256, 9001, 8),    # eight M-tiles: 2-SM pair form, two pair tiles per pass; the array's limit
    (300, 512, 20011, 2),    # three M-tiles: the vocabulary-major 2-SM pair form
    (200, 128, 7001, 3),     # two M-tiles: 2-SM pair form, one pair tile
    (37, 256, 4099, 1),      # one M-tile: <256, 1>
]


def _case(M, H, V, G, seed):
    hid = synth.normal_bf16((M, H), seed, 1)
    W = synth.normal_bf16((V, H), seed, 2, 0.0, 0.05)
    tgt = synth.uniform_i32((M, G), seed, 3, 0, V)
    tgt[0, 0] = -1                       # an out-of-range id: NaN on every path
    return hid, W, tgt


def _close(a, b):
    assert np.array_equal(np.isnan(a), np.isnan(b))
    ok = ~np.isnan(b)
    assert np.max(np.abs(a[ok] - b[ok])) <= LOGPROB_ATOL


def test_noalloc_matches_workspace_entry_point_and_oracle():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    L = ensure_built()
    stream = torch.cuda.current_stream()
    for call, (M, H, V, G) in enumerate(CASES):
        hid, W, tgt = _case(M, H, V, G, seed=4242 + call)
        th, tw, tt = dev_bf16(hid), dev_bf16(W), dev(tgt)
        d = fvrag.LmDesc(M, H, V, G, 0)
        ws = torch.zeros(fvrag.lm_workspace_bytes(d), dtype=torch.uint8, device="cuda")
        ref_lp = torch.empty((M, G), dtype=torch.float32, device="cuda")
        ref_lse = torch.empty((M,), dtype=torch.float32, device="cuda")
        fvrag.score_logprobs(th, tw, tt, ref_lp, ws, lse=ref_lse)
        assert fvrag.read_status(ws) == fvrag.OK

        lp = torch.full((M, G), 7.0, dtype=torch.float32, device="cuda")
        lse = torch.full((M,), 7.0, dtype=torch.float32, device="cuda")
        st = L.fvrag_score_logprobs_noalloc(
            ctypes.byref(d), ctypes.c_void_p(th.data_ptr()), ctypes.c_void_p(tw.data_ptr()),
            ctypes.c_void_p(tt.data_ptr()), ctypes.c_void_p(lp.data_ptr()),
            ctypes.c_void_p(lse.data_ptr()), ctypes.c_void_p(stream.cuda_stream))
        assert st == fvrag.OK, fvrag.status_string(st)
        # the device-side status of this call, from the static array's status word
        assert L.fvrag_score_logprobs_noalloc_status(ctypes.c_void_p(stream.cuda_stream)) == fvrag.OK
        a, a_lse = lp.cpu().numpy(), lse.cpu().numpy()
        assert np.isnan(a[0, 0])
        _close(a, ref_lp.cpu().numpy())                       # the workspace entry point
        assert np.max(np.abs(a_lse - ref_lse.cpu().numpy())) <= LOGPROB_ATOL
        o_lp, o_lse = oracle.score_logprobs(hid, W, tgt)       # the oracle
        _close(a, o_lp)
        assert np.max(np.abs(a_lse - o_lse)) <= LOGPROB_ATOL

    # beyond the static array's limit (1024 rows): refused, nothing enqueued
    big = fvrag.LmDesc(1025, 512, 20011, 1, 0)
    st = L.fvrag_score_logprobs_noalloc(ctypes.byref(big), ctypes.c_void_p(th.data_ptr()),
                                        ctypes.c_void_p(tw.data_ptr()), ctypes.c_void_p(tt.data_ptr()),
                                        ctypes.c_void_p(lp.data_ptr()), None, None)
    assert st == fvrag.ERR_UNSUPPORTED
