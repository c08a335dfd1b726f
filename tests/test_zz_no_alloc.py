"""The allocation-free LM-head entry point (fvrag_score_logprobs_noalloc).

It serves callers that cannot call cudaMalloc (their device memory belongs to
another allocator, or they may not allocate once running): the scratch lives in
a static device array inside the library instead of a caller workspace.  This
test calls it through the C ABI and checks it against the workspace entry point
on two calls in a row (the second smaller than the first, so contents the first
call left in the shared array must not leak into the second), and checks that
shapes beyond the array's limit are refused.  It lives in its own file so that
it runs after every other test, and it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2601_01513_gb300 import fvrag, synth

from gpu_helpers import LOGPROB_ATOL, dev, dev_bf16, ensure_built

pytestmark = pytest.mark.gpu


def _case(M, H, V, G, seed):
    hid = synth.normal_bf16((M, H), seed, 1)
    W = synth.normal_bf16((V, H), seed, 2, 0.0, 0.05)
    tgt = synth.uniform_i32((M, G), seed, 3, 0, V)
    tgt[0, 0] = -1                       # an out-of-range id: NaN on both paths
    return dev_bf16(hid), dev_bf16(W), dev(tgt)


def test_noalloc_matches_workspace_entry_point():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    L = ensure_built()
    for call, (M, H, V, G) in enumerate([(300, 512, 20011, 2), (37, 256, 4099, 1)]):
        th, tw, tt = _case(M, H, V, G, seed=4242 + call)
        d = fvrag.LmDesc(M, H, V, G, 0)
        ws = torch.zeros(fvrag.lm_workspace_bytes(d), dtype=torch.uint8, device="cuda")
        ref_lp = torch.empty((M, G), dtype=torch.float32, device="cuda")
        ref_lse = torch.empty((M,), dtype=torch.float32, device="cuda")
        fvrag.score_logprobs(th, tw, tt, ref_lp, ws, lse=ref_lse)

        lp = torch.full((M, G), 7.0, dtype=torch.float32, device="cuda")
        lse = torch.full((M,), 7.0, dtype=torch.float32, device="cuda")
        stream = torch.cuda.current_stream()
        st = L.fvrag_score_logprobs_noalloc(
            ctypes.byref(d), ctypes.c_void_p(th.data_ptr()), ctypes.c_void_p(tw.data_ptr()),
            ctypes.c_void_p(tt.data_ptr()), ctypes.c_void_p(lp.data_ptr()),
            ctypes.c_void_p(lse.data_ptr()), ctypes.c_void_p(stream.cuda_stream))
        assert st == fvrag.OK, fvrag.status_string(st)
        torch.cuda.synchronize()
        a, b = lp.cpu().numpy(), ref_lp.cpu().numpy()
        assert np.array_equal(np.isnan(a), np.isnan(b)) and np.isnan(a[0, 0])
        ok = ~np.isnan(b)
        assert np.max(np.abs(a[ok] - b[ok])) <= LOGPROB_ATOL
        assert np.max(np.abs(lse.cpu().numpy() - ref_lse.cpu().numpy())) <= LOGPROB_ATOL

    # beyond the static array's limit (1024 rows): refused, nothing enqueued
    big = fvrag.LmDesc(1025, 512, 20011, 1, 0)
    st = L.fvrag_score_logprobs_noalloc(ctypes.byref(big), ctypes.c_void_p(th.data_ptr()),
                                        ctypes.c_void_p(tw.data_ptr()), ctypes.c_void_p(tt.data_ptr()),
                                        ctypes.c_void_p(lp.data_ptr()), None, None)
    assert st == fvrag.ERR_UNSUPPORTED
