"""logq_quantize_noalloc -- the entry point for callers that cannot allocate
device memory (it keeps its scratch in a static device array instead of a
caller workspace) -- must give exactly what logq_quantize gives.

Called through the C ABI with ctypes, twice in a row, so that the second call
runs on the scratch the first one left behind.  This file sorts last so that a
run that stops at the first failure has already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2607_01127_gb300 import workloads

from gpu_common import lib

pytestmark = pytest.mark.gpu

# (N, K, bits, base, range, flags): 4-bit and 3-bit with the automatic range,
# a given range with the floor shift, 8-bit codes (the 8-bit estimate kernel),
# and bases outside the quantiser's estimate guards (1.05 at 4 bits, 1.005 at
# 8 bits), which take the boundary-search kernels.
CASES = [(512, 2048, 4, 1.5, 0.0, 0), (33, 1152, 3, 1.25, 0.0, 0), (64, 2048, 4, 2.0, 0.05, 1),
         (300, 4096, 4, 1.7, 0.0, 0), (96, 1024, 8, 1.04, 0.0, 0), (64, 512, 4, 1.05, 0.0, 0),
         (40, 384, 8, 1.005, 0.0, 1)]


def _cb_fields(cb):
    return (cb.bits, cb.qmax, cb.flags, cb.base, cb.shift, cb.range, list(cb.level), list(cb.thresh),
            list(cb.level_bf16), list(cb.level_f16))


def test_noalloc_matches_allocating_entry_point_twice():
    logq = lib()
    L = logq.lib
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    for call in range(2):
        for i, (N, K, bits, base, rng, flags) in enumerate(CASES):
            w = workloads.weights_np(N, K, seed=100 + i, outliers=True)
            W = torch.from_numpy(w).cuda()
            ref_codes, ref_cb = logq.logq_quantize(W, bits, base, rng, flags)
            nbytes = logq.logq_packed_bytes(N, K, bits)
            out = torch.full((nbytes,), 0xAB, dtype=torch.uint8, device="cuda")
            cb = logq.Codebook()
            st = L.logq_quantize_noalloc(ctypes.c_void_p(W.data_ptr()), N, K, bits, base, rng, flags,
                                         ctypes.c_void_p(out.data_ptr()), ctypes.byref(cb), stream)
            assert st == logq.LOGQ_OK, logq.status_string(st)
            assert torch.equal(out, ref_codes), f"call {call} case {i}: codes differ"
            assert _cb_fields(cb) == _cb_fields(ref_cb)


def test_noalloc_reports_nonfinite_then_recovers():
    logq = lib()
    L = logq.lib
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    w = workloads.weights_np(16, 256, 7)
    w[5, 9] = np.nan
    W = torch.from_numpy(w).cuda()
    out = torch.empty(16 * 128, dtype=torch.uint8, device="cuda")
    cb = logq.Codebook()
    for rng in (0.0, 1.0):
        st = L.logq_quantize_noalloc(ctypes.c_void_p(W.data_ptr()), 16, 256, 4, 1.5, rng, 0,
                                     ctypes.c_void_p(out.data_ptr()), ctypes.byref(cb), stream)
        assert st == logq.LOGQ_ERR_NONFINITE
    # the flag left in the static scratch is cleared by the next call
    W2 = torch.from_numpy(np.nan_to_num(w)).cuda()
    ref, _ = logq.logq_quantize(W2, 4, 1.5)
    st = L.logq_quantize_noalloc(ctypes.c_void_p(W2.data_ptr()), 16, 256, 4, 1.5, 0.0, 0,
                                 ctypes.c_void_p(out.data_ptr()), ctypes.byref(cb), stream)
    assert st == logq.LOGQ_OK and torch.equal(out, ref)
