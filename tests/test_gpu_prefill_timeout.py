"""The prefill kernel's bounded waits, made to run out on purpose.

Every mbarrier wait of the tensor-core prefill GEMM gives up after about one
second of clock cycles: it records LOGQ_ERR_TIMEOUT in the caller's workspace,
raises the CTA's abort flag, every role leaves its loop, the kernel waits for
the copies and multiply-adds it issued, frees its tensor memory and returns.
That path never runs in a correct launch, so this test builds the library once
more with a test-only hook (-DLOGQ_TEST_WAIT_HOOK; the shipped library has no
such code): when the workspace holds the trigger word, the MMA warp first waits
on a barrier that nothing completes.  The test checks that the call reports the
timeout (and a role's wait code), that the context stays usable, and that a
normal call right after it on the same library is correct.  No fault, trap or
unbounded wait is involved: the stalled wait ends by its own bound.
"""
import ctypes
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import check_linear, lib

pytestmark = pytest.mark.gpu

STALL_WORD = 0x57A11      # kTestStallWord in csrc/prefill.cu
# detail codes of the roles' waits (producer, MMA, epilogue, decode): the MMA
# warp stalls, and whichever role's one-second bound runs out first records it
ROLE_WAITS = (1, 2, 3, 4)


@pytest.fixture(scope="module")
def hooked(tmp_path_factory):
    from paper_2607_01127_gb300 import build
    out = str(tmp_path_factory.mktemp("hook") / "liblogq_hook.so")
    build.build_library(extra=("-DLOGQ_TEST_WAIT_HOOK",), out=out)
    L = ctypes.CDLL(out)
    P = ctypes.c_void_p
    logq = lib()
    L.logq_linear.argtypes = [P, ctypes.POINTER(logq.Codebook), P, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                              ctypes.c_int64, P, ctypes.c_int, P, ctypes.c_size_t, P]
    L.logq_linear.restype = ctypes.c_int
    L.logq_workspace_status.argtypes = [P, P, ctypes.POINTER(ctypes.c_uint32)]
    L.logq_workspace_status.restype = ctypes.c_int
    return logq, L


def test_prefill_wait_bound_reports_timeout_and_recovers(hooked):
    logq, L = hooked
    N, K, B = 300, 1024, 96
    w = workloads.weights_np(N, K, 31, outliers=True)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 4, 1.5)
    ocb = oracle.build_codebook(4, 1.5, cb.range)
    X = workloads.activations_torch(B, K, 31, torch.bfloat16, "cuda")
    Y = torch.empty(B, N, dtype=torch.float32, device="cuda")
    ws = logq.new_workspace()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)

    def call():
        return L.logq_linear(ctypes.c_void_p(codes.data_ptr()), ctypes.byref(cb), ctypes.c_void_p(X.data_ptr()),
                             logq.LOGQ_BF16, B, N, K, ctypes.c_void_p(Y.data_ptr()), logq.LOGQ_F32,
                             ctypes.c_void_p(ws.data_ptr()), ws.numel(), stream)

    ws.view(torch.int32)[4] = STALL_WORD                  # reserved[0]
    assert call() == logq.LOGQ_OK                         # the launch itself succeeds
    detail = ctypes.c_uint32(0)
    st = L.logq_workspace_status(ctypes.c_void_p(ws.data_ptr()), stream, ctypes.byref(detail))
    assert st == logq.LOGQ_ERR_TIMEOUT and detail.value in ROLE_WAITS, (st, detail.value)
    torch.cuda.synchronize()                              # the context is still usable

    ws.view(torch.int32)[4] = 0
    Y.fill_(float("nan"))
    assert call() == logq.LOGQ_OK
    st = L.logq_workspace_status(ctypes.c_void_p(ws.data_ptr()), stream, ctypes.byref(detail))
    assert st == logq.LOGQ_OK
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, 4)
    Yr, A = oracle.linear(X.float().cpu().double().numpy(), oracle.dequant(q, ocb, oracle.TABLE_BF16))
    check_linear(Y.double().cpu().numpy(), Yr, A)
