"""8-bit Log_b codes (Sec. 3.1 with n = 8: q_max = 127, one code per byte)
against the oracle: packed codes bit-exact (elements within one fp32 ulp of a
boundary counted), decode GEMV and prefill GEMM outputs within
1e-3 * sum_k |x_k w_k| + 1e-6, and the self-calibrating range with the
paper's 8-bit eps."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import check_codes, check_linear, lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def logq():
    return lib()


def reference(X, q, ocb):
    table = oracle.TABLE_BF16 if X.dtype == torch.bfloat16 else oracle.TABLE_F16
    return oracle.linear(X.float().cpu().double().numpy(), oracle.dequant(q, ocb, table), nthreads=0)


@pytest.mark.parametrize("N,K", [(512, 2048), (1, 128), (7, 384), (300, 4096)])
@pytest.mark.parametrize("base", [1.02, 1.05, 1.1])
def test_quantize8_auto_range_bit_exact(logq, N, K, base):
    w = workloads.weights_np(N, K, seed=N + K, outliers=(N * K >= 100000))
    W = torch.from_numpy(w).cuda()
    codes, cb = logq.logq_quantize(W, 8, base)
    rng_ = float(np.abs(w).max())
    assert cb.bits == 8 and cb.qmax == 127 and cb.range == rng_
    ocb = oracle.build_codebook(8, base, rng_)
    np.testing.assert_array_equal(np.array(cb.thresh[:127], np.float32), ocb.taus32_up)
    assert codes.numel() == N * K
    assert check_codes(codes.cpu().numpy(), w, ocb, 8) <= 2


@pytest.mark.parametrize("mode", [0, 1])
def test_quantize8_given_range_and_special_values(logq, mode):
    w = workloads.weights_np(64, 1024, seed=3, outliers=True)
    w[0, :6] = [0.0, -0.0, 1e-30, -1e-30, 50.0, -50.0]          # zeros, pruned, clamped from above
    rng_ = 0.5 * float(np.abs(w[1:]).max())
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.05, rng_, mode)
    ocb = oracle.build_codebook(8, 1.05, rng_, mode)
    check_codes(codes.cpu().numpy(), w, ocb, 8)
    c = codes.view(64, 1024).cpu().numpy()
    np.testing.assert_array_equal(c[0, :6], [0, 0, 0, 0, 127, 255])


@pytest.mark.parametrize("N,K", [(512, 2048), (7, 128), (300, 1152), (1000, 4096), (129, 14336), (2049, 384)])
@pytest.mark.parametrize("B", [1, 2, 3, 4])
def test_gemv8_bf16(logq, N, K, B):
    w = workloads.weights_np(N, K, seed=N + 2 * K + B)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.04)
    ocb = oracle.build_codebook(8, 1.04, cb.range)
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, 8)
    X = workloads.activations_torch(B, K, N + B, torch.bfloat16, "cuda")
    Y = logq.logq_linear(codes, cb, X, N, K)
    Yr, A = reference(X, q, ocb)
    check_linear(Y.double().cpu().numpy(), Yr, A)


@pytest.mark.parametrize("B", [1, 4])
@pytest.mark.parametrize("xdt,ydt", [(torch.float16, None), (torch.bfloat16, torch.bfloat16),
                                     (torch.float16, torch.float16)])
def test_gemv8_dtypes(logq, B, xdt, ydt):
    N, K = 640, 2048
    w = workloads.weights_np(N, K, seed=17)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.06)
    ocb = oracle.build_codebook(8, 1.06, cb.range)
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, 8)
    X = workloads.activations_torch(B, K, 5, xdt, "cuda")
    Y = logq.logq_linear(codes, cb, X, N, K, y_dtype=ydt)
    Yr, A = reference(X, q, ocb)
    name = {None: "f32", torch.bfloat16: "bf16", torch.float16: "f16"}[ydt]
    check_linear(Y.double().cpu().numpy(), Yr, A, name)


def test_gemv8_large_launch_and_grouped(logq):
    """A launch above the 20 MiB split (one 16-warp CTA per SM) and a grouped
    launch of two 8-bit matrices equal to the single calls."""
    N, K = 10247, 2048
    w = workloads.weights_np(N, K, seed=23)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.05)
    ocb = oracle.build_codebook(8, 1.05, cb.range)
    X = workloads.activations_torch(1, K, 24, torch.bfloat16, "cuda")
    Y = logq.logq_linear(codes, cb, X, N, K).double().cpu().numpy()
    rows = np.random.default_rng(1).choice(N, 256, replace=False)
    q = oracle.unpack(codes.view(N, K).cpu().numpy()[rows], len(rows), K, 8)
    Yr, A = reference(X, q, ocb)
    check_linear(Y[:, rows], Yr, A)
    w2 = workloads.weights_np(333, K, seed=25)
    c2, cb2 = logq.logq_quantize(torch.from_numpy(w2).cuda(), 8, 1.08)
    ya, yb = logq.logq_linear_grouped([(codes, cb, N, None), (c2, cb2, 333, None)], X, K)
    assert torch.equal(ya, logq.logq_linear(codes, cb, X, N, K))
    assert torch.equal(yb, logq.logq_linear(c2, cb2, X, 333, K))


def test_one_hot_returns_decoded_column(logq):
    N, K = 96, 256
    w = workloads.weights_np(N, K, seed=31)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.05)
    ocb = oracle.build_codebook(8, 1.05, cb.range)
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, 8)
    What = oracle.dequant(q, ocb, oracle.TABLE_BF16)
    for k in (0, 1, 77, 255):
        X = torch.zeros(1, K, dtype=torch.bfloat16, device="cuda")
        X[0, k] = 1.0
        Y = logq.logq_linear(codes, cb, X, N, K).double().cpu().numpy()[0]
        np.testing.assert_array_equal(Y, What[:, k])          # one product: exact in fp32


def test_energy_range_8bit(logq):
    """Self-calibrating 8-bit quantisation with the paper's 8-bit eps = 1e-6."""
    w = workloads.weights_np(512, 2048, seed=41, outliers=True)
    codes, cb, wmin = logq.logq_quantize_energy(torch.from_numpy(w).cuda(), 8, 1e-6)
    assert wmin == oracle.energy_wmin(w, 1e-6)
    wmax = float(np.abs(w).max())
    base = oracle.base_from_range(wmax, wmin, 8)
    assert cb.range == wmax and cb.base == base
    ocb = oracle.build_codebook(8, base, wmax)
    check_codes(codes.cpu().numpy(), w, ocb, 8)


@pytest.mark.parametrize("N,K,B", [(64, 256, 5), (256, 512, 128), (300, 1152, 200), (1024, 2048, 256),
                                   (512, 4096, 2048)])
@pytest.mark.parametrize("ydt", [None, torch.bfloat16])
def test_prefill8(logq, N, K, B, ydt):
    """Batches above 4 run the tensor-core prefill with 8-bit codes (ragged
    token tiles and weight-row tiles included)."""
    w = workloads.weights_np(N, K, seed=N + K + B)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, 1.05)
    ocb = oracle.build_codebook(8, 1.05, cb.range)
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, 8)
    X = workloads.activations_torch(B, K, B, torch.bfloat16, "cuda")
    ws = logq.new_workspace()
    Y = logq.logq_linear(codes, cb, X, N, K, y_dtype=ydt, workspace=ws)
    Yr, A = reference(X, q, ocb)
    check_linear(Y.double().cpu().numpy(), Yr, A, "f32" if ydt is None else "bf16")
    st, _ = logq.logq_workspace_status(ws)
    assert st == logq.LOGQ_OK


@pytest.mark.parametrize("base", [1.005, 1.0075, 1.02, 1.05, 1.1, 1.5, 2.0])
@pytest.mark.parametrize("mode", [0, 1])
def test_quantize8_every_boundary_and_neighbours(logq, base, mode):
    """8-bit codes of all 127 fp32 boundaries, their fp32 neighbours, both signs,
    subnormals, zeros and values far outside the range: bit-exact.  The bases cover
    the estimate-and-correct kernel (boundary ratios 2^0.01 .. 2^4, first boundary at
    least 2^-120) and the boundary search on both sides of its guards."""
    rng_ = 0.75
    ocb = oracle.build_codebook(8, base, rng_, mode)
    t = np.asarray(ocb.taus32_up, np.float32)
    t = t[t > 0]
    near = np.concatenate([t, np.nextafter(t, np.float32(0)), np.nextafter(t, np.float32(np.inf))])
    extra = np.float32([0.0, -0.0, 1e-45, -1e-45, 1e-39, 1.1754942e-38, 1e-30, 0.5, 0.75, 0.7500001,
                        3.0, 1e30, 3.4e38, -3.4e38])
    rnd = (np.random.default_rng(int(base * 1e4) + mode).standard_normal(128 * 32) * 0.2).astype(np.float32)
    w = np.concatenate([near, -near, extra, rnd]).astype(np.float32)
    w = np.concatenate([w, np.zeros((-w.size) % 128, np.float32)]).reshape(-1, 128)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 8, base, rng_, mode)
    assert check_codes(codes.cpu().numpy(), w, ocb, 8) == 0
