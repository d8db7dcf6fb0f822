"""Quantise + pack kernels against the oracle: packed codes bit-exact
(elements within one fp32 ulp of a decision boundary counted), codebook
identical, non-finite weights reported."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import check_codes, lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def logq():
    return lib()


@pytest.mark.parametrize("N,K", [(512, 2048), (1, 128), (3, 128), (7, 384), (33, 1152), (300, 4096)])
@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("base", [1.25, 1.5, 2.0])
def test_quantize_auto_range_bit_exact(logq, N, K, bits, base):
    w = workloads.weights_np(N, K, seed=N * 7 + K + bits, outliers=(N * K >= 100000))
    W = torch.from_numpy(w).cuda()
    codes, cb = logq.logq_quantize(W, bits, base)
    rng_ = float(np.abs(w).max())
    assert cb.range == rng_                                   # w_max = max |W| (Sec. 3.2)
    ocb = oracle.build_codebook(bits, base, rng_)
    np.testing.assert_array_equal(np.array(cb.thresh[:ocb.qmax], np.float32), ocb.taus32_up)
    nb = check_codes(codes.cpu().numpy(), w, ocb, bits)
    assert nb <= 2


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("mode", [0, 1])
def test_quantize_given_range_and_shift_modes(logq, bits, mode):
    N, K = 64, 2048
    w = workloads.weights_np(N, K, seed=11, outliers=True)
    W = torch.from_numpy(w).cuda()
    rng_ = 0.5 * float(np.abs(w).max())                       # values above clamp to q_max
    codes, cb = logq.logq_quantize(W, bits, 1.5, rng_, mode)
    ocb = oracle.build_codebook(bits, 1.5, rng_, mode)
    assert cb.range == rng_ and cb.flags == mode
    check_codes(codes.cpu().numpy(), w, ocb, bits)


def test_quantize_config_single_layer(logq):
    """512 x 2048, Student-t(4)*0.02, b = 1.5, range = max|W|, 4 bits, seed 0."""
    w = workloads.weights_np(512, 2048, 0)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 4, 1.5)
    ocb = oracle.build_codebook(4, 1.5, float(np.abs(w).max()))
    assert check_codes(codes.cpu().numpy(), w, ocb, 4) == 0


def test_quantize_special_values(logq):
    K = 128
    w = np.zeros((2, K), np.float32)
    cb0 = oracle.build_codebook(4, 2.0, 1.0)
    w[0, :8] = [0.0, -0.0, 1.0, -1.0, 1e-30, -1e-30, 3.0, -3.0]
    w[0, 8:15] = cb0.levels32[1:]                              # each level maps to itself
    w[1, :7] = -cb0.levels32[1:]
    w[1, 7:14] = cb0.taus32_up                                 # exactly on the fp32 boundary: rounds up
    w[1, 14:21] = np.nextafter(cb0.taus32_up, np.float32(0))   # one ulp below: rounds down
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), 4, 2.0, 1.0)
    q = oracle.unpack(codes.cpu().numpy().reshape(2, -1), 2, K, 4)
    assert list(q[0, :8]) == [0, 0, 7, -7, 0, 0, 7, -7]
    assert list(q[0, 8:15]) == list(range(1, 8))
    assert list(q[1, :7]) == [-m for m in range(1, 8)]
    assert list(q[1, 7:14]) == list(range(1, 8))
    assert list(q[1, 14:21]) == list(range(0, 7))
    check_codes(codes.cpu().numpy(), w, cb0, 4)


@pytest.mark.parametrize("bad", [np.nan, np.inf, -np.inf])
@pytest.mark.parametrize("given_range", [0.0, 1.0])
@pytest.mark.parametrize("bits", [3, 4])
def test_quantize_nonfinite_reported(logq, bad, given_range, bits):
    w = workloads.weights_np(16, 256, 5)
    w[3, 17] = bad
    with pytest.raises(logq.LogqError) as ei:
        logq.logq_quantize(torch.from_numpy(w).cuda(), bits, 1.5, given_range)
    assert ei.value.status == logq.LOGQ_ERR_NONFINITE
    # the context stays usable
    codes, _ = logq.logq_quantize(torch.from_numpy(np.nan_to_num(w, posinf=0, neginf=0)).cuda(), 4, 1.5)
    torch.cuda.synchronize()


def test_quantize_all_zero_auto_range(logq):
    with pytest.raises(logq.LogqError) as ei:
        logq.logq_quantize(torch.zeros(4, 128, device="cuda"), 4, 1.5)
    assert ei.value.status == logq.LOGQ_ERR_INVALID_ARG
    codes, _ = logq.logq_quantize(torch.zeros(4, 128, device="cuda"), 4, 1.5, 1.0)
    assert int(codes.sum()) == 0


def test_quantize_repeatable(logq):
    w = workloads.weights_np(256, 1024, 3, outliers=True)
    W = torch.from_numpy(w).cuda()
    a, _ = logq.logq_quantize(W, 4, 1.7)
    b, _ = logq.logq_quantize(W, 4, 1.7)
    assert torch.equal(a, b)


@pytest.mark.parametrize("base", [1.05, 1.087, 1.1, 1.5, 3.0, 7.9, 9.0])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("bits", [3, 4])
def test_quantize_every_boundary_and_neighbours(logq, base, mode, bits):
    """3- and 4-bit codes of every fp32 boundary, its two fp32 neighbours on each side,
    both signs, subnormals, zeros and values far outside the range: bit-exact.  Bases
    from 1.05 to 9 cover the boundary search and the estimate-and-correct kernels (used
    for boundary ratios 2^0.12 to 2^3) on both sides of their guards."""
    rng_ = 0.75
    ocb = oracle.build_codebook(bits, base, rng_, mode)
    t = np.asarray(ocb.taus32_up, np.float32)
    near = np.concatenate([t, np.nextafter(t, np.float32(0)), np.nextafter(t, np.float32(np.inf)),
                           np.nextafter(np.nextafter(t, np.float32(0)), np.float32(0)),
                           np.nextafter(np.nextafter(t, np.float32(np.inf)), np.float32(np.inf))])
    extra = np.float32([0.0, -0.0, 1e-45, -1e-45, 1e-39, 1.1754942e-38, 1.1754944e-38, 1e-20, 0.5, 0.75,
                        0.7500001, 3.0, 1e30, 3.4e38, -3.4e38])
    rnd = (np.random.default_rng(int(base * 1000) + mode).standard_normal(128 * 64) * 0.3).astype(np.float32)
    w = np.concatenate([near, -near, extra, rnd]).astype(np.float32)
    w = np.concatenate([w, np.zeros((-w.size) % 128, np.float32)]).reshape(-1, 128)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), bits, base, rng_, mode)
    assert check_codes(codes.cpu().numpy(), w, ocb, bits) == 0
