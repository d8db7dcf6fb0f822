"""Self-calibrating quantisation (Sec. 3.2, Eqs. (3)-(5)) against the oracle:
w_min equals the oracle's energy-based w_min (Eq. (5)) -- except where the
energy share at the two candidates lies within a rounding step of eps, which is
reported -- the base is Eq. (3) of (w_max, w_min), and the packed codes are
bit-exact against the oracle's quantiser with that codebook."""
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


def energy_share(w: np.ndarray, t: float) -> float:
    a = np.abs(w.astype(np.float64)).ravel()
    return float(np.sum(a[a <= t] ** 2) / np.sum(a * a))


def check_wmin(w: np.ndarray, eps: float, got: float) -> bool:
    """True when got is the oracle's w_min; False when both are valid readings
    of a near-tie (the share at the smaller one is within 1e-9 of eps)."""
    want = oracle.energy_wmin(w, eps)
    if got == want:
        return True
    lo = min(got, want)
    assert np.any(np.abs(w) == np.float32(got)), "w_min must be one of the |w_i|"
    assert abs(energy_share(w, lo) - eps) <= 1e-9 * eps, f"w_min {got} != oracle {want}"
    return False


def run_and_check(logq, w, bits, eps, flags=0):
    W = torch.from_numpy(w).cuda()
    codes, cb, wmin = logq.logq_quantize_energy(W, bits, eps, flags)
    exact = check_wmin(w, eps, wmin)
    wmax = float(np.abs(w).max())
    assert cb.range == wmax                                           # w_max = max |W|
    base = oracle.base_from_range(wmax, wmin, bits)                   # Eq. (3)
    assert cb.base == base and cb.flags == flags
    ocb = oracle.build_codebook(bits, base, wmax, flags)
    nb = check_codes(codes.cpu().numpy(), w, ocb, bits)
    return wmin, exact, nb


@pytest.mark.parametrize("N,K,bits,eps", [(512, 2048, 4, 4e-3), (300, 4096, 3, 4e-3), (1, 128, 4, 4e-3),
                                          (7, 384, 4, 0.25), (64, 2048, 4, 1e-6), (33, 1152, 3, 0.9),
                                          (1000, 4096, 4, 4e-3)])
def test_energy_range_matches_oracle(logq, N, K, bits, eps):
    w = workloads.weights_np(N, K, seed=N + 3 * K + bits, outliers=(N * K >= 100000))
    wmin, exact, nb = run_and_check(logq, w, bits, eps)
    assert exact
    assert nb <= 2
    # Eq. (5) by itself: the share reaches eps at w_min and not below it
    a = np.abs(w.astype(np.float64))
    assert energy_share(w, wmin) >= eps * (1 - 1e-12)
    below = a[a < wmin]
    assert float(np.sum(below * below) / np.sum(a * a)) < eps * (1 + 1e-12)


def test_energy_range_floor_shift(logq):
    w = workloads.weights_np(128, 2048, seed=5, outliers=True)
    run_and_check(logq, w, 4, 4e-3, flags=1)


def test_energy_range_duplicates_and_zeros(logq):
    """Few distinct magnitudes (every threshold value has many copies) and a
    third of the weights exactly zero."""
    rng = np.random.default_rng(7)
    vals = np.array([0.0, 1e-3, 2.5e-3, 0.01, 0.02, 0.05, 0.3], dtype=np.float32)
    w = rng.choice(vals, size=(96, 1024), p=[0.33, 0.2, 0.15, 0.12, 0.1, 0.08, 0.02]).astype(np.float32)
    w *= np.where(rng.random(w.shape) < 0.5, -1.0, 1.0).astype(np.float32)
    for eps in (1e-4, 4e-3, 0.05, 0.1):                 # the 0.3 magnitude alone holds 87 % of the energy
        wmin, exact, _ = run_and_check(logq, w, 4, eps)
        assert exact and np.float32(wmin) in vals


def test_energy_range_subnormal_wmin(logq):
    """eps so small that the smallest non-zero magnitude (subnormal) is w_min."""
    w = workloads.weights_np(16, 1024, seed=9)
    w[0, :3] = np.array([1e-40, -3e-42, 2e-39], dtype=np.float32)
    wmin, exact, _ = run_and_check(logq, w, 4, 1e-300)
    assert exact and wmin == float(np.float32(3e-42))


def test_energy_range_rejects_degenerate(logq):
    W = torch.zeros(4, 128, device="cuda")
    with pytest.raises(logq.LogqError) as e:
        logq.logq_quantize_energy(W, 4, 4e-3)                          # all zero: no range
    assert e.value.status == logq.LOGQ_ERR_INVALID_ARG
    W = torch.full((4, 128), -0.5, device="cuda")
    with pytest.raises(logq.LogqError) as e:
        logq.logq_quantize_energy(W, 4, 4e-3)                          # one magnitude: b = 1
    assert e.value.status == logq.LOGQ_ERR_INVALID_ARG
    w = workloads.weights_np(8, 256, seed=2)
    with pytest.raises(logq.LogqError) as e:
        logq.logq_quantize_energy(torch.from_numpy(w).cuda(), 4, 1.0)   # eps = 1: w_min = w_max
    assert e.value.status == logq.LOGQ_ERR_INVALID_ARG
    w[3, 17] = np.nan
    with pytest.raises(logq.LogqError) as e:
        logq.logq_quantize_energy(torch.from_numpy(w).cuda(), 4, 4e-3)
    assert e.value.status == logq.LOGQ_ERR_NONFINITE


def test_energy_range_repeatable(logq):
    W = torch.from_numpy(workloads.weights_np(256, 4096, seed=4, outliers=True)).cuda()
    c1, cb1, m1 = logq.logq_quantize_energy(W, 4, 4e-3)
    c2, cb2, m2 = logq.logq_quantize_energy(W, 4, 4e-3)
    assert m1 == m2 and cb1.base == cb2.base and torch.equal(c1, c2)


def test_energy_range_full_size_gate_8b(logq):
    """Llama-3.1-8B gate shape (14336 x 4096, Student-t(4)*0.02 + 0.1 % x20
    outliers, as the bench generates it): Eq. (5) holds at the device's w_min
    (fp64 shares over all 58.7 M weights), w_min is a data value, and the codes
    of sampled rows are bit-exact against the oracle with the derived codebook."""
    N, K = 14336, 4096
    Wt = workloads.weights_torch(N, K, workloads.layer_seed(4, 0, 4), outliers=True, device="cuda")
    codes, cb, wmin = logq.logq_quantize_energy(Wt, 4, 4e-3)
    w = Wt.cpu().numpy()
    a = np.abs(w.astype(np.float64)).ravel()
    tot = np.sum(a * a)
    assert np.sum(a[a <= wmin] ** 2) / tot >= 4e-3 * (1 - 1e-12)
    assert np.sum(a[a < wmin] ** 2) / tot < 4e-3 * (1 + 1e-12)
    assert np.any(a == wmin)
    wmax = float(a.max())
    assert cb.range == wmax and cb.base == oracle.base_from_range(wmax, wmin, 4)
    ocb = oracle.build_codebook(4, cb.base, wmax)
    rows = np.random.default_rng(0).choice(N, 64, replace=False)
    c = codes.view(N, K // 2).cpu().numpy()
    for r in rows:
        check_codes(c[r:r + 1].ravel(), w[r:r + 1], ocb, 4)
