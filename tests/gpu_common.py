"""Shared helpers of the GPU parity tests (CUDA path vs fp64 oracle)."""
import numpy as np

import oracle

TOL_REL = 1e-3      # |y_gpu - y_ref| <= 1e-3 * sum_k |x_k w_k| + 1e-6
TOL_ABS = 1e-6


def lib():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_01127_gb300 as logq
    return logq


def boundary_mask(w: np.ndarray, cb) -> np.ndarray:
    """Elements whose |w| lies within one fp32 ulp of a fp64 decision boundary."""
    a = np.abs(w.astype(np.float32))
    lo = np.nextafter(a, np.float32(0)).astype(np.float64)
    hi = np.nextafter(a, np.float32(np.inf)).astype(np.float64)
    m = np.zeros(a.shape, dtype=bool)
    for t in cb.taus:
        m |= (lo <= t) & (t <= hi)
    return m


def check_codes(codes_gpu: np.ndarray, w: np.ndarray, ocb, bits: int):
    """Packed codes must equal the oracle's bit for bit, except elements within
    one ulp of a boundary, which are counted.  Returns that count."""
    N, K = w.shape
    want_q = oracle.quantize_log(w, ocb)
    got_q = oracle.unpack(codes_gpu.reshape(N, -1), N, K, bits)
    diff = got_q != want_q
    if not diff.any():
        np.testing.assert_array_equal(codes_gpu.reshape(N, -1), oracle.pack(want_q, bits))
        return 0
    bm = boundary_mask(w, ocb)
    assert not np.any(diff & ~bm), f"{int((diff & ~bm).sum())} code mismatches away from boundaries"
    assert np.all(np.abs(got_q[diff].astype(int) - want_q[diff].astype(int)) == 1)
    return int(diff.sum())


def half_ulp(v: np.ndarray, dtype: str) -> np.ndarray:
    a = np.abs(v)
    mant = 8 if dtype == "bf16" else 11
    e = np.floor(np.log2(np.maximum(a, 1e-300)))
    return np.ldexp(1.0, (e - mant + 1).astype(int)) / 2


def check_linear(Y_gpu: np.ndarray, Y_ref: np.ndarray, A: np.ndarray, ydtype: str = "f32"):
    err = np.abs(Y_gpu.astype(np.float64) - Y_ref)
    bound = TOL_REL * A + TOL_ABS
    if ydtype != "f32":
        bound = bound + half_ulp(Y_ref, ydtype) * (1 + 1e-3)
    bad = err > bound
    assert not bad.any(), (f"{int(bad.sum())} outputs out of tolerance; worst excess "
                           f"{float((err - bound).max()):.3g}")
    return float((err / np.maximum(A, 1e-30)).max())
