"""The level estimate of the estimate-and-correct quantise kernels, emulated on
the CPU with numpy integers: for every codebook inside the kernels' guards the
estimate is the true boundary count m = #{j : |w| >= thresh_j} or m - 1, so one
comparison with the fp32 boundary the estimate points at gives m exactly.

The integer steps follow the kernels: u2 = 2|w| as a bit pattern (the bit
pattern of a positive normal float, read as an integer, is a piecewise-linear
log2 at most 0.0861 below log2), optionally corrected by a 64-entry table of
lower bounds of log2(1 + f) - f over the top 6 mantissa bits (8 bits), then
floor((u2 K + C) / 2^S) clamped to [0, q_max] with K = round(2^(S-24) / lambda),
C = round(-(log2 thresh_0 + 127) 2^24 K + 0.95 2^S): S = 32 for 3 and 4 bits
(lambda in [0.12, 3]), S = 40 for 8 bits (lambda in [0.01, 4], thresh_0 >= 2^-120).
The boundaries come from the oracle's codebook (Eq. (2) midpoints rounded up to fp32).

The 3-bit kernel also packs differently from a plain per-code loop: each weight
adds m + 4 * sign into its 3-bit slot of a 30-bit word and the signs of zero
magnitudes are cleared per word with slot masks; that packing is emulated here
too and compared byte for byte with the oracle's packing of its own codes."""
import numpy as np
import pytest

import oracle


def _g(f):
    return np.log2(1.0 + f) - f


CORR = np.array([np.floor(2.0 ** 24 * min(_g(i / 64), _g((i + 1) / 64))) for i in range(64)], dtype=np.int64)


def _params(t32, q, shift):
    l0 = np.log2(np.float64(t32[0]))
    lam = (np.log2(np.float64(t32[q - 1])) - l0) / (q - 1)
    k = int(round(2.0 ** (shift - 24) / lam))
    c = int(round(-(l0 + 127.0) * 2.0 ** 24 * k + 0.95 * 2.0 ** shift))
    return lam, k, c


def _estimate(u2, k, c, q, shift, table):
    v = u2.astype(np.int64)
    if table:
        v = v + CORR[(v >> 18) & 63]
    return np.clip(np.floor_divide(v * k + c, 2 ** shift), 0, q)


def _check(bits, base, rng_, mode, rng):
    q = (1 << (bits - 1)) - 1
    shift, table = (32, False) if bits in (3, 4) else (40, True)
    cb = oracle.build_codebook(bits, base, rng_, mode)
    t32 = np.asarray(cb.taus32_up, dtype=np.float32)
    lam, k, c = _params(t32, q, shift)
    if bits in (3, 4):
        inside = t32[0] >= np.finfo(np.float32).tiny and 0.12 <= lam <= 3.0
    else:
        inside = t32[0] >= 2.0 ** -120 and 0.01 <= lam <= 4.0
    if not inside:
        return False
    w = (rng.standard_normal(20000) * rng_ * rng.uniform(0.001, 2)).astype(np.float32)
    near = np.concatenate([t32, np.nextafter(t32, np.float32(0)), np.nextafter(t32, np.float32(np.inf))])
    w = np.concatenate([w, near, -near, np.float32([0.0, -0.0, 1e-45, 1e-39, 1e-38, 3.4e38])])
    u = w.view(np.uint32).astype(np.uint64) & 0x7FFFFFFF
    m_true = np.searchsorted(t32.view(np.uint32).astype(np.uint64), u, side="right")
    u2 = u * 2
    mh = _estimate(u2, k, c, q, shift, table)
    assert np.all((m_true - mh >= 0) & (m_true - mh <= 1)), (bits, base, rng_, mode)
    t2 = np.concatenate([2 * t32.view(np.uint32).astype(np.uint64), [0xFFFFFFFF]])
    assert np.array_equal(mh + (u2 >= t2[mh]), m_true)
    return True


@pytest.mark.parametrize("bits,lo,hi", [(3, 1.087, 8.0), (4, 1.087, 8.0), (8, 1.007, 1.6)])
def test_estimate_is_m_or_m_minus_1(bits, lo, hi):
    rng = np.random.default_rng(bits)
    checked = 0
    for _ in range(60):
        base = float(np.exp(rng.uniform(np.log(lo), np.log(hi))))
        checked += _check(bits, base, float(10 ** rng.uniform(-3, 3)), int(rng.integers(0, 2)), rng)
    assert checked >= 40


def test_correction_table_is_a_lower_bound():
    f = np.linspace(0.0, 1.0, 64 * 1024 + 1)[:-1]
    idx = (f * 64).astype(int)
    gap = 2.0 ** 24 * _g(f) - CORR[idx]
    assert gap.min() >= 0.0 and gap.max() <= 2.0 ** 24 * 0.0069


K_LOW, K_BIT2 = 0x1B6DB6DB, 0x24924924      # 0b011 / 0b100 in each of ten 3-bit slots


def _pack3e(w, t32, k, c):
    """quantize3e_kernel's steps for rows of w (K a multiple of 32): estimate,
    one boundary comparison, m + 4 * sign per 3-bit slot, per-word clearing of
    the signs of zero magnitudes, pair 15 split over the words' top bits."""
    N, K = w.shape
    bits = w.view(np.uint32).astype(np.uint64)
    u2 = (bits << 1) & 0xFFFFFFFF
    mh = np.clip(np.floor_divide(u2.astype(np.int64) * k + c, 2 ** 32), 0, 3)
    t2 = np.concatenate([2 * t32.view(np.uint32).astype(np.uint64), [0xFFFFFFFF]])
    val = (mh + (u2 >= t2[mh]) + ((bits >> 31) << 2)).astype(np.uint64).reshape(N, K // 32, 32)
    words = np.zeros((N, K // 32, 3), dtype=np.uint64)
    for e in range(30):
        words[:, :, e // 10] += val[:, :, e] << np.uint64(3 * (e % 10))
    lo = words & K_LOW
    words = lo | (words & ((lo + K_LOW) & K_BIT2))
    c30, c31 = val[:, :, 30], val[:, :, 31]
    c30 = (c30 & 3) | (c30 & (((c30 & 3) + 3) & 4))
    c31 = (c31 & 3) | (c31 & (((c31 & 3) + 3) & 4))
    f15 = c30 | (c31 << np.uint64(3))
    for j in range(3):
        words[:, :, j] |= ((f15 >> np.uint64(2 * j)) & 3) << np.uint64(30)
    return words.astype(np.uint32).reshape(N, -1).view(np.uint8)


def test_pack3e_matches_oracle_packing():
    rng = np.random.default_rng(33)
    done = 0
    for _ in range(40):
        base = float(np.exp(rng.uniform(np.log(1.087), np.log(8.0))))
        rng_ = float(10 ** rng.uniform(-3, 3))
        cb = oracle.build_codebook(3, base, rng_, int(rng.integers(0, 2)))
        t32 = np.asarray(cb.taus32_up, dtype=np.float32)
        lam, k, c = _params(t32, 3, 32)
        if not (t32[0] >= np.finfo(np.float32).tiny and 0.12 <= lam <= 3.0):
            continue
        near = np.concatenate([t32, np.nextafter(t32, np.float32(0)), np.nextafter(t32, np.float32(np.inf))])
        special = np.float32([0.0, -0.0, 1e-45, -1e-45, 1e-39, -1e-38, 3.4e38, -3.4e38])
        w = (rng.standard_normal(64 * 96) * rng_ * rng.uniform(0.001, 2)).astype(np.float32)
        extra = np.concatenate([near, -near, special])
        w[: extra.size] = extra
        w = rng.permutation(w).reshape(64, 96)
        assert np.array_equal(_pack3e(w, t32, k, c), oracle.pack(oracle.quantize_log(w, cb), 3))
        done += 1
    assert done >= 25
