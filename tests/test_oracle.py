"""Pins of the fp64 oracle against what the paper and mathematics fix.

Nothing here compares the oracle with itself: every check is a closed form,
a hand-worked example (tests/golden), a library routine (numpy / torch
casts and matmul), an independent route (frexp for base 2, brute force), or
an invariant that a dropped term, a wrong sign or a swapped index breaks.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2607_01127_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------ codebook ---

# 8-bit codes (q_max = 127) use bases near 1, as Eq. (3) gives them for 127 steps
@pytest.mark.parametrize("bits,base", [(b, x) for b in (3, 4) for x in (1.2, 1.25, 1.5, 2.0, 3.7)]
                         + [(8, x) for x in (1.02, 1.05, 1.1)])
@pytest.mark.parametrize("rng_", [0.0173, 0.5, 1.0, 2.75])
def test_codebook_closed_forms_exact_shift(bits, base, rng_):
    cb = oracle.build_codebook(bits, base, rng_)
    qmax = 2 ** (bits - 1) - 1
    assert cb.qmax == qmax                                   # Sec. 3.1
    L = cb.levels
    assert L.size == qmax + 1 and L[0] == 0.0                # Dequant(q=0) = 0, Eq. (2)
    # top level equals the range: b^(q_max - s) with s = q_max - log_b(range)
    assert L[qmax] == rng_
    assert np.float32(cb.levels32[qmax]) == np.float32(rng_)
    # strictly increasing, constant ratio b (q_max log steps, Eq. (3))
    assert np.all(np.diff(L[1:]) > 0)
    np.testing.assert_allclose(L[2:] / L[1:-1], base, rtol=1e-13)
    # closed form of the lowest level
    assert math.isclose(L[1], rng_ * base ** (1 - qmax), rel_tol=1e-13)
    # s from its definition
    assert math.isclose(cb.shift, qmax - math.log(rng_) / math.log(base), rel_tol=1e-13, abs_tol=1e-13)
    # Eq. (2) directly: b^(m - s)
    for m in range(1, qmax + 1):
        assert math.isclose(L[m], base ** (m - cb.shift), rel_tol=1e-12)
    # decision boundaries are geometric midpoints of neighbouring levels
    T = cb.taus
    assert T.size == qmax
    np.testing.assert_allclose(T[1:], np.sqrt(L[1:-1] * L[2:]), rtol=1e-13)
    assert math.isclose(T[0], L[1] / math.sqrt(base), rel_tol=1e-13)
    # fp32 boundaries are the smallest fp32 not below the fp64 boundary
    T32 = cb.taus32_up.astype(np.float64)
    assert np.all(T32 >= T)
    below = np.nextafter(cb.taus32_up, np.float32(0)).astype(np.float64)
    assert np.all(below < T)


@pytest.mark.parametrize("bits", [3, 4, 8])
@pytest.mark.parametrize("base,rng_,top", [(2.0, 0.75, 0.5), (2.0, 1.0, 1.0), (2.0, 0.25, 0.25),
                                           (1.5, 1.0, 1.0), (1.5, 2.0, 1.5), (4.0, 0.2, 1 / 16)])
def test_codebook_floor_shift(bits, base, rng_, top):
    """Eq. (4) as printed: s = q_max - floor(log_b w_max); top level = b^floor(log_b range)."""
    cb = oracle.build_codebook(bits, base, rng_, oracle.SHIFT_FLOOR)
    qmax = cb.qmax
    assert cb.shift == round(cb.shift)                      # integer shift
    L = cb.levels
    assert math.isclose(L[qmax], top, rel_tol=1e-13)
    assert L[qmax] <= rng_ < L[qmax] * base
    np.testing.assert_allclose(L[2:] / L[1:-1], base, rtol=1e-13)


def test_codebook_golden_hand_example():
    g = json.load(open(os.path.join(GOLDEN, "codebook_b2_r1_4bit.json")))
    cb = oracle.build_codebook(g["bits"], g["base"], g["range"])
    assert cb.qmax == g["qmax"]
    assert cb.shift == g["shift"]
    np.testing.assert_array_equal(cb.levels, np.array(g["levels"]))
    np.testing.assert_allclose(np.log2(cb.taus), g["tau_log2"], rtol=0, atol=1e-13)
    w = np.array([c["w"] for c in g["quant_cases"]], dtype=np.float32)
    want = np.array([c["q"] for c in g["quant_cases"]], dtype=np.int8)
    for route in (oracle.quantize_log, oracle.quantize_argmin, oracle.quantize_thresh):
        np.testing.assert_array_equal(route(w, cb), want)


@pytest.mark.parametrize("args", [(5, 1.5, 1.0), (1, 1.5, 1.0), (4, 1.0, 1.0), (4, 0.5, 1.0),
                                  (4, 1.5, 0.0), (4, 1.5, -1.0), (4, float("nan"), 1.0),
                                  (4, 1.5, float("inf"))])
def test_codebook_rejects_invalid(args):
    bits, base, r = args
    if bits == 5:
        # 5-bit codebooks have 16 levels: outside the tables this oracle holds
        with pytest.raises(ValueError):
            oracle.build_codebook(bits, base, r)
        return
    with pytest.raises(ValueError):
        oracle.build_codebook(bits, base, r)


# ------------------------------------------------------------ rounding ---

def test_rounding_matches_library_casts():
    import torch
    rng = np.random.Generator(np.random.PCG64(1))
    v = np.concatenate([
        rng.standard_normal(4000) * 10.0 ** rng.uniform(-8, 4, 4000),
        np.ldexp(rng.integers(1, 1 << 12, 500).astype(np.float64), -36),   # fp16 subnormals
        np.array([0.0, 65504.0, 65519.9, 1.0, -1.0, 2.0 ** -24, 2.0 ** -25 * 1.5]),
    ])
    f32 = v.astype(np.float32)
    for x, x32 in zip(v, f32):
        assert oracle.round_f32(x) == float(x32)
    bf = torch.from_numpy(f32).to(torch.bfloat16)
    bf_bits = bf.view(torch.int16).numpy().astype(np.uint16)
    f16 = f32.astype(np.float16)
    f16_bits = f16.view(np.uint16)
    for i, x32 in enumerate(f32):
        assert oracle.round_bf16(float(x32)) == float(bf[i].float())
        assert oracle.bf16_bits(float(x32)) == int(bf_bits[i])
        if abs(float(x32)) <= 65504.0:
            assert oracle.round_f16(float(x32)) == float(f16[i])
            assert oracle.f16_bits(float(x32)) == int(f16_bits[i])


@pytest.mark.parametrize("bits,base", [(b, x) for b in (3, 4) for x in (1.25, 1.5, 2.0)]
                         + [(8, x) for x in (1.02, 1.05)])
def test_codebook_16bit_tables_match_casts(bits, base):
    import torch
    cb = oracle.build_codebook(bits, base, 0.731)
    l32 = torch.from_numpy(cb.levels32)
    np.testing.assert_array_equal(cb.levels_bf16_bits,
                                  l32.to(torch.bfloat16).view(torch.int16).numpy().astype(np.uint16))
    np.testing.assert_array_equal(cb.levels_f16_bits, cb.levels32.astype(np.float16).view(np.uint16))


# ------------------------------------------------------------ quantize ---

def _weights(n=20000, seed=3):
    w = workloads.weights_np(1, n, seed, outliers=True).reshape(-1)
    w[:5] = [0.0, -0.0, 1e-30, -1e-30, 5.0]
    return w


@pytest.mark.parametrize("bits,base", [(b, x) for b in (3, 4) for x in (1.25, 1.5, 2.0)]
                         + [(8, x) for x in (1.02, 1.05, 1.1)])
@pytest.mark.parametrize("mode", [oracle.SHIFT_EXACT, oracle.SHIFT_FLOOR])
def test_three_routes_agree(bits, base, mode):
    w = _weights()
    rng_ = float(np.max(np.abs(w[5:])))
    cb = oracle.build_codebook(bits, base, rng_, mode)
    q1 = oracle.quantize_log(w, cb)
    q2 = oracle.quantize_argmin(w, cb)
    q3 = oracle.quantize_thresh(w, cb)
    np.testing.assert_array_equal(q1, q2)
    np.testing.assert_array_equal(q1, q3)
    assert q1.min() >= -cb.qmax and q1.max() <= cb.qmax
    assert q1[0] == 0 and q1[1] == 0 and q1[2] == 0 and q1[3] == 0   # zero and pruned
    assert q1[4] == cb.qmax                                         # clamped from above
    # every used magnitude bucket is non-trivial on heavy-tailed weights (at 8 bits
    # the top buckets see only the rare outliers)
    assert len(np.unique(np.abs(q1))) >= (cb.qmax if bits < 8 else 64)


@pytest.mark.parametrize("bits,base", [(b, x) for b in (3, 4) for x in (1.2, 1.5, 2.0)]
                         + [(8, x) for x in (1.02, 1.05, 1.1)])
def test_quantizing_a_level_returns_it(bits, base):
    cb = oracle.build_codebook(bits, base, 0.37)
    L = cb.levels32
    q = oracle.quantize_log(np.concatenate([L[1:], -L[1:]]), cb)
    m = np.arange(1, cb.qmax + 1, dtype=np.int8)
    np.testing.assert_array_equal(q, np.concatenate([m, -m]))


@pytest.mark.parametrize("bits", [3, 4, 8])
def test_idempotence_sign_symmetry_monotone(bits):
    w = _weights(seed=11)
    cb = oracle.build_codebook(bits, 1.5 if bits < 8 else 1.05, float(np.max(np.abs(w[5:]))))
    q = oracle.quantize_log(w, cb)
    wq = oracle.dequant(q, cb, oracle.TABLE_F32).astype(np.float32)
    np.testing.assert_array_equal(oracle.quantize_log(wq, cb), q)           # Quant(Dequant(Quant)) = Quant
    np.testing.assert_array_equal(oracle.quantize_log(-w, cb), -q)          # odd function
    a = np.sort(np.abs(w))
    qa = oracle.quantize_log(a, cb)
    assert np.all(np.diff(qa.astype(np.int32)) >= 0)                        # monotone in |w|


@pytest.mark.parametrize("bits", [3, 4, 8])
@pytest.mark.parametrize("e", [-3, 0, 2])
def test_base2_frexp_route(bits, e):
    """b = 2, range = 2^e: round(log2|x|) from frexp's exponent and a mantissa
    compare against 1/sqrt(2) -- no logarithm involved."""
    w = _weights(seed=5)[5:] * 2.0 ** e
    w = w.astype(np.float32)
    cb = oracle.build_codebook(bits, 2.0, 2.0 ** e)
    f, E = np.frexp(np.abs(w).astype(np.float64))          # |w| = f 2^E, f in [0.5, 1)
    r = np.where(f >= 1 / math.sqrt(2), E, E - 1)            # round(log2|w|), ties up
    m = np.clip(r - e + cb.qmax, 0, cb.qmax)
    want = np.where(w < 0, -m, m).astype(np.int8)
    want[w == 0] = 0
    np.testing.assert_array_equal(oracle.quantize_log(w, cb), want)


def test_absmax():
    w = _weights(seed=2)
    mx, bad = oracle.absmax(w)
    assert mx == float(np.max(np.abs(w))) and not bad
    w2 = w.copy()
    w2[7] = np.nan
    assert oracle.absmax(w2)[1]
    w2[7] = -np.inf
    assert oracle.absmax(w2)[1]


# ------------------------------------------------------------ packing ---

def test_pack_golden():
    g = json.load(open(os.path.join(GOLDEN, "codebook_b2_r1_4bit.json")))
    q4 = np.array([g["pack4_case"]["q"]], dtype=np.int8)
    np.testing.assert_array_equal(oracle.pack(q4, 4)[0], g["pack4_case"]["bytes"])
    q3 = np.zeros((1, 32), dtype=np.int8)
    for k, v in g["pack3_case"]["q_nonzero"].items():
        q3[0, int(k)] = v
    np.testing.assert_array_equal(oracle.pack(q3, 3)[0], g["pack3_case"]["bytes"])


@pytest.mark.parametrize("bits,K", [(4, 128), (4, 384), (3, 128), (3, 256), (8, 128), (8, 256)])
def test_pack_roundtrip(bits, K):
    rng = np.random.Generator(np.random.PCG64(K + bits))
    qmax = 2 ** (bits - 1) - 1
    q = rng.integers(-qmax, qmax + 1, size=(5, K)).astype(np.int8)
    p = oracle.pack(q, bits)
    assert p.shape == (5, {4: K // 2, 3: 3 * K // 8, 8: K}[bits])
    np.testing.assert_array_equal(oracle.unpack(p, 5, K, bits), q)
    if bits == 4:        # low nibble = even k, sign bit 3
        codes = np.where(q < 0, 8 | -q.astype(np.int32), q.astype(np.int32))
        np.testing.assert_array_equal(p, (codes[:, 0::2] | (codes[:, 1::2] << 4)).astype(np.uint8))
    if bits == 8:        # one code per byte, sign bit 7
        codes = np.where(q < 0, 128 | -q.astype(np.int32), q.astype(np.int32))
        np.testing.assert_array_equal(p, codes.astype(np.uint8))


# ------------------------------------------------------------ dequant + linear ---

@pytest.mark.parametrize("table", [oracle.TABLE_F64, oracle.TABLE_F32, oracle.TABLE_BF16, oracle.TABLE_F16])
def test_dequant_tables(table):
    cb = oracle.build_codebook(4, 1.5, 0.9)
    q = np.arange(-7, 8, dtype=np.int8)
    v = oracle.dequant(q, cb, table)
    ref = {oracle.TABLE_F64: cb.levels, oracle.TABLE_F32: cb.levels32.astype(np.float64),
           oracle.TABLE_BF16: oracle.bf16_bits_to_f64(cb.levels_bf16_bits),
           oracle.TABLE_F16: oracle.f16_bits_to_f64(cb.levels_f16_bits)}[table]
    np.testing.assert_array_equal(v[7:], ref)
    np.testing.assert_array_equal(v[:7], -ref[1:][::-1])


def test_linear_matches_matmul_and_probes():
    rng = np.random.Generator(np.random.PCG64(9))
    X = rng.standard_normal((3, 96))
    W = rng.standard_normal((17, 96))
    Y, A = oracle.linear(X, W)
    np.testing.assert_allclose(Y, X @ W.T, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(A, np.abs(X) @ np.abs(W).T, rtol=1e-12)
    E = np.zeros((1, 96))
    E[0, 40] = 1.0
    np.testing.assert_array_equal(oracle.linear(E, W)[0][0], W[:, 40])   # one-hot picks column k
    np.testing.assert_array_equal(oracle.linear(np.zeros((1, 96)), W)[0], 0.0)


@pytest.mark.parametrize("bits", [3, 4, 8])
def test_linear_sampled_matches_dense(bits):
    rng = np.random.Generator(np.random.PCG64(21))
    N, K = 9, 256
    w = workloads.weights_np(N, K, 4)
    cb = oracle.build_codebook(bits, 1.5, float(np.abs(w).max()))
    q = oracle.quantize_log(w, cb)
    p = oracle.pack(q, bits)
    X = rng.standard_normal((2, K))
    Y, A = oracle.linear(X, oracle.dequant(q, cb, oracle.TABLE_BF16))
    bs = np.array([0, 1, 1, 0]); ns = np.array([0, 8, 3, 5])
    Ys, As = oracle.linear_sampled(X, p, bits, cb, oracle.TABLE_BF16, bs, ns)
    np.testing.assert_array_equal(Ys, Y[bs, ns])
    np.testing.assert_array_equal(As, A[bs, ns])


# ------------------------------------------------------------ Eqs. (3), (5) ---

def _wmin_bruteforce(w, eps):
    a = np.abs(w.astype(np.float64))
    tot = np.sum(a * a)
    best = None
    for t in np.unique(a):
        if np.sum(a[a <= t] ** 2) / tot >= eps and (best is None or t < best):
            best = t
    return best


def test_energy_wmin_hand_and_bruteforce():
    w = np.array([1.0, -2.0, 3.0], dtype=np.float32)      # energies 1, 4, 9 of 14
    assert oracle.energy_wmin(w, 1 / 14) == 1.0
    assert oracle.energy_wmin(w, 0.1) == 2.0
    assert oracle.energy_wmin(w, 5 / 14 + 1e-9) == 3.0
    assert oracle.energy_wmin(w, 1.0) == 3.0
    rng = np.random.Generator(np.random.PCG64(4))
    for trial in range(20):
        v = (rng.standard_t(4, size=rng.integers(1, 60)) * 0.02).astype(np.float32)
        v[rng.integers(0, v.size)] = 0.0
        if not np.any(v):
            continue
        for eps in (1e-6, 4e-3, 0.05, 0.5, 0.999):
            assert oracle.energy_wmin(v, eps) == _wmin_bruteforce(v, eps)
    assert oracle.energy_wmin(np.zeros(4, np.float32), 0.1) == -1.0
    assert oracle.energy_wmin(w, 0.0) == -1.0


@pytest.mark.parametrize("bits", [3, 4, 8])
def test_base_from_range_spans_qmax_steps(bits):
    wmax, wmin = 0.8, 0.013
    b = oracle.base_from_range(wmax, wmin, bits)
    qmax = 2 ** (bits - 1) - 1
    assert math.isclose(b ** qmax, wmax / wmin, rel_tol=1e-12)
    cb = oracle.build_codebook(bits, b, wmax)
    # q_max steps of ratio b lead from w_min (the virtual level of q = 0,
    # b^(0 - s), which Eq. (2) maps to zero) up to w_max = L_qmax
    assert math.isclose(b ** (0 - cb.shift), wmin, rel_tol=1e-12)
    assert math.isclose(cb.levels[1], wmin * b, rel_tol=1e-12)


# ------------------------------------------------------------ GPTQ ---

def _hessian(K, seed, T=None):
    rng = np.random.Generator(np.random.PCG64(seed))
    X = rng.standard_normal((T or 4 * K, K)) * (1.0 + rng.random(K))   # correlated-free, varied scales
    X[:, 1:] += 0.5 * X[:, :-1]                                        # neighbouring inputs correlate
    return X.T @ X


@pytest.mark.parametrize("bits", [4, 8])
def test_gptq_diagonal_hessian_is_plain_rounding(bits):
    """With a diagonal Hessian no column informs another: GPTQ = rounding to nearest."""
    w = workloads.weights_np(16, 64, 8)
    cb = oracle.build_codebook(bits, 1.5 if bits == 4 else 1.05, float(np.abs(w).max()))
    H = np.diag(np.random.Generator(np.random.PCG64(1)).random(64) + 0.5)
    q, w_at = oracle.gptq(w, H, cb)
    np.testing.assert_array_equal(q, oracle.quantize_thresh(w, cb))
    np.testing.assert_array_equal(w_at, w.astype(np.float64))


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("K", [2, 7, 24])
def test_gptq_compensation_is_least_squares(bits, K):
    """The value column j is quantised at is the j-th entry of the minimiser of
    (x - w) Hd (x - w)^T with the earlier columns fixed at their levels --
    solved here directly, without the Cholesky route the oracle takes."""
    N, damp = 5, 0.01
    w = workloads.weights_np(N, K, 9 + K)
    cb = oracle.build_codebook(bits, 1.4 if bits == 4 else 1.05, float(np.abs(w).max()))
    H = _hessian(K, K)
    q, w_at = oracle.gptq(w, H, cb, damp)
    Hd = H + damp * np.mean(np.diag(H)) * np.eye(K)
    deq = oracle.dequant(q, cb, oracle.TABLE_F32)
    wd = w.astype(np.float64)
    for j in range(1, K):
        d, r = slice(0, j), slice(j, K)
        delta = deq[:, d] - wd[:, d]                                  # fixed changes of done columns
        x_r = wd[:, r] - np.linalg.solve(Hd[r, r], Hd[r, d] @ delta.T).T
        np.testing.assert_allclose(w_at[:, j], x_r[:, 0], rtol=1e-9, atol=1e-12)


def test_gptq_lowers_the_layer_loss():
    """tr((W - What) Hd (W - What)^T) below that of plain rounding on correlated inputs."""
    w = workloads.weights_np(32, 96, 12)
    cb = oracle.build_codebook(4, 1.5, float(np.abs(w).max()))
    H = _hessian(96, 3)
    q, _ = oracle.gptq(w, H, cb)
    loss = lambda qq: float(np.trace((w - oracle.dequant(qq, cb, oracle.TABLE_F32)) @ H @
                                     (w - oracle.dequant(qq, cb, oracle.TABLE_F32)).T))
    assert loss(q) < 0.9 * loss(oracle.quantize_thresh(w, cb))


@pytest.mark.parametrize("bits", [4, 8])
def test_gptq_dead_input_is_the_reduced_problem(bits):
    """An input that never fires (zero Hessian row and column) is dropped: its
    weights code 0, and the other columns come out as GPTQ of the matrix without
    that column (damping rescaled so that damp * mean(diag) is the same)."""
    N, K, d = 6, 20, 7
    w = workloads.weights_np(N, K, 21)
    cb = oracle.build_codebook(bits, 1.4 if bits == 4 else 1.05, float(np.abs(w).max()))
    H = _hessian(K, 22)
    H[d, :] = H[:, d] = 0.0
    q, w_at = oracle.gptq(w, H, cb, 0.01)
    keep = [k for k in range(K) if k != d]
    q_r, w_r = oracle.gptq(np.ascontiguousarray(w[:, keep]), H[np.ix_(keep, keep)], cb, 0.01 * (K - 1) / K)
    assert np.all(q[:, d] == 0) and np.all(w_at[:, d] == 0.0)
    np.testing.assert_array_equal(q[:, keep], q_r)
    np.testing.assert_allclose(w_at[:, keep], w_r, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("K", [1, 5, 64])
def test_gptq_factor_is_the_cholesky_factor_of_the_inverse(K):
    """U is upper triangular with a positive diagonal and U^T U Hd = I: the
    Cholesky factor of Hd^-1 is the only such matrix."""
    H = _hessian(K, 30 + K)
    if K > 2:
        H[2, :] = H[:, 2] = 0.0                       # a dead input: decoupled, diagonal 1 + damping
    damp = 0.01
    U = oracle.gptq_factor(H, damp)
    mean = np.mean(np.diag(H))
    Hd = H + damp * mean * np.eye(K)
    if K > 2:
        Hd[2, 2] = 1.0 + damp * mean
        assert U[2, 2] == pytest.approx(1.0 / np.sqrt(Hd[2, 2]), rel=1e-14)
        assert np.all(U[2, 3:] == 0.0) and np.all(U[:2, 2] == 0.0)
    assert np.all(np.tril(U, -1) == 0.0) and np.all(np.diag(U) > 0)
    np.testing.assert_allclose(U.T @ U @ Hd, np.eye(K), atol=1e-9)


# ---------------------------------------------------------------- linear_asym ---
# The comparison quantiser of the error study (tensor-wise asymmetric uniform).

@pytest.mark.parametrize("bits", [3, 4, 8])
def test_linear_asym_is_the_nearest_grid_value(bits):
    """Brute force: each code is the nearest of all 2^n grid values (ties may go
    either way), the grid is uniform with step scale, and no value errs by more than
    half a step inside [min, max] except the top, which a rounded zero point can clip
    by at most one step."""
    rng = np.random.Generator(np.random.PCG64(bits))
    w = rng.standard_t(4, size=2000) * 0.02
    q, v, scale, zero = oracle.linear_asym(w, bits)
    top = (1 << bits) - 1
    grid = (np.arange(top + 1) - zero) * scale
    d = np.abs(w[:, None] - grid[None, :])
    best = d.min(axis=1)
    assert np.allclose(np.abs(w - v), best, rtol=0, atol=1e-15)
    assert np.allclose(np.diff(grid), scale)
    assert np.isclose(scale, (w.max() - w.min()) / top)
    inside = (w >= grid[0]) & (w <= grid[-1])
    assert np.all(np.abs(w - v)[inside] <= scale / 2 + 1e-15)
    assert np.all(np.abs(w - v) <= scale + 1e-15)


@pytest.mark.parametrize("bits", [3, 4, 8])
def test_linear_asym_idempotent_on_its_grid(bits):
    w = workloads.weights_np(64, 64, 3 + bits, outliers=True).reshape(-1)
    q, v, scale, zero = oracle.linear_asym(w, bits)
    q2, v2, _, _ = oracle.linear_asym(v, bits, scale, zero)
    assert np.array_equal(q, q2) and np.array_equal(v, v2)


def test_linear_asym_uniform_mse_is_step_squared_over_12():
    """For inputs spread uniformly over many grid steps the rounding error is uniform
    on [-scale/2, scale/2]: mean square error scale^2 / 12."""
    rng = np.random.Generator(np.random.PCG64(9))
    w = rng.uniform(-1.0, 3.0, size=400_000)
    _, v, scale, _ = oracle.linear_asym(w, 4)
    mse = float(np.mean((w - v) ** 2))
    assert abs(mse / (scale ** 2 / 12) - 1) < 0.02
