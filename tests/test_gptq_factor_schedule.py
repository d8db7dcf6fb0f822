"""The launch schedule of the GPTQ factor (blocked Cholesky of the
index-reversed damped Hessian on 64-wide blocks, diagonal blocks replaced by
their inverses, then the triangular inverse by doubling with complete and
shortened pairs, then the reversal), emulated on the CPU in fp64 with numpy:
every product reads and writes inside its buffers, and the result equals the
oracle's factor (the Cholesky factor of the inverse, computed the textbook
way).  The products follow the kernels' operand conventions: element
offsets, leading dimensions and per-pair strides."""
import numpy as np
import pytest

import oracle

NB = 64


def gemm(buf, a, b, c, M, N, Kd, alpha, beta, batch=1, strides=(0, 0, 0), bt=False, lower=False):
    """C = beta C + alpha A B (B given transposed when bt), operands as
    (buffer, element offset, leading dimension)."""
    (ba, oa, lda), (bb, ob, ldb), (bc, oc, ldc) = a, b, c
    for z in range(batch):
        a0, b0, c0 = oa + z * strides[0], ob + z * strides[1], oc + z * strides[2]
        assert a0 + (M - 1) * lda + Kd <= buf[ba].size
        assert b0 + ((N - 1) * ldb + Kd if bt else (Kd - 1) * ldb + N) <= buf[bb].size
        assert c0 + (M - 1) * ldc + N <= buf[bc].size
        A = np.lib.stride_tricks.as_strided(buf[ba][a0:], (M, Kd), (8 * lda, 8)).copy()
        if bt:
            B = np.lib.stride_tricks.as_strided(buf[bb][b0:], (N, Kd), (8 * ldb, 8)).T.copy()
        else:
            B = np.lib.stride_tricks.as_strided(buf[bb][b0:], (Kd, N), (8 * ldb, 8)).copy()
        C = np.lib.stride_tricks.as_strided(buf[bc][c0:], (M, N), (8 * ldc, 8))
        P = alpha * (A @ B) + (beta * C if beta != 0 else 0.0)
        if lower:                     # tiles of 128 strictly above the diagonal are skipped
            ti = np.arange(M)[:, None] // 128
            tj = np.arange(N)[None, :] // 128
            P = np.where(tj > ti, C, P)
        C[...] = P


def factor(H, damp):
    K = H.shape[0]
    mean = np.mean(np.diag(H))
    A = H[::-1, ::-1].copy()
    d = np.diag(A).copy()
    A[np.diag_indices(K)] = np.where(d == 0, 1.0, d) + damp * mean
    buf = {0: A.reshape(-1).copy(), 1: np.zeros(K * K // 4)}
    W = buf[0].reshape(K, K)
    for k0 in range(0, K, NB):
        blk = np.tril(W[k0:k0 + NB, k0:k0 + NB])
        L = np.linalg.cholesky(blk + np.tril(blk, -1).T)
        W[k0:k0 + NB, k0:k0 + NB] = np.linalg.inv(L)
        k1, m = k0 + NB, K - k0 - NB
        if m <= 0:
            break
        gemm(buf, (0, k1 * K + k0, K), (0, k0 * K + k0, K), (0, k1 * K + k0, K), m, NB, NB, 1.0, 0.0, bt=True)
        gemm(buf, (0, k1 * K + k0, K), (0, k1 * K + k0, K), (0, k1 * K + k1, K), m, m, NB, -1.0, 1.0,
             bt=True, lower=True)
    W[np.triu_indices(K, 1)] = 0.0
    half = NB
    while half < K:
        s = 2 * half
        full = K // s

        def combine(p0, count, c, xoff):
            t0 = p0 * s
            b0 = t0 + half
            st = s * K + s
            gemm(buf, (0, b0 * K + t0, K), (0, t0 * K + t0, K), (1, xoff, half), c, half, half, 1.0, 0.0,
                 count, (st, st, c * half))
            gemm(buf, (0, b0 * K + b0, K), (1, xoff, half), (0, b0 * K + t0, K), c, half, c, -1.0, 0.0,
                 count, (st, c * half, st))

        if full > 0:
            combine(0, full, half, 0)
        b0 = full * s + half
        if b0 < K:
            combine(full, 1, K - b0, full * half * half)
        half *= 2
    return W[::-1, ::-1].copy()


@pytest.mark.parametrize("K", [128, 384, 640, 1152, 1408])
def test_factor_schedule_matches_oracle(K):
    rng = np.random.default_rng(K)
    X = rng.standard_normal((2 * K, K))
    X[:, 1:] += 0.5 * X[:, :-1]
    H = X.T @ X
    H[3, :] = H[:, 3] = 0.0
    U = factor(H, 0.01)
    Uo = oracle.gptq_factor(H, 0.01)
    assert np.all(np.tril(U, -1) == 0.0)
    np.testing.assert_allclose(U, Uo, rtol=0, atol=1e-12 * np.max(np.abs(Uo)))
