"""GPTQ with the Log_b quantiser on the device against the fp64 oracle: the
factor U (fp32 on the device) against the oracle's within fp32 accuracy; a
diagonal Hessian reduces GPTQ to plain rounding (codes bit-exact against
logq_quantize); on correlated synthetic inputs the codes agree with the
oracle's except where fp32 and fp64 compensations put a weight on different
sides of a boundary (a small, counted fraction), and the layer loss
tr((W - What) H (W - What)^T) matches the oracle's and beats plain rounding."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def logq():
    return lib()


def hessian(K, seed, T=None):
    """Synthetic layer inputs (correlated neighbours, varied scales): H = X^T X."""
    rng = np.random.Generator(np.random.PCG64(seed))
    X = rng.standard_normal((T or 4 * K, K)) * (1.0 + rng.random(K))
    X[:, 1:] += 0.5 * X[:, :-1]
    return X.T @ X


def loss(w, q, cb, H):
    d = w.astype(np.float64) - oracle.dequant(q, cb, oracle.TABLE_F32)
    return float(np.einsum("ij,jk,ik->", d, H, d))


@pytest.mark.parametrize("K", [128, 384, 640, 1152])
def test_gptq_factor_matches_oracle(logq, K):
    """U from the device (fp32 Cholesky of the reversed Hessian, blocked triangular
    inverse; 2, 6, 10 and 18 blocks of 64, so the inverse's doubling meets
    complete and shortened pairs) against the oracle's fp64 factor, with a
    dead input."""
    H = hessian(K, 50 + K)
    H[3, :] = H[:, 3] = 0.0
    Hf = H.astype(np.float32)
    U, dead = logq.gptq_factor(torch.from_numpy(Hf).cuda(), 0.01)
    U = U.double().cpu().numpy()
    Uo = oracle.gptq_factor(Hf.astype(np.float64), 0.01)
    assert np.all(np.tril(U, -1) == 0.0)
    err = float(np.max(np.abs(U - Uo)) / np.max(np.abs(Uo)))
    assert err < 2e-4, err
    np.testing.assert_array_equal(dead.cpu().numpy(), (np.diag(Hf) == 0).astype(np.uint8))
    assert np.all(U[3, 4:] == 0.0) and np.all(U[:3, 3] == 0.0)


def test_gptq_factor_not_positive_definite(logq):
    H = -torch.eye(256, device="cuda")
    with pytest.raises(logq.LogqError) as ei:
        logq.gptq_factor(H, 0.01)
    assert ei.value.status == logq.LOGQ_ERR_NOT_PD


@pytest.mark.parametrize("bits,base", [(4, 1.5), (8, 1.05)])
def test_gptq_diagonal_hessian_is_plain_rounding(logq, bits, base):
    N, K = 96, 384
    w = workloads.weights_np(N, K, seed=3, outliers=True)
    W = torch.from_numpy(w).cuda()
    cb = logq.logq_build_codebook(bits, base, float(np.abs(w).max()))
    H = torch.diag(torch.rand(K, dtype=torch.float32, generator=torch.Generator().manual_seed(1)) + 0.5).cuda()
    codes = logq.logq_gptq(W, H, cb)
    ref, _ = logq.logq_quantize(W, bits, base, float(np.abs(w).max()))
    assert torch.equal(codes, ref)


@pytest.mark.parametrize("bits,base", [(4, 1.5), (8, 1.05)])
@pytest.mark.parametrize("N,K", [(256, 512), (100, 256)])
def test_gptq_matches_oracle(logq, bits, base, N, K):
    w = workloads.weights_np(N, K, seed=N + K + bits, outliers=True)
    H = hessian(K, K + bits)
    cb = logq.logq_build_codebook(bits, base, float(np.abs(w).max()))
    codes = logq.logq_gptq(torch.from_numpy(w).cuda(), torch.from_numpy(H).float().cuda(), cb)
    q_dev = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, bits)
    ocb = oracle.build_codebook(bits, base, float(np.abs(w).max()))
    q_ref, _ = oracle.gptq(w, H, ocb)
    agree = float(np.mean(q_dev == q_ref))
    assert agree >= 0.98, agree
    l_dev, l_ref = loss(w, q_dev, ocb, H), loss(w, q_ref, ocb, H)
    l_rtn = loss(w, oracle.quantize_thresh(w, ocb), ocb, H)
    assert abs(l_dev - l_ref) <= 0.01 * l_ref, (l_dev, l_ref)
    assert l_dev < l_rtn


def test_gptq_repeatable_and_dead_columns(logq):
    N, K = 64, 256
    w = workloads.weights_np(N, K, seed=8)
    H = hessian(K, 9)
    H[:, 5] = H[5, :] = 0.0                           # an input that never fires
    cb = logq.logq_build_codebook(4, 1.4, float(np.abs(w).max()))
    W, Ht = torch.from_numpy(w).cuda(), torch.from_numpy(H).float().cuda()
    c1, c2 = logq.logq_gptq(W, Ht, cb), logq.logq_gptq(W, Ht, cb)
    assert torch.equal(c1, c2)
    q = oracle.unpack(c1.cpu().numpy().reshape(N, -1), N, K, 4)
    assert np.all(q[:, 5] == 0)                       # its weights are dropped (zeroed before rounding)
    ocb = oracle.build_codebook(4, 1.4, float(np.abs(w).max()))
    q_ref, _ = oracle.gptq(w, H, ocb)
    assert float(np.mean(q == q_ref)) >= 0.98


def test_gptq_rejects_3bit(logq):
    W = torch.zeros(32, 128, device="cuda")
    H = torch.eye(128, device="cuda")
    with pytest.raises(logq.LogqError) as ei:
        logq.logq_gptq(W, H, logq.logq_build_codebook(3, 1.5, 1.0))
    assert ei.value.status == logq.LOGQ_ERR_UNSUPPORTED


def test_gptq_full_size_q_8b(logq):
    """Llama-3.1-8B q shape (4096 x 4096) with a full-rank Hessian of 3 K
    synthetic tokens and the self-calibrated codebook: the loss beats plain
    rounding at full size (losses in fp64 on the device)."""
    N, K = 4096, 4096
    W = workloads.weights_torch(N, K, 5, outliers=True, device="cuda")
    g = torch.Generator(device="cuda").manual_seed(6)
    X = torch.randn(3 * K, K, device="cuda", generator=g, dtype=torch.float64)
    X[:, 1:] += 0.5 * X[:, :-1].clone()
    H = (X.T @ X).float()
    del X
    # the paper's codebook: range and base from the weights (Eqs. (3)-(5), eps = 4e-3);
    # logq_quantize_energy's own codes are plain rounding with it
    rtn, cb, _ = logq.logq_quantize_energy(W, 4, 4e-3)
    codes = logq.logq_gptq(W, H, cb)
    lv = torch.tensor(np.array(cb.level[:16], np.float32), device="cuda")
    def deq(c):
        b = c.view(N, K // 2)
        q = torch.stack([b & 15, b >> 4], dim=-1).view(N, K).long()
        return lv[q].double()
    def L(c):
        d = W.double() - deq(c)
        return float(((d @ H.double()) * d).sum())
    l_gptq, l_rtn = L(codes), L(rtn)
    print(f"layer loss: GPTQ {l_gptq:.6g}, rounding {l_rtn:.6g}")
    assert l_gptq < l_rtn
