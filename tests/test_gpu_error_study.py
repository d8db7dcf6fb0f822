"""Synthetic quantisation-error study: Log_b against tensor-wise asymmetric linear
quantisation at 3, 4 and 8 bits (the comparison of Sec. 2 / Fig. 1 of the paper,
data-free: no model weights or calibration text are used).

Weights: an Llama-3.1-8B q-shaped matrix (4096 x 4096) of Student-t(4) * 0.02 with
0.1 % x20 outliers, standing in for the bell-shaped, heavy-tailed weight
histograms of Fig. 1; activations: 16 rows of N(0, 1) in bf16.

  Log_b:  the library's self-calibrating quantiser (logq_quantize_energy: w_max,
          the Eq. (5) w_min with eps = 4e-3 at 3 and 4 bits and 1e-6 at 8 bits, the
          Eq. (3) base), then the library's linear layer (logq_linear) for X What^T;
          both checked against the oracle (codes and outputs) first.
  linear: the oracle's asymmetric uniform quantiser (scale and zero point from
          min / max of W), output in fp64.

Reported per bit width: the weight mean square error and the relative output
error ||X What^T - X W^T||_F / ||X W^T||_F, printed.  The paper's claim checked: at
3 and 4 bits Log_b quantises these weights with a smaller error than the linear
grid, on both measures.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import check_linear, lib

pytestmark = pytest.mark.gpu

EPS = {3: 4e-3, 4: 4e-3, 8: 1e-6}


@pytest.fixture(scope="module")
def logq():
    return lib()


def test_log_vs_linear_error_study(logq):
    N, K, B = 4096, 4096, 16
    Wt = workloads.weights_torch(N, K, workloads.layer_seed(6, 0, 0), outliers=True, device="cuda")
    w = Wt.cpu().numpy().astype(np.float64)
    X = workloads.activations_torch(B, K, 6, torch.bfloat16, "cuda")
    x = X.float().cpu().double().numpy()
    y_true = x @ w.T
    ny = np.linalg.norm(y_true)
    rows = []
    for bits in (3, 4, 8):
        codes, cb, wmin = logq.logq_quantize_energy(Wt, bits, EPS[bits])
        ocb = oracle.build_codebook(bits, cb.base, cb.range)
        q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, bits)
        # Log_b weights: the fp32 levels of the codes (Eq. (2)); the linear layer
        # multiplies with the bf16 table of X's dtype (checked against the oracle)
        w_log = oracle.dequant(q, ocb, oracle.TABLE_F32)
        Y = logq.logq_linear(codes, cb, X, N, K).double().cpu().numpy()
        Yr, A = oracle.linear(x, oracle.dequant(q, ocb, oracle.TABLE_BF16))
        check_linear(Y, Yr, A)
        _, w_lin, _, _ = oracle.linear_asym(w, bits)
        r = dict(bits=bits, base=cb.base,
                 mse_log=float(np.mean((w - w_log) ** 2)), mse_lin=float(np.mean((w - w_lin) ** 2)),
                 out_log=float(np.linalg.norm(Y - y_true) / ny),
                 out_lin=float(np.linalg.norm(x @ w_lin.T - y_true) / ny))
        rows.append(r)
        print(f"\n[error study] bits={bits} base={r['base']:.4f}: weight MSE log {r['mse_log']:.3e} "
              f"linear {r['mse_lin']:.3e}; output rel. error log {r['out_log']:.4f} linear {r['out_lin']:.4f}")
    for r in rows:
        if r["bits"] in (3, 4):
            assert r["mse_log"] < r["mse_lin"] and r["out_log"] < r["out_lin"], r
