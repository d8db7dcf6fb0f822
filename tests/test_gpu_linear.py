"""Decode GEMV / skinny GEMM and prefill GEMM against the fp64 oracle:
|y_gpu - y_ref| <= 1e-3 * sum_k |x_k w_k| + 1e-6 for every output, with the
oracle evaluating X * What^T on the same codes and the same 16-bit table."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_01127_gb300 import workloads

from gpu_common import check_linear, lib

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def logq():
    return lib()


def make_layer(logq, N, K, bits, base, seed, outliers=False):
    w = workloads.weights_np(N, K, seed, outliers=outliers)
    codes, cb = logq.logq_quantize(torch.from_numpy(w).cuda(), bits, base)
    ocb = oracle.build_codebook(bits, base, cb.range)
    q = oracle.unpack(codes.cpu().numpy().reshape(N, -1), N, K, bits)
    return codes, cb, ocb, q


def reference(X, q, ocb):
    table = oracle.TABLE_BF16 if X.dtype == torch.bfloat16 else oracle.TABLE_F16
    return oracle.linear(X.float().cpu().double().numpy(), oracle.dequant(q, ocb, table), nthreads=0)


def run_case(logq, N, K, bits, B, xdt, ydt=None, seed=0, base=1.5):
    codes, cb, ocb, q = make_layer(logq, N, K, bits, base, seed)
    X = workloads.activations_torch(B, K, seed, xdt, "cuda")
    Y = logq.logq_linear(codes, cb, X, N, K, y_dtype=ydt)
    Yr, A = reference(X, q, ocb)
    name = {None: "f32", torch.float32: "f32", torch.bfloat16: "bf16", torch.float16: "f16"}[ydt]
    return check_linear(Y.double().cpu().numpy(), Yr, A, name)


@pytest.mark.parametrize("N,K", [(512, 2048), (7, 128), (300, 1152), (1000, 4096), (129, 14336),
                                 (2049, 384)])
@pytest.mark.parametrize("B", [1, 2, 3, 4, 5, 8, 16])
def test_gemv_4bit_bf16(logq, N, K, B):
    run_case(logq, N, K, 4, B, torch.bfloat16, seed=N + K + B)


@pytest.mark.parametrize("N,K", [(512, 2048), (7, 128), (300, 1152), (129, 14336)])
@pytest.mark.parametrize("B", [1, 2, 3, 4])
def test_gemv_3bit_bf16(logq, N, K, B):
    run_case(logq, N, K, 3, B, torch.bfloat16, seed=N + K + B, base=1.25)


@pytest.mark.parametrize("bits,B", [(4, 1), (4, 4), (4, 16), (3, 1), (3, 4)])
def test_gemv_fp16_activations(logq, bits, B):
    run_case(logq, 512, 2048, bits, B, torch.float16, seed=B)


@pytest.mark.parametrize("xdt", [torch.bfloat16, torch.float16])
@pytest.mark.parametrize("B", [1, 4, 16])
def test_gemv_16bit_output(logq, xdt, B):
    run_case(logq, 384, 1024, 4, B, xdt, ydt=xdt, seed=3)


@pytest.mark.parametrize("bits,N,K,B", [(4, 20491, 2048, 1), (4, 20491, 2048, 2), (3, 27403, 2048, 1),
                                         (3, 27403, 2048, 2), (4, 5131, 8192, 1)])
def test_gemv_large_launch(logq, bits, N, K, B):
    """Launches above the size at which the batch-1/2 decode kernel switches to
    one 16-warp CTA per SM (20 MiB of codes), ragged row counts."""
    run_case(logq, N, K, bits, B, torch.bfloat16, seed=N + B + bits)


@pytest.mark.parametrize("N,K", [(4095, 2048), (4096, 2048), (20479, 2048), (20480, 2048)])
def test_gemv_launch_shape_boundaries(logq, N, K):
    """Batch-1 launches on either side of the sizes where the decode kernel
    changes shape (4 MiB and 20 MiB of codes)."""
    run_case(logq, N, K, 4, 1, torch.bfloat16, seed=N)


def test_gemv_config_single_layer(logq):
    """512 x 2048 layer, fp16 x [1, 2048], b = 1.5, seed 0."""
    run_case(logq, 512, 2048, 4, 1, torch.float16, seed=0)


@pytest.mark.parametrize("bits", [3, 4])
def test_one_hot_returns_decoded_column(logq, bits):
    """x = e_k picks column k of What exactly (pins the code layout)."""
    N, K = 96, 256
    codes, cb, ocb, q = make_layer(logq, N, K, bits, 1.5, 4)
    wq = oracle.dequant(q, ocb, oracle.TABLE_BF16)
    for k in (0, 1, 2, 31, 32, 33, 127, 200, 255):
        X = torch.zeros(1, K, dtype=torch.bfloat16, device="cuda")
        X[0, k] = 1.0
        Y = logq.logq_linear(codes, cb, X, N, K).double().cpu().numpy()[0]
        np.testing.assert_array_equal(Y, wq[:, k])


def test_zero_and_ones(logq):
    N, K = 64, 512
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 1.5, 8)
    Y0 = logq.logq_linear(codes, cb, torch.zeros(3, K, dtype=torch.bfloat16, device="cuda"), N, K)
    assert torch.count_nonzero(Y0) == 0
    X1 = torch.ones(1, K, dtype=torch.bfloat16, device="cuda")
    Y1 = logq.logq_linear(codes, cb, X1, N, K).double().cpu().numpy()[0]
    rows = oracle.dequant(q, ocb, oracle.TABLE_BF16)
    check_linear(Y1[None], rows.sum(1)[None], np.abs(rows).sum(1)[None])


def test_hand_written_codes(logq):
    """Codes written by hand (not by the quantiser): row n holds code c(n) at
    every k, so y[n] = table[c(n)] * sum_k x_k."""
    K = 256
    cb = logq.logq_build_codebook(4, 2.0, 1.0)     # levels 2^(m-7), exact in bf16
    codes = np.zeros((16, K // 2), np.uint8)
    for c in range(16):
        codes[c, :] = c | (c << 4)
    X = torch.full((1, K), 0.5, dtype=torch.bfloat16, device="cuda")
    Y = logq.logq_linear(torch.from_numpy(codes.reshape(-1)).cuda(), cb, X, 16, K).cpu().numpy()[0]
    want = np.array([cb.level[c] * 0.5 * K for c in range(16)], dtype=np.float32)
    np.testing.assert_array_equal(Y, want)


def test_gemv_repeatable_and_stream(logq):
    N, K = 4096, 4096
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 1.5, 1)
    X = workloads.activations_torch(1, K, 1, torch.bfloat16, "cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        Ya = logq.logq_linear(codes, cb, X, N, K)
        Yb = logq.logq_linear(codes, cb, X, N, K)
    s.synchronize()
    assert torch.equal(Ya, Yb)                        # deterministic reduction order


def test_gemv_cuda_graph_capture(logq):
    N, K = 2048, 2048
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 1.5, 2)
    X = workloads.activations_torch(1, K, 2, torch.bfloat16, "cuda")
    Y = torch.empty(1, N, device="cuda")
    ws = logq.new_workspace()
    logq.logq_linear(codes, cb, X, N, K, Y=Y, workspace=ws)          # warm-up outside capture
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            logq.logq_linear(codes, cb, X, N, K, Y=Y, workspace=ws)
    Y.zero_()
    g.replay()
    torch.cuda.synchronize()
    Yr, A = reference(X, q, ocb)
    check_linear(Y.double().cpu().numpy(), Yr, A)


@pytest.mark.parametrize("N,K,B", [(256, 512, 128), (300, 1152, 200), (1024, 2048, 256), (512, 4096, 2048),
                                   (4096, 4096, 256), (200, 128, 17)])
@pytest.mark.parametrize("bits", [3, 4])
def test_prefill_bf16(logq, N, K, B, bits):
    run_case(logq, N, K, bits, B, torch.bfloat16, seed=N + B + bits)


@pytest.mark.parametrize("N,K,B,ydt", [(4096, 8192, 16, torch.bfloat16), (4100, 8192, 12, None),
                                       (4096, 14336, 16, torch.bfloat16), (4096, 8192, 9, torch.bfloat16)])
def test_small_batch_tensor_cores_split_k(logq, N, K, B, ydt):
    """4-bit batches of 9..16 on long-K shapes run on the tensor cores with each
    output tile's k range split over CTAs (fp32 partials, fixed-order sum) when the
    workspace has room; with the minimal workspace the same call keeps the
    CUDA-core kernel.  Both match the oracle; base 3 makes almost every code
    non-zero, so the two summation orders give different fp32 sums."""
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 3.0, N + B)
    X = workloads.activations_torch(B, K, N + K, torch.bfloat16, "cuda")
    wsb = logq.logq_linear_workspace_bytes(B, N, K, 4)
    assert wsb > logq.logq_workspace_bytes()
    Yt = logq.logq_linear(codes, cb, X, N, K, y_dtype=ydt, workspace=logq.new_workspace(nbytes=wsb))
    Yc = logq.logq_linear(codes, cb, X, N, K, y_dtype=ydt, workspace=logq.new_workspace())
    Yr, A = reference(X, q, ocb)
    name = "f32" if ydt is None else "bf16"
    check_linear(Yt.double().cpu().numpy(), Yr, A, name)
    check_linear(Yc.double().cpu().numpy(), Yr, A, name)
    assert not torch.equal(Yt, Yc)


def test_small_batch_tensor_cores_without_split(logq):
    """112 output tiles of 128 rows fill enough SMs without splitting the k range;
    the tensor cores beat the CUDA-core kernel at batch 16 here, workspace or not."""
    N, K, B = 14336, 2048, 16
    assert logq.logq_linear_workspace_bytes(B, N, K, 4) == logq.logq_workspace_bytes()
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 3.0, 77)
    X = workloads.activations_torch(B, K, 77, torch.bfloat16, "cuda")
    Y = logq.logq_linear(codes, cb, X, N, K, y_dtype=torch.bfloat16, workspace=logq.new_workspace())
    Yr, A = reference(X, q, ocb)
    check_linear(Y.double().cpu().numpy(), Yr, A, "bf16")


@pytest.mark.parametrize("bits,B", [(3, 8), (8, 16), (3, 5)])
def test_small_batch_3_and_8_bit_on_tensor_cores(logq, bits, B):
    """3- and 8-bit batches above 4 run on the tensor cores in 16-token tiles (split or not)."""
    run_case(logq, 2048, 2048, bits, B, torch.bfloat16, ydt=torch.bfloat16, seed=bits * 10 + B,
             base=1.25 if bits == 3 else 1.05)
    run_case(logq, 300, 1152, bits, B, torch.bfloat16, seed=bits + B, base=1.25 if bits == 3 else 1.05)


@pytest.mark.parametrize("N,K,B", [(1024, 4096, 64), (1000, 4096, 300), (200, 2048, 40)])
def test_prefill_split_k(logq, N, K, B):
    """Prefill shapes with too few output tiles split the k range (ragged N and B)."""
    assert logq.logq_linear_workspace_bytes(B, N, K, 4) > logq.logq_workspace_bytes()
    run_case(logq, N, K, 4, B, torch.bfloat16, ydt=torch.bfloat16, seed=N + B)


@pytest.mark.parametrize("bits,N,K,B,xdt", [(4, 1024, 4096, 64, torch.float16), (3, 1000, 2048, 40, torch.bfloat16),
                                            (8, 1024, 4096, 48, torch.bfloat16)])
def test_prefill_split_k_dtypes(logq, bits, N, K, B, xdt):
    """Split k ranges with fp16 activations and output, 3-bit groups and 8-bit codes."""
    assert logq.logq_linear_workspace_bytes(B, N, K, bits) > logq.logq_workspace_bytes()
    run_case(logq, N, K, bits, B, xdt, ydt=xdt, seed=N + B + bits, base=1.25 if bits == 3 else 1.5)


def test_grouped_split_k_equals_single_calls(logq):
    """A grouped call at batch 64 runs its three matrices in one tensor-core launch with
    every k range split in eight (the partial sums of each matrix after the previous
    one's in the workspace), as each single call splits its own: each output equals the
    single call's bit for bit and matches the oracle."""
    K, B = 4096, 64
    shapes = [(1024, 1.4), (512, 1.7), (512, 2.0)]
    layers = [make_layer(logq, N, K, 4, base, seed=90 + i) for i, (N, base) in enumerate(shapes)]
    X = workloads.activations_torch(B, K, 91, torch.bfloat16, "cuda")
    wsb = logq.logq_linear_grouped_workspace_bytes(B, [N for N, _ in shapes], K, 4)
    # one launch: partial sums of all three matrices, 8 ranges each
    assert wsb == logq.logq_workspace_bytes() + 8 * B * sum(N for N, _ in shapes) * 4
    ws = logq.new_workspace(nbytes=wsb)
    items = [(codes, cb, N, None) for (codes, cb, ocb, q), (N, _) in zip(layers, shapes)]
    outs = logq.logq_linear_grouped(items, X, K, y_dtype=torch.bfloat16, workspace=ws)
    for (codes, cb, ocb, q), (N, _), Y in zip(layers, shapes, outs):
        assert torch.equal(Y, logq.logq_linear(codes, cb, X, N, K, y_dtype=torch.bfloat16, workspace=ws))
        Yr, A = reference(X, q, ocb)
        check_linear(Y.double().cpu().numpy(), Yr, A, "bf16")
    st, detail = logq.logq_workspace_status(ws)
    assert st == logq.LOGQ_OK and detail == 0


@pytest.mark.parametrize("bits,B,shapes,K", [
    (4, 300, [(2000, 1.4), (500, 1.7), (520, 2.0)], 1024),      # q/k/v-like, ragged rows and tokens
    (4, 512, [(2048, 1.3), (512, 1.6)], 1024),
    (3, 96, [(640, 1.25), (256, 1.4)], 1152),
    (8, 200, [(384, 1.05), (136, 1.02), (64, 1.03), (256, 1.04)], 512),
    (4, 12, [(8192, 1.5), (8192, 1.8)], 4096),                   # gate/up-like, 16-token tiles
])
def test_grouped_tensor_core_launch(logq, bits, B, shapes, K):
    """Matrices sharing X in one tensor-core launch (each a share of the CTAs, its own
    table): every output matches the oracle, with and without room for split k ranges.
    Unsplit, above batch 16 (where a single call also runs on the tensor cores), each
    equals the single call's bit for bit (same tiles, same k order)."""
    layers = [make_layer(logq, N, K, bits, base, seed=110 + i) for i, (N, base) in enumerate(shapes)]
    X = workloads.activations_torch(B, K, 111, torch.bfloat16, "cuda")
    items = [(codes, cb, N, None) for (codes, cb, ocb, q), (N, _) in zip(layers, shapes)]
    outs = logq.logq_linear_grouped(items, X, K, y_dtype=torch.bfloat16)
    for (codes, cb, ocb, q), Y in zip(layers, outs):
        Yr, A = reference(X, q, ocb)
        check_linear(Y.double().cpu().numpy(), Yr, A, "bf16")
    ws = logq.new_workspace()
    outs1 = logq.logq_linear_grouped(items, X, K, y_dtype=torch.bfloat16, workspace=ws)
    for (codes, cb, ocb, q), (N, _), Y in zip(layers, shapes, outs1):
        if B > 16:
            assert torch.equal(Y, logq.logq_linear(codes, cb, X, N, K, y_dtype=torch.bfloat16, workspace=ws))
        else:
            Yr, A = reference(X, q, ocb)
            check_linear(Y.double().cpu().numpy(), Yr, A, "bf16")
    st, detail = logq.logq_workspace_status(ws)
    assert st == logq.LOGQ_OK and detail == 0


@pytest.mark.parametrize("ydt", [torch.bfloat16, None])
def test_prefill_output_dtypes_and_fp16(logq, ydt):
    run_case(logq, 512, 1024, 4, 256, torch.bfloat16, ydt=ydt, seed=5)
    run_case(logq, 512, 1024, 4, 256, torch.float16, ydt=None, seed=6)


def test_prefill_workspace_status_clean(logq):
    N, K, B = 1024, 2048, 512
    codes, cb, ocb, q = make_layer(logq, N, K, 4, 1.5, 9)
    ws = logq.new_workspace()
    X = workloads.activations_torch(B, K, 9, torch.bfloat16, "cuda")
    logq.logq_linear(codes, cb, X, N, K, workspace=ws)
    st, detail = logq.logq_workspace_status(ws)
    assert st == logq.LOGQ_OK and detail == 0


@pytest.mark.parametrize("B", [1, 4, 16, 256])
def test_grouped_matches_oracle(logq, B):
    """q/k/v-like group sharing X (each matrix its own codebook), with an L2 warm-up range."""
    K = 2048
    shapes = [(2048, 1.35), (512, 1.8), (512, 1.5)]
    layers = [make_layer(logq, N, K, 4, base, seed=70 + i) for i, (N, base) in enumerate(shapes)]
    X = workloads.activations_torch(B, K, 77, torch.bfloat16, "cuda")
    warm = torch.empty(3 << 20, dtype=torch.uint8, device="cuda")
    items = [(codes, cb, N, None) for (codes, cb, ocb, q), (N, _) in zip(layers, shapes)]
    outs = logq.logq_linear_grouped(items, X, K, prefetch=warm, prefetch_bytes=warm.numel())
    for (codes, cb, ocb, q), Y in zip(layers, outs):
        Yr, A = reference(X, q, ocb)
        check_linear(Y.double().cpu().numpy(), Yr, A)


@pytest.mark.parametrize("bits,B", [(3, 1), (3, 4), (4, 2)])
def test_grouped_two_items_equal_single_calls(logq, bits, B):
    K = 1152
    a = make_layer(logq, 700, K, bits, 1.3, seed=81)
    b = make_layer(logq, 300, K, bits, 1.7, seed=82)
    X = workloads.activations_torch(B, K, 83, torch.bfloat16, "cuda")
    ya, yb = logq.logq_linear_grouped([(a[0], a[1], 700, None), (b[0], b[1], 300, None)], X, K)
    assert torch.equal(ya, logq.logq_linear(a[0], a[1], X, 700, K))
    assert torch.equal(yb, logq.logq_linear(b[0], b[1], X, 300, K))


def test_grouped_rejects_bad_groups(logq):
    K = 256
    a = make_layer(logq, 64, K, 4, 1.5, seed=90)
    c = make_layer(logq, 64, K, 3, 1.5, seed=91)
    X = workloads.activations_torch(1, K, 92, torch.bfloat16, "cuda")
    with pytest.raises(logq.LogqError) as ei:
        logq.logq_linear_grouped([(a[0], a[1], 64, None), (c[0], c[1], 64, None)], X, K)
    assert ei.value.status == logq.LOGQ_ERR_INVALID_ARG
    with pytest.raises(logq.LogqError):
        logq.logq_linear_grouped([(a[0], a[1], 64, None)] * 5, X, K)
