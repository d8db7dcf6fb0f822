"""Host-side tests of the C ABI (no GPU needed): the library builds and loads,
exports every symbol that include/logq.h declares, builds the same codebooks
as the oracle, sizes buffers, and rejects invalid arguments before touching
the device."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="session")
def logq():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_01127_gb300 as m
    return m


def declared_symbols():
    src = open(os.path.join(ROOT, "include", "logq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(logq_[a-z0-9_]+)\s*\(", src)))


def test_exports_every_declared_symbol(logq):
    names = declared_symbols()
    assert len(names) >= 8
    for n in names:
        assert hasattr(logq.lib, n), n          # dlsym succeeds
    assert set(names) == set(logq.EXPORTED)


def test_struct_layout_matches_header(logq):
    # 4 int32 + 3 double + 256 float + 128 float + 2 x 256 uint16
    assert ctypes.sizeof(logq.Codebook) == 16 + 24 + 1024 + 512 + 1024


@pytest.mark.parametrize("bits,base", [(b, x) for b in (3, 4) for x in (1.2, 1.25, 1.5, 1.7351, 2.0)]
                         + [(8, x) for x in (1.02, 1.0473, 1.1)])
@pytest.mark.parametrize("rng_", [0.0173, 0.31, 1.0, 2.75])
@pytest.mark.parametrize("mode", [0, 1])
def test_codebook_matches_oracle(logq, bits, base, rng_, mode):
    cb = logq.logq_build_codebook(bits, base, rng_, mode)
    ocb = oracle.build_codebook(bits, base, rng_, mode)
    qmax = ocb.qmax
    half = 1 << (bits - 1)
    assert cb.bits == bits and cb.qmax == qmax and cb.flags == mode
    assert cb.base == base and cb.range == rng_
    assert math.isclose(cb.shift, ocb.shift, rel_tol=0, abs_tol=1e-12)
    lv = np.array(cb.level[: 2 * half], dtype=np.float32)
    np.testing.assert_array_equal(lv[:half], ocb.levels32)
    np.testing.assert_array_equal(lv[half:], -ocb.levels32)
    assert np.signbit(lv[half])                          # code 1 << (n-1) is -0.0
    np.testing.assert_array_equal(np.array(cb.thresh[:qmax], dtype=np.float32), ocb.taus32_up)
    assert all(math.isinf(t) for t in cb.thresh[qmax:])
    bf = np.array(cb.level_bf16[: 2 * half], dtype=np.uint16)
    f16 = np.array(cb.level_f16[: 2 * half], dtype=np.uint16)
    np.testing.assert_array_equal(bf[:half], ocb.levels_bf16_bits)
    np.testing.assert_array_equal(bf[half:], ocb.levels_bf16_bits | 0x8000)
    np.testing.assert_array_equal(f16[:half], ocb.levels_f16_bits)
    np.testing.assert_array_equal(f16[half:], ocb.levels_f16_bits | 0x8000)


@pytest.mark.parametrize("args", [(2, 1.5, 1.0, 0), (5, 1.5, 1.0, 0), (4, 1.0, 1.0, 0), (4, -2.0, 1.0, 0),
                                  (4, float("inf"), 1.0, 0), (4, 1.5, 0.0, 0), (4, 1.5, -3.0, 0),
                                  (4, 1.5, float("nan"), 0), (4, 1.5, 1.0, 2)])
def test_codebook_invalid(logq, args):
    with pytest.raises(logq.LogqError) as ei:
        logq.logq_build_codebook(*args)
    assert ei.value.status == logq.LOGQ_ERR_INVALID_ARG


def test_codebook_null_out(logq):
    assert logq.lib.logq_build_codebook(4, 1.5, 1.0, 0, None) == logq.LOGQ_ERR_INVALID_ARG


@pytest.mark.parametrize("N,K,bits,want", [(512, 2048, 4, 512 * 1024), (3, 128, 3, 3 * 48), (5, 256, 8, 5 * 256),
                                           (1, 128, 4, 64), (0, 128, 4, 0), (4, 100, 4, 0),
                                           (4, 0, 4, 0), (4, 128, 5, 0), (-1, 128, 4, 0),
                                           (14336, 4096, 3, 14336 * 1536)])
def test_packed_bytes(logq, N, K, bits, want):
    assert logq.logq_packed_bytes(N, K, bits) == want
    if want:
        assert want == N * oracle.packed_row_bytes(K, bits)


def test_workspace_bytes(logq):
    assert logq.logq_workspace_bytes() == 256


def test_linear_workspace_bytes(logq):
    """4-bit products that stay on the CUDA cores need only the base workspace
    (batches up to 7, and batches 8..16 where that kernel is estimated faster);
    tensor-core products whose output tiles are too few to fill the GPU ask for
    room for split-k partial sums (splits x B x N fp32); invalid sizes give 0."""
    base = logq.logq_workspace_bytes()
    assert logq.logq_linear_workspace_bytes(1, 4096, 4096, 4) == base
    assert logq.logq_linear_workspace_bytes(4, 14336, 4096, 4) == base
    assert logq.logq_linear_workspace_bytes(8, 4096, 14336, 4) == base
    assert logq.logq_linear_workspace_bytes(16, 4096, 4096, 4) == base
    for B, N, K, bits in [(16, 4096, 8192, 4), (16, 4096, 14336, 4), (64, 1024, 4096, 4), (12, 2048, 2048, 3)]:
        extra = logq.logq_linear_workspace_bytes(B, N, K, bits) - base
        assert extra > 0 and extra % (B * N * 4) == 0, (B, N, K, bits, extra)
        splits = extra // (B * N * 4)
        assert 2 <= splits <= K // 64 // 8
    assert logq.logq_linear_workspace_bytes(0, 4096, 4096, 4) == 0
    assert logq.logq_linear_workspace_bytes(16, 4096, 100, 4) == 0


def test_linear_grouped_workspace_bytes(logq):
    """A group that runs as one tensor-core launch asks for the partial sums of all its
    matrices (splits x B x sum(N) fp32), one that runs on the CUDA cores or unsplit only
    for the base workspace; a single matrix asks what logq_linear asks; invalid groups
    give 0."""
    base = logq.logq_workspace_bytes()
    g = logq.logq_linear_grouped_workspace_bytes
    assert g(64, [1024, 512, 512], 4096, 4) == base + 8 * 64 * 2048 * 4
    assert g(2048, [4096, 1024, 1024], 4096, 4) == base        # one unsplit launch fills the GPU
    assert g(4, [4096, 1024, 1024], 4096, 4) == base
    assert g(1, [14336, 14336], 4096, 4) == base
    # 3-bit group at batch 96: one launch, every k range split in two
    assert g(96, [640, 256], 1152, 3) == base + 2 * 96 * 896 * 4
    # q/k/v at batch 16: the tensor-core group with k split in three beats the
    # CUDA-core group launch and the single calls
    assert g(16, [4096, 1024, 1024], 4096, 4) == base + 3 * 16 * 6144 * 4
    for B, N, K, bits in [(16, 4096, 8192, 4), (64, 1024, 4096, 4), (2048, 1024, 4096, 4), (1, 4096, 4096, 4)]:
        assert g(B, [N], K, bits) == logq.logq_linear_workspace_bytes(B, N, K, bits)
    assert g(64, [], 4096, 4) == 0
    assert g(64, [64] * 5, 4096, 4) == 0
    assert g(64, [64, 64], 100, 4) == 0
    assert g(0, [64], 4096, 4) == 0


def test_status_strings(logq):
    for s in range(7):
        assert len(logq.status_string(s)) >= 2
    assert logq.status_string(99) == "unknown status"


def _fake(addr):
    return ctypes.c_void_p(addr)


def test_quantize_rejects_before_launch(logq):
    """Invalid requests fail in host validation (these run without a GPU:
    nothing is enqueued, so the fake device addresses are never touched)."""
    L = logq.lib
    W, C, ws = _fake(0x10000), _fake(0x20000), _fake(0x30000)
    cb = logq.Codebook()
    ok_args = dict(N=4, K=128, bits=4, base=1.5, rng=1.0, flags=0)

    def call(W=W, C=C, ws=ws, wsb=256, **kw):
        a = dict(ok_args, **kw)
        return L.logq_quantize(W, a["N"], a["K"], a["bits"], a["base"], a["rng"], a["flags"], C,
                               ctypes.byref(cb), ws, wsb, None)

    assert call(W=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(C=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(W=_fake(0x10004)) == logq.LOGQ_ERR_INVALID_ARG          # misaligned
    assert call(K=100) == logq.LOGQ_ERR_INVALID_ARG
    assert call(N=0) == logq.LOGQ_ERR_INVALID_ARG
    assert call(bits=5) == logq.LOGQ_ERR_INVALID_ARG
    assert call(base=1.0) == logq.LOGQ_ERR_INVALID_ARG
    assert call(base=float("nan")) == logq.LOGQ_ERR_INVALID_ARG
    assert call(rng=float("inf")) == logq.LOGQ_ERR_INVALID_ARG
    assert call(flags=7) == logq.LOGQ_ERR_INVALID_ARG
    assert call(ws=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(wsb=16) == logq.LOGQ_ERR_WORKSPACE
    assert call(ws=_fake(0x30008)) == logq.LOGQ_ERR_WORKSPACE


def test_energy_quantize_rejects_before_launch(logq):
    """logq_quantize_energy validates eps, sizes, workspace and scratch on the
    host before anything is enqueued (fake device addresses, no GPU)."""
    L = logq.lib
    W, C, ws, sc = _fake(0x10000), _fake(0x20000), _fake(0x30000), _fake(0x40000)
    cb = logq.Codebook()
    wmin = ctypes.c_double(0.0)
    scb = L.logq_energy_scratch_bytes()
    assert 16 * 1024 < scb < 128 * 1024

    def call(W=W, C=C, ws=ws, wsb=256, sc=sc, scb=scb, N=4, K=128, bits=4, eps=4e-3, flags=0):
        return L.logq_quantize_energy(W, N, K, bits, eps, flags, C, ctypes.byref(cb), ctypes.byref(wmin),
                                      ws, wsb, sc, scb, None)

    assert call(W=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(C=_fake(0x20008)) == logq.LOGQ_ERR_INVALID_ARG         # misaligned
    assert call(K=100) == logq.LOGQ_ERR_INVALID_ARG
    assert call(bits=2) == logq.LOGQ_ERR_INVALID_ARG
    for eps in (0.0, -1e-3, 1.0000001, float("nan"), float("inf")):
        assert call(eps=eps) == logq.LOGQ_ERR_INVALID_ARG
    assert call(flags=3) == logq.LOGQ_ERR_INVALID_ARG
    assert call(ws=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(sc=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(scb=scb - 8) == logq.LOGQ_ERR_WORKSPACE
    assert call(sc=_fake(0x40004)) == logq.LOGQ_ERR_WORKSPACE


def test_gptq_rejects_before_launch(logq):
    """logq_gptq validates sizes, codebook and scratch before anything is enqueued."""
    L = logq.lib
    W, U, C, sc = _fake(0x10000), _fake(0x20000), _fake(0x30000), _fake(0x40000)
    cb4 = logq.logq_build_codebook(4, 1.5, 1.0)
    cb3 = logq.logq_build_codebook(3, 1.5, 1.0)
    scb = L.logq_gptq_scratch_bytes(64, 256)
    assert scb == (64 * 256 + 64 * 128) * 4
    assert L.logq_gptq_scratch_bytes(64, 100) == 0

    def call(W=W, U=U, cb=cb4, C=C, sc=sc, scb=scb, N=64, K=256):
        return L.logq_gptq(W, N, K, U, None, ctypes.byref(cb), C, sc, scb, None)

    assert call(W=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(U=_fake(0x20004)) == logq.LOGQ_ERR_INVALID_ARG
    assert call(K=100) == logq.LOGQ_ERR_INVALID_ARG
    assert call(cb=cb3) == logq.LOGQ_ERR_UNSUPPORTED
    assert call(sc=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(scb=scb - 16) == logq.LOGQ_ERR_WORKSPACE


def test_gptq_factor_rejects_before_launch(logq):
    """logq_gptq_factor validates sizes, damping and scratch before anything is enqueued."""
    L = logq.lib
    H, U, sc = _fake(0x10000), _fake(0x20000), _fake(0x40000)
    scb = L.logq_gptq_factor_scratch_bytes(256)
    assert scb == 256 + (256 * 256 + 256 * 256 // 4) * 4
    assert L.logq_gptq_factor_scratch_bytes(100) == 0
    assert L.logq_gptq_factor_scratch_bytes(0) == 0

    def call(H=H, K=256, damp=0.01, U=U, sc=sc, scb=scb):
        return L.logq_gptq_factor(H, K, damp, U, None, sc, scb, None)

    assert call(H=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(U=_fake(0x20004)) == logq.LOGQ_ERR_INVALID_ARG
    assert call(K=100) == logq.LOGQ_ERR_INVALID_ARG
    assert call(K=-128) == logq.LOGQ_ERR_INVALID_ARG
    for damp in (-0.01, float("nan"), float("inf")):
        assert call(damp=damp) == logq.LOGQ_ERR_INVALID_ARG
    assert call(sc=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(scb=scb - 4) == logq.LOGQ_ERR_WORKSPACE
    assert logq.status_string(logq.LOGQ_ERR_NOT_PD) == "damped Hessian is not positive definite"


def test_linear_rejects_before_launch(logq):
    L = logq.lib
    cb = logq.logq_build_codebook(4, 1.5, 1.0)
    C, X, Y, ws = _fake(0x10000), _fake(0x20000), _fake(0x30000), _fake(0x40000)

    def call(C=C, cbp=ctypes.byref(cb), X=X, xd=logq.LOGQ_BF16, B=1, N=8, K=128, Y=Y,
             yd=logq.LOGQ_F32, ws=ws, wsb=256):
        return L.logq_linear(C, cbp, X, xd, B, N, K, Y, yd, ws, wsb, None)

    assert call(C=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(cbp=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(X=None) == logq.LOGQ_ERR_INVALID_ARG
    assert call(Y=_fake(0x30002)) == logq.LOGQ_ERR_INVALID_ARG
    assert call(B=0) == logq.LOGQ_ERR_INVALID_ARG
    assert call(K=96) == logq.LOGQ_ERR_INVALID_ARG
    assert call(N=-2) == logq.LOGQ_ERR_INVALID_ARG
    assert call(xd=logq.LOGQ_F32) == logq.LOGQ_ERR_UNSUPPORTED
    assert call(xd=logq.LOGQ_BF16, yd=logq.LOGQ_F16) == logq.LOGQ_ERR_UNSUPPORTED
    assert call(ws=None) == logq.LOGQ_ERR_WORKSPACE
    assert call(wsb=255) == logq.LOGQ_ERR_WORKSPACE
    bad = logq.logq_build_codebook(4, 1.5, 1.0)
    bad.qmax = 3                                                     # inconsistent codebook
    assert call(cbp=ctypes.byref(bad)) == logq.LOGQ_ERR_INVALID_ARG


def test_workspace_status_rejects_null(logq):
    assert logq.lib.logq_workspace_status(None, None, None) == logq.LOGQ_ERR_WORKSPACE
