"""Python binding of liblogq, the GB300 (sm_103a) Log_bQuant inference library.

Argument marshalling only: every step of the quantise / dequantise-and-multiply
path runs in the CUDA kernels of ``liblogq.so`` behind the C ABI declared in
``include/logq.h``.  PyTorch provides device memory and the current stream.
The functions carry the C names:

  logq_build_codebook(bits, base, range, flags)          -> Codebook
  logq_packed_bytes(N, K, bits)                         -> int
  logq_workspace_bytes()                                -> int
  logq_quantize(W, bits, base, range, flags, ...)       -> (codes, Codebook)
  logq_linear(codes, cb, X, N, K, y_dtype, ...)         -> Y
  logq_workspace_status(workspace)                      -> (status, detail)
  logq_status_string(status), logq_device_sm_count()

There is no CPU fallback: the first call raises ImportError when the library
is not built (importing the package alone, e.g. for ``workloads``, does not
load it).
"""
from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "liblogq.so")

LOGQ_OK = 0
LOGQ_ERR_INVALID_ARG = 1
LOGQ_ERR_NONFINITE = 2
LOGQ_ERR_UNSUPPORTED = 3
LOGQ_ERR_CUDA = 4
LOGQ_ERR_WORKSPACE = 5
LOGQ_ERR_TIMEOUT = 6
LOGQ_ERR_NOT_PD = 7

LOGQ_F32, LOGQ_BF16, LOGQ_F16 = 0, 1, 2
LOGQ_SHIFT_EXACT, LOGQ_SHIFT_FLOOR = 0, 1

EXPORTED = ("logq_build_codebook", "logq_packed_bytes", "logq_workspace_bytes", "logq_linear_workspace_bytes",
            "logq_linear_grouped_workspace_bytes", "logq_quantize",
            "logq_linear", "logq_workspace_status", "logq_status_string", "logq_device_sm_count",
            "logq_quantize_noalloc", "logq_linear_grouped", "logq_energy_scratch_bytes",
            "logq_quantize_energy", "logq_gptq_factor_scratch_bytes", "logq_gptq_factor",
            "logq_gptq_scratch_bytes", "logq_gptq")


class Codebook(ctypes.Structure):
    """Mirror of ``logq_codebook`` (include/logq.h)."""
    _fields_ = [
        ("bits", ctypes.c_int32),
        ("qmax", ctypes.c_int32),
        ("flags", ctypes.c_int32),
        ("_pad", ctypes.c_int32),
        ("base", ctypes.c_double),
        ("shift", ctypes.c_double),
        ("range", ctypes.c_double),
        ("level", ctypes.c_float * 256),
        ("thresh", ctypes.c_float * 128),
        ("level_bf16", ctypes.c_uint16 * 256),
        ("level_f16", ctypes.c_uint16 * 256),
    ]


class LinearItem(ctypes.Structure):
    """Mirror of ``logq_linear_item`` (include/logq.h)."""
    _fields_ = [
        ("codes", ctypes.c_void_p),
        ("cb", ctypes.POINTER(Codebook)),
        ("N", ctypes.c_int64),
        ("Y", ctypes.c_void_p),
    ]


class LogqError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"liblogq.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    c_i64, c_int, c_dbl, P = ctypes.c_int64, ctypes.c_int, ctypes.c_double, ctypes.c_void_p
    lib.logq_build_codebook.argtypes = [c_int, c_dbl, c_dbl, c_int, ctypes.POINTER(Codebook)]
    lib.logq_build_codebook.restype = c_int
    lib.logq_packed_bytes.argtypes = [c_i64, c_i64, c_int]
    lib.logq_packed_bytes.restype = ctypes.c_size_t
    lib.logq_workspace_bytes.argtypes = []
    lib.logq_workspace_bytes.restype = ctypes.c_size_t
    lib.logq_linear_workspace_bytes.argtypes = [c_i64, c_i64, c_i64, c_int]
    lib.logq_linear_workspace_bytes.restype = ctypes.c_size_t
    lib.logq_linear_grouped_workspace_bytes.argtypes = [c_i64, ctypes.POINTER(c_i64), c_int, c_i64, c_int]
    lib.logq_linear_grouped_workspace_bytes.restype = ctypes.c_size_t
    lib.logq_quantize.argtypes = [P, c_i64, c_i64, c_int, c_dbl, c_dbl, c_int, P,
                                  ctypes.POINTER(Codebook), P, ctypes.c_size_t, P]
    lib.logq_quantize.restype = c_int
    lib.logq_quantize_noalloc.argtypes = [P, c_i64, c_i64, c_int, c_dbl, c_dbl, c_int, P,
                                          ctypes.POINTER(Codebook), P]
    lib.logq_quantize_noalloc.restype = c_int
    lib.logq_energy_scratch_bytes.argtypes = []
    lib.logq_energy_scratch_bytes.restype = ctypes.c_size_t
    lib.logq_quantize_energy.argtypes = [P, c_i64, c_i64, c_int, c_dbl, c_int, P, ctypes.POINTER(Codebook),
                                         ctypes.POINTER(c_dbl), P, ctypes.c_size_t, P, ctypes.c_size_t, P]
    lib.logq_quantize_energy.restype = c_int
    lib.logq_gptq_scratch_bytes.argtypes = [c_i64, c_i64]
    lib.logq_gptq_scratch_bytes.restype = ctypes.c_size_t
    lib.logq_gptq_factor_scratch_bytes.argtypes = [c_i64]
    lib.logq_gptq_factor_scratch_bytes.restype = ctypes.c_size_t
    lib.logq_gptq_factor.argtypes = [P, c_i64, c_dbl, P, P, P, ctypes.c_size_t, P]
    lib.logq_gptq_factor.restype = c_int
    lib.logq_gptq.argtypes = [P, c_i64, c_i64, P, P, ctypes.POINTER(Codebook), P, P, ctypes.c_size_t, P]
    lib.logq_gptq.restype = c_int
    lib.logq_linear.argtypes = [P, ctypes.POINTER(Codebook), P, c_int, c_i64, c_i64, c_i64, P,
                                c_int, P, ctypes.c_size_t, P]
    lib.logq_linear.restype = c_int
    lib.logq_linear_grouped.argtypes = [ctypes.POINTER(LinearItem), c_int, P, c_int, c_i64, c_i64, c_int,
                                        P, ctypes.c_size_t, P, ctypes.c_size_t, P]
    lib.logq_linear_grouped.restype = c_int
    lib.logq_workspace_status.argtypes = [P, P, ctypes.POINTER(ctypes.c_uint32)]
    lib.logq_workspace_status.restype = c_int
    lib.logq_status_string.argtypes = [c_int]
    lib.logq_status_string.restype = ctypes.c_char_p
    lib.logq_device_sm_count.argtypes = []
    lib.logq_device_sm_count.restype = c_int
    return lib


_LIB = None


def _lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        _LIB = _load()
    return _LIB


def __getattr__(name):
    if name == "lib":
        return _lib()
    raise AttributeError(name)


def status_string(status: int) -> str:
    return _lib().logq_status_string(int(status)).decode()


logq_status_string = status_string


def _check(status: int, where: str) -> None:
    if status != LOGQ_OK:
        raise LogqError(status, where)


def _stream_ptr(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(dt) -> int:
    import torch
    return {torch.float32: LOGQ_F32, torch.bfloat16: LOGQ_BF16, torch.float16: LOGQ_F16}[dt]


def _torch_dtype(code: int):
    import torch
    return {LOGQ_F32: torch.float32, LOGQ_BF16: torch.bfloat16, LOGQ_F16: torch.float16}[code]


def logq_build_codebook(bits: int, base: float, range_: float, flags: int = LOGQ_SHIFT_EXACT) -> Codebook:
    cb = Codebook()
    _check(_lib().logq_build_codebook(int(bits), float(base), float(range_), int(flags), ctypes.byref(cb)),
           "logq_build_codebook")
    return cb


def logq_packed_bytes(N: int, K: int, bits: int) -> int:
    return int(_lib().logq_packed_bytes(int(N), int(K), int(bits)))


def logq_workspace_bytes() -> int:
    return int(_lib().logq_workspace_bytes())


def logq_linear_workspace_bytes(B: int, N: int, K: int, bits: int) -> int:
    return int(_lib().logq_linear_workspace_bytes(int(B), int(N), int(K), int(bits)))


def logq_linear_grouped_workspace_bytes(B: int, Ns, K: int, bits: int) -> int:
    arr = (ctypes.c_int64 * len(Ns))(*[int(n) for n in Ns])
    return int(_lib().logq_linear_grouped_workspace_bytes(int(B), arr, len(Ns), int(K), int(bits)))


def new_workspace(device=None, nbytes: int | None = None):
    """Zero-filled device workspace: logq_workspace_bytes() bytes, or nbytes (at
    least that) -- e.g. the largest logq_linear_workspace_bytes() of the
    products it will serve, so that tensor-core launches may split k ranges."""
    import torch
    n = logq_workspace_bytes() if nbytes is None else max(int(nbytes), logq_workspace_bytes())
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def logq_quantize(W, bits: int, base: float, range_: float = 0.0, flags: int = LOGQ_SHIFT_EXACT,
                  codes=None, workspace=None, stream=None):
    """Quantise fp32 device weights W[N, K]; returns (codes uint8 tensor, Codebook)."""
    import torch
    assert W.dtype == torch.float32 and W.is_cuda and W.dim() == 2 and W.is_contiguous()
    N, K = W.shape
    nbytes = logq_packed_bytes(N, K, bits)
    if codes is None:
        codes = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=W.device)
    if workspace is None:
        workspace = new_workspace(W.device)
    cb = Codebook()
    st = _lib().logq_quantize(ctypes.c_void_p(W.data_ptr()), N, K, int(bits), float(base), float(range_),
                           int(flags), ctypes.c_void_p(codes.data_ptr()), ctypes.byref(cb),
                           ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_ptr(stream))
    _check(st, "logq_quantize")
    return codes[:nbytes], cb


def logq_quantize_noalloc(W, bits: int, base: float, range_: float = 0.0,
                          flags: int = LOGQ_SHIFT_EXACT, codes=None, stream=None):
    """logq_quantize without a caller workspace (static device scratch; see logq.h)."""
    import torch
    assert W.dtype == torch.float32 and W.is_cuda and W.dim() == 2 and W.is_contiguous()
    N, K = W.shape
    nbytes = logq_packed_bytes(N, K, bits)
    if codes is None:
        codes = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=W.device)
    cb = Codebook()
    st = _lib().logq_quantize_noalloc(ctypes.c_void_p(W.data_ptr()), N, K, int(bits), float(base),
                                      float(range_), int(flags), ctypes.c_void_p(codes.data_ptr()),
                                      ctypes.byref(cb), _stream_ptr(stream))
    _check(st, "logq_quantize_noalloc")
    return codes[:nbytes], cb


def logq_energy_scratch_bytes() -> int:
    return int(_lib().logq_energy_scratch_bytes())


def logq_quantize_energy(W, bits: int, eps: float = 4e-3, flags: int = LOGQ_SHIFT_EXACT, codes=None,
                         workspace=None, scratch=None, stream=None):
    """Self-calibrating quantisation (Sec. 3.2, Eqs. (3)-(5)): w_max = max|W|, w_min from the
    energy share eps, b = (w_max / w_min)^(1 / q_max).  Returns (codes, Codebook, w_min)."""
    import torch
    assert W.dtype == torch.float32 and W.is_cuda and W.dim() == 2 and W.is_contiguous()
    N, K = W.shape
    nbytes = logq_packed_bytes(N, K, bits)
    if codes is None:
        codes = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=W.device)
    if workspace is None:
        workspace = new_workspace(W.device)
    if scratch is None:
        scratch = torch.empty(logq_energy_scratch_bytes(), dtype=torch.uint8, device=W.device)
    cb = Codebook()
    wmin = ctypes.c_double(0.0)
    st = _lib().logq_quantize_energy(ctypes.c_void_p(W.data_ptr()), N, K, int(bits), float(eps), int(flags),
                                     ctypes.c_void_p(codes.data_ptr()), ctypes.byref(cb), ctypes.byref(wmin),
                                     ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                     ctypes.c_void_p(scratch.data_ptr()), scratch.numel(), _stream_ptr(stream))
    _check(st, "logq_quantize_energy")
    return codes[:nbytes], cb, wmin.value


def gptq_factor(H, damp: float = 0.01, U=None, dead=None, scratch=None, stream=None):
    """U (fp32, upper) with Hd^-1 = U^T U, Hd = H + damp * mean(diag H) * I, and the
    mask of inputs whose Hessian diagonal is zero, computed by logq_gptq_factor from
    an fp32 device Hessian H[K, K].  Returns (U, dead)."""
    import torch
    assert H.dtype == torch.float32 and H.is_cuda and H.dim() == 2 and H.is_contiguous()
    assert H.shape[0] == H.shape[1], "H must be square"
    K = H.shape[0]
    if U is None:
        U = torch.empty(K, K, dtype=torch.float32, device=H.device)
    if dead is None:
        dead = torch.empty(K, dtype=torch.uint8, device=H.device)
    if scratch is None:
        scratch = torch.empty(int(_lib().logq_gptq_factor_scratch_bytes(K)), dtype=torch.uint8, device=H.device)
    st = _lib().logq_gptq_factor(ctypes.c_void_p(H.data_ptr()), K, float(damp), ctypes.c_void_p(U.data_ptr()),
                                 ctypes.c_void_p(dead.data_ptr()), ctypes.c_void_p(scratch.data_ptr()),
                                 scratch.numel(), _stream_ptr(stream))
    _check(st, "logq_gptq_factor")
    return U, dead


def logq_gptq(W, H, cb: Codebook, damp: float = 0.01, codes=None, scratch=None, stream=None):
    """GPTQ with the Log_b quantiser: fp32 device weights W[N, K], the layer's fp32
    device Hessian H[K, K] (e.g. 2 X^T X of calibration inputs) and a codebook;
    returns the packed codes.  The factor (logq_gptq_factor), the column loop and
    the compensations all run in the library's kernels."""
    import torch
    assert W.dtype == torch.float32 and W.is_cuda and W.dim() == 2 and W.is_contiguous()
    N, K = W.shape
    assert tuple(H.shape) == (K, K), "H must be K x K for W of K columns"
    U, dead = gptq_factor(H, damp, stream=stream)
    nbytes = logq_packed_bytes(N, K, cb.bits)
    if codes is None:
        codes = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=W.device)
    if scratch is None:
        scratch = torch.empty(int(_lib().logq_gptq_scratch_bytes(N, K)), dtype=torch.uint8, device=W.device)
    st = _lib().logq_gptq(ctypes.c_void_p(W.data_ptr()), N, K, ctypes.c_void_p(U.data_ptr()),
                          ctypes.c_void_p(dead.data_ptr()), ctypes.byref(cb), ctypes.c_void_p(codes.data_ptr()),
                          ctypes.c_void_p(scratch.data_ptr()), scratch.numel(), _stream_ptr(stream))
    _check(st, "logq_gptq")
    if stream is not None:          # the temporaries above belong to the current stream
        stream.synchronize()
    return codes[:nbytes]


def logq_linear(codes, cb: Codebook, X, N: int, K: int, y_dtype=None, Y=None, workspace=None,
                stream=None):
    """Y[B, N] = X[B, K] @ What^T through the codebook's 16-bit table of X's dtype."""
    import torch
    assert X.is_cuda and X.dim() == 2 and X.is_contiguous() and X.shape[1] == K
    B = X.shape[0]
    xd = _dtype_code(X.dtype)
    yd = LOGQ_F32 if y_dtype is None else (_dtype_code(y_dtype) if not isinstance(y_dtype, int) else y_dtype)
    if Y is None:
        Y = torch.empty((B, N), dtype=_torch_dtype(yd), device=X.device)
    assert Y.dtype == _torch_dtype(yd) and Y.is_contiguous() and Y.numel() == B * N, \
        "Y must be a contiguous [B, N] tensor of the output dtype"
    if workspace is None:
        workspace = new_workspace(X.device, logq_linear_workspace_bytes(B, N, K, cb.bits))
    st = _lib().logq_linear(ctypes.c_void_p(codes.data_ptr()), ctypes.byref(cb), ctypes.c_void_p(X.data_ptr()),
                         xd, B, int(N), int(K), ctypes.c_void_p(Y.data_ptr()), yd,
                         ctypes.c_void_p(workspace.data_ptr()), workspace.numel(), _stream_ptr(stream))
    _check(st, "logq_linear")
    return Y


def logq_linear_grouped(items, X, K: int, y_dtype=None, workspace=None, prefetch=None,
                        prefetch_bytes: int = 0, stream=None):
    """Up to four matrices sharing X in one launch: items = [(codes, cb, N, Y or None), ...].
    prefetch: optional device tensor (or (tensor, bytes)) the call warms L2 with.
    Returns the list of outputs."""
    import torch
    assert X.is_cuda and X.dim() == 2 and X.is_contiguous() and X.shape[1] == K
    B = X.shape[0]
    xd = _dtype_code(X.dtype)
    yd = LOGQ_F32 if y_dtype is None else (_dtype_code(y_dtype) if not isinstance(y_dtype, int) else y_dtype)
    arr = (LinearItem * len(items))()
    outs = []
    keep = []
    for i, (codes, cb, N, Y) in enumerate(items):
        if Y is None:
            Y = torch.empty((B, N), dtype=_torch_dtype(yd), device=X.device)
        assert Y.dtype == _torch_dtype(yd) and Y.is_contiguous() and Y.numel() == B * N, \
            "Y must be a contiguous [B, N] tensor of the output dtype"
        outs.append(Y)
        keep.append(cb)
        arr[i] = LinearItem(ctypes.c_void_p(codes.data_ptr()), ctypes.pointer(cb), int(N),
                            ctypes.c_void_p(Y.data_ptr()))
    if workspace is None:
        workspace = new_workspace(X.device, logq_linear_grouped_workspace_bytes(
            B, [int(N) for _, _, N, _ in items], K, items[0][1].bits))
    pf_ptr = ctypes.c_void_p(prefetch.data_ptr()) if prefetch is not None else None
    pf_bytes = int(prefetch_bytes) if prefetch is not None else 0
    st = _lib().logq_linear_grouped(arr, len(items), ctypes.c_void_p(X.data_ptr()), xd, B, int(K), yd, pf_ptr,
                                    pf_bytes, ctypes.c_void_p(workspace.data_ptr()), workspace.numel(),
                                    _stream_ptr(stream))
    _check(st, "logq_linear_grouped")
    return outs


def logq_workspace_status(workspace, stream=None):
    detail = ctypes.c_uint32(0)
    st = _lib().logq_workspace_status(ctypes.c_void_p(workspace.data_ptr()), _stream_ptr(stream),
                                   ctypes.byref(detail))
    return st, detail.value


def logq_device_sm_count() -> int:
    return int(_lib().logq_device_sm_count())
