"""Log_bQuant reference oracle -- TEST INFRASTRUCTURE ONLY.

Python access (ctypes + numpy) to ``logq_oracle.c``, a plain fp64 CPU
restatement of the paper's quantiser (Eq. (1)), dequantiser (Eq. (2)),
range/base heuristics (Eqs. (3)-(5)) and the dequantised linear layer.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never does, and
this package imports nothing from the library: the two share only the
seeded input generators, which hold none of the method's arithmetic.

Parity status of each function (what pins it is in ``tests/test_oracle.py``):
  build_codebook       pinned (closed forms, symmetry, monotonicity, fp32/bf16/fp16
                        rounding against library casts)
  quantize_*           pinned (three independent routes, level round trip,
                        idempotence, sign symmetry, base-2 frexp route)
  pack / unpack        pinned for the value set; the bit layout itself is a
                        choice of this library ("parity unpinned" for the layout)
  dequant              pinned through the codebook tables
  linear               pinned (float64 matmul of the dequantised weights,
                        one-hot and zero inputs)
  energy_wmin          pinned (brute force over all candidate thresholds)
  gptq_factor          pinned (upper triangular, positive diagonal and U^T U Hd = I,
                        which fix the Cholesky factor uniquely; a decoupled dead input)
  gptq                 pinned (diagonal Hessian = plain rounding; every compensated
                        value equals the least-squares minimiser given the columns
                        already quantised, solved directly; a dead input = the
                        reduced problem)
  base_from_range      pinned (closed form: q_max log steps span the range)
  linear_asym          pinned (brute-force nearest of all 2^n grid values, uniform
                        spacing, error bound, idempotence on its own grid, the
                        scale^2 / 12 mean square error of uniform inputs); the
                        comparison quantiser of the error study only, not part of the
                        method
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "logq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liblogq_oracle.so")
_lock = threading.Lock()
_lib = None

SHIFT_EXACT = 0
SHIFT_FLOOR = 1
TABLE_F64, TABLE_F32, TABLE_BF16, TABLE_F16 = 0, 1, 2, 3


class Codebook(ctypes.Structure):
    _fields_ = [
        ("bits", ctypes.c_int32),
        ("qmax", ctypes.c_int32),
        ("shift_mode", ctypes.c_int32),
        ("_pad", ctypes.c_int32),
        ("base", ctypes.c_double),
        ("range", ctypes.c_double),
        ("shift", ctypes.c_double),
        ("level", ctypes.c_double * 128),
        ("tau", ctypes.c_double * 128),
        ("level32", ctypes.c_float * 128),
        ("tau32_up", ctypes.c_float * 128),
        ("level_bf16", ctypes.c_uint16 * 128),
        ("level_f16", ctypes.c_uint16 * 128),
    ]

    @property
    def levels(self):
        return np.array(self.level[: self.qmax + 1], dtype=np.float64)

    @property
    def taus(self):
        return np.array(self.tau[: self.qmax], dtype=np.float64)

    @property
    def levels32(self):
        return np.array(self.level32[: self.qmax + 1], dtype=np.float32)

    @property
    def taus32_up(self):
        return np.array(self.tau32_up[: self.qmax], dtype=np.float32)

    @property
    def levels_bf16_bits(self):
        return np.array(self.level_bf16[: self.qmax + 1], dtype=np.uint16)

    @property
    def levels_f16_bits(self):
        return np.array(self.level_f16[: self.qmax + 1], dtype=np.uint16)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available) into oracle/_build."""
    with _lock:
        if not force and os.path.exists(_LIB_PATH) and \
                os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
            return _LIB_PATH
        os.makedirs(_BUILD, exist_ok=True)
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        base = ["gcc", "-O2", "-fPIC", "-shared", "-std=c11", "-fno-fast-math",
                "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
        try:
            subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                           capture_output=True)
        except subprocess.CalledProcessError:
            subprocess.run(base, check=True, capture_output=True)
        os.replace(tmp, _LIB_PATH)
        return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    c_i64, c_int, c_dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_double
    P = ctypes.c_void_p
    lib.oracle_build_codebook.argtypes = [c_int, c_dbl, c_dbl, c_int, ctypes.POINTER(Codebook)]
    lib.oracle_build_codebook.restype = c_int
    for name in ("oracle_quantize_log", "oracle_quantize_argmin", "oracle_quantize_thresh"):
        getattr(lib, name).argtypes = [P, c_i64, ctypes.POINTER(Codebook), P]
        getattr(lib, name).restype = None
    lib.oracle_absmax.argtypes = [P, c_i64, ctypes.POINTER(c_int)]
    lib.oracle_absmax.restype = c_dbl
    lib.oracle_pack.argtypes = [P, c_i64, c_i64, c_int, P]
    lib.oracle_pack.restype = c_int
    lib.oracle_unpack.argtypes = [P, c_i64, c_i64, c_int, P]
    lib.oracle_unpack.restype = c_int
    lib.oracle_packed_row_bytes.argtypes = [c_i64, c_int]
    lib.oracle_packed_row_bytes.restype = c_i64
    lib.oracle_dequant.argtypes = [P, c_i64, ctypes.POINTER(Codebook), c_int, P]
    lib.oracle_dequant.restype = None
    lib.oracle_linear.argtypes = [P, c_i64, P, c_i64, c_i64, P, P, c_int]
    lib.oracle_linear.restype = None
    lib.oracle_linear_sampled.argtypes = [P, c_i64, P, c_int, ctypes.POINTER(Codebook), c_int,
                                          P, P, c_i64, P, P, c_int]
    lib.oracle_linear_sampled.restype = None
    for name in ("oracle_round_f32", "oracle_round_bf16", "oracle_round_f16"):
        getattr(lib, name).argtypes = [c_dbl]
        getattr(lib, name).restype = c_dbl
    for name in ("oracle_bf16_bits", "oracle_f16_bits"):
        getattr(lib, name).argtypes = [c_dbl]
        getattr(lib, name).restype = ctypes.c_uint16
    lib.oracle_energy_wmin.argtypes = [P, c_i64, c_dbl]
    lib.oracle_energy_wmin.restype = c_dbl
    lib.oracle_base_from_range.argtypes = [c_dbl, c_dbl, c_int]
    lib.oracle_base_from_range.restype = c_dbl
    lib.oracle_gptq.argtypes = [P, c_i64, c_i64, P, c_dbl, ctypes.POINTER(Codebook), P, P]
    lib.oracle_gptq.restype = c_int
    lib.oracle_gptq_factor.argtypes = [P, c_i64, c_dbl, P]
    lib.oracle_gptq_factor.restype = c_int
    _lib = lib
    return lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f32(w) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(w, dtype=np.float32))


def build_codebook(bits: int, base: float, range_: float, shift_mode: int = SHIFT_EXACT) -> Codebook:
    """Codebook of Sec. 3.1 (levels by Eq. (2), shift by Eq. (4) or its exact variant)."""
    cb = Codebook()
    rc = _load().oracle_build_codebook(int(bits), float(base), float(range_), int(shift_mode),
                                       ctypes.byref(cb))
    if rc != 0:
        raise ValueError(f"invalid codebook parameters bits={bits} base={base} range={range_}")
    return cb


def _quant(name: str, w, cb: Codebook) -> np.ndarray:
    w = _f32(w)
    q = np.empty(w.shape, dtype=np.int8)
    getattr(_load(), name)(_ptr(w), w.size, ctypes.byref(cb), _ptr(q))
    return q


def quantize_log(w, cb: Codebook) -> np.ndarray:
    """Eq. (1) evaluated through fp64 logarithms; signed codes in [-q_max, q_max]."""
    return _quant("oracle_quantize_log", w, cb)


def quantize_argmin(w, cb: Codebook) -> np.ndarray:
    """Brute force: nearest of all levels in log space (ties to the larger level)."""
    return _quant("oracle_quantize_argmin", w, cb)


def quantize_thresh(w, cb: Codebook) -> np.ndarray:
    """Count of fp64 decision boundaries tau_j not above |w|."""
    return _quant("oracle_quantize_thresh", w, cb)


def absmax(w) -> tuple[float, bool]:
    w = _f32(w)
    bad = ctypes.c_int(0)
    mx = _load().oracle_absmax(_ptr(w), w.size, ctypes.byref(bad))
    return mx, bool(bad.value)


def packed_row_bytes(K: int, bits: int) -> int:
    return int(_load().oracle_packed_row_bytes(int(K), int(bits)))


def pack(q: np.ndarray, bits: int) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.int8)
    N, K = q.shape
    out = np.zeros((N, packed_row_bytes(K, bits)), dtype=np.uint8)
    if _load().oracle_pack(_ptr(q), N, K, int(bits), _ptr(out)) != 0:
        raise ValueError("pack: unsupported shape")
    return out


def unpack(packed: np.ndarray, N: int, K: int, bits: int) -> np.ndarray:
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    q = np.empty((N, K), dtype=np.int8)
    if _load().oracle_unpack(_ptr(packed), N, K, int(bits), _ptr(q)) != 0:
        raise ValueError("unpack: unsupported shape")
    return q


def dequant(q: np.ndarray, cb: Codebook, table: int = TABLE_F64) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.int8)
    out = np.empty(q.shape, dtype=np.float64)
    _load().oracle_dequant(_ptr(q), q.size, ctypes.byref(cb), int(table), _ptr(out))
    return out


def linear(X: np.ndarray, What: np.ndarray, nthreads: int = 0) -> tuple[np.ndarray, np.ndarray]:
    """Y = X @ What^T in fp64 and A = |X| @ |What|^T (per-output error scale)."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    What = np.ascontiguousarray(What, dtype=np.float64)
    B, K = X.shape
    N, K2 = What.shape
    assert K == K2
    Y = np.empty((B, N), dtype=np.float64)
    A = np.empty((B, N), dtype=np.float64)
    _load().oracle_linear(_ptr(X), B, _ptr(What), N, K, _ptr(Y), _ptr(A), int(nthreads))
    return Y, A


def linear_sampled(X: np.ndarray, packed: np.ndarray, bits: int, cb: Codebook, table: int,
                   bs: np.ndarray, ns: np.ndarray, nthreads: int = 0):
    """Selected outputs Y[bs[i], ns[i]] (and A) straight from packed codes."""
    X = np.ascontiguousarray(X, dtype=np.float64)
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    bs = np.ascontiguousarray(bs, dtype=np.int64)
    ns = np.ascontiguousarray(ns, dtype=np.int64)
    K = X.shape[1]
    Y = np.empty(bs.size, dtype=np.float64)
    A = np.empty(bs.size, dtype=np.float64)
    _load().oracle_linear_sampled(_ptr(X), K, _ptr(packed), int(bits), ctypes.byref(cb),
                                  int(table), _ptr(bs), _ptr(ns), bs.size, _ptr(Y), _ptr(A),
                                  int(nthreads))
    return Y, A


def gptq_factor(H, damp: float = 0.01):
    """U (fp64, upper) with Hd^-1 = U^T U, Hd = H + damp * mean(diag H) * I (a zero
    diagonal entry of H set to 1 first)."""
    H = np.ascontiguousarray(H, dtype=np.float64)
    K = H.shape[0]
    U = np.empty((K, K), dtype=np.float64)
    if _load().oracle_gptq_factor(_ptr(H), K, float(damp), _ptr(U)) != 0:
        raise ValueError("gptq_factor: damped Hessian is not positive definite")
    return U


def gptq(w, H, cb: Codebook, damp: float = 0.01):
    """GPTQ with the Log_b quantiser (fp64, column by column).  Returns the signed
    codes and the value each weight had when its column was quantised."""
    w = _f32(w)
    N, K = w.shape
    H = np.ascontiguousarray(H, dtype=np.float64)
    q = np.empty((N, K), dtype=np.int8)
    w_at = np.empty((N, K), dtype=np.float64)
    rc = _load().oracle_gptq(_ptr(w), N, K, _ptr(H), float(damp), ctypes.byref(cb), _ptr(q), _ptr(w_at))
    if rc != 0:
        raise ValueError("gptq: damped Hessian is not positive definite")
    return q, w_at


def round_f32(v: float) -> float:
    return _load().oracle_round_f32(float(v))


def round_bf16(v: float) -> float:
    return _load().oracle_round_bf16(float(v))


def round_f16(v: float) -> float:
    return _load().oracle_round_f16(float(v))


def bf16_bits(v: float) -> int:
    return int(_load().oracle_bf16_bits(float(v)))


def f16_bits(v: float) -> int:
    return int(_load().oracle_f16_bits(float(v)))


def energy_wmin(w, eps: float) -> float:
    """Eq. (5): smallest magnitude threshold that discards an eps share of the energy."""
    w = _f32(w)
    return float(_load().oracle_energy_wmin(_ptr(w), w.size, float(eps)))


def base_from_range(wmax: float, wmin: float, bits: int) -> float:
    """Eq. (3)."""
    return float(_load().oracle_base_from_range(float(wmax), float(wmin), int(bits)))


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bit patterns (a bf16 is the top half of an fp32)."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def f16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return np.asarray(bits, dtype=np.uint16).view(np.float16).astype(np.float64)


def linear_asym(w, bits: int, scale: float | None = None, zero: int | None = None):
    """Tensor-wise asymmetric uniform (linear) quantisation with 2^bits levels: the
    linear quantiser the paper contrasts Log_b with (Sec. 2 and Fig. 1: a uniform
    grid spends its levels evenly over [min w, max w], while weight histograms are
    bell-shaped), written from its standard definition in fp64:
        scale = (max w - min w) / (2^bits - 1),   zero = round(-min w / scale),
        q = clamp(round(w / scale) + zero, 0, 2^bits - 1),   value = (q - zero) * scale,
    round() to nearest, ties to even.  scale and zero may be given (to requantise on a
    fixed grid).  Returns (q, values, scale, zero).  Used only by the error study;
    the library does not implement it."""
    x = np.asarray(w, dtype=np.float64)
    top = (1 << bits) - 1
    if scale is None:
        lo, hi = float(x.min()), float(x.max())
        scale = (hi - lo) / top if hi > lo else 1.0
        zero = int(np.rint(-lo / scale))
    q = np.clip(np.rint(x / scale) + zero, 0, top).astype(np.int64)
    return q, (q - zero).astype(np.float64) * scale, scale, zero
