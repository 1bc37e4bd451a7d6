"""CPU oracle for the exact integer GEMM substrate -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never imports,
links or calls it; it shares no code with the CUDA path.

Every routine is a thin ctypes call into ``qx_oracle.c`` (plain C loops, int64
accumulation for the integer paths, float64 for the FP32 variants).  Inputs
are numpy arrays or CPU torch tensors; they are widened to int32 / float64
before the call, which is lossless for the int16 and int32 operands the
substrate accepts.

Definitions (paper: Abstract, Methodology paragraph, Table 1, Table 2):

* ``gemm``    C = A B, int64, plus the largest |partial sum| in k order (the
  accumulation contract of the Methodology paragraph).
* ``conv2d``  direct NCHW/KCRS cross-correlation with zero padding, no bias.
* ``attn``    S = Q K^T then O = S V, no softmax and no scale; given (heads,
  L, d) operands, the same core independently for every head.
* ``minmax``  smallest and largest element (Table 2 min/max rows).
* ``pool2d``  NCHW max / average pooling without padding (Table 2 pooling
  rows); integer averages are floor(window sum / window size).
* ``requant`` min(max(acc, 0) >> shift, hi): ReLU, arithmetic right shift and
  clamp between the layers of an integer pipeline.
* ``lenet``   the LeNet-shaped INT32 pipeline (Results, CNN performance): the
  classic LeNet-5 layer shapes composed from conv2d, requant, pool2d and
  gemm above.
* ``*_f64``   the same three definitions in float64; ``*_absref`` applies them
  to element-wise absolute values, giving the per-element magnitude
  sum |a_k||b_k| that the FP32 tolerance is stated against.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qx_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None
_lock = threading.Lock()

_i64 = ctypes.c_int64
_p = ctypes.c_void_p


def build(force: bool = False) -> str:
    """Compile qx_oracle.c into oracle/liboracle.so with gcc (OpenMP)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O3", "-fopenmp", "-fPIC", "-shared", "-std=c11",
           _SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            lib.qxo_threads.restype = ctypes.c_int
            lib.qxo_gemm_i64.argtypes = [_i64, _i64, _i64, _p, _i64, _p, _i64, _p, _i64, _p]
            lib.qxo_conv2d_i64.argtypes = [_i64] * 9 + [_p, _p, _p]
            lib.qxo_attn_i64.argtypes = [_i64, _i64, _p, _p, _p, _p, _p, _p]
            lib.qxo_gemm_f64.argtypes = [_i64, _i64, _i64, _p, _i64, _p, _i64, _p, _i64]
            lib.qxo_conv2d_f64.argtypes = [_i64] * 9 + [_p, _p, _p]
            lib.qxo_attn_f64.argtypes = [_i64, _i64, _p, _p, _p, _p, _p]
            lib.qxo_minmax_i64.argtypes = [_i64, _p, _p, _p]
            lib.qxo_minmax_f64.argtypes = [_i64, _p, _p, _p]
            lib.qxo_pool2d_i64.argtypes = [_i64] * 7 + [ctypes.c_int, _p, _p]
            lib.qxo_pool2d_f64.argtypes = [_i64] * 7 + [ctypes.c_int, _p, _p]
            _lib = lib
    return _lib


def _np(a):
    if hasattr(a, "detach"):  # torch tensor
        a = a.detach().cpu().numpy()
    return np.asarray(a)


def _as_i32(a) -> np.ndarray:
    a = _np(a)
    if a.dtype.kind not in "iu":
        raise TypeError(f"integer operand expected, got {a.dtype}")
    if a.size and (a.min() < -(2**31) or a.max() > 2**31 - 1):
        raise ValueError("operand outside int32")
    return np.ascontiguousarray(a, dtype=np.int32)


def _as_f64(a) -> np.ndarray:
    return np.ascontiguousarray(_np(a), dtype=np.float64)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def threads() -> int:
    """OpenMP threads the oracle uses (OMP_NUM_THREADS, else all cores)."""
    return int(_load().qxo_threads())


# --------------------------------------------------------------------- GEMM
def gemm(A, B):
    """Exact C = A B for integer A (M x K) and B (K x N).

    Returns ``(C, max_abs_partial)``: C as int64 and the largest
    |sum_{t<=k} A[i][t] B[t][j]| over all i, j, k.
    """
    A = _as_i32(A)
    B = _as_i32(B)
    if A.ndim != 2 or B.ndim != 2 or A.shape[1] != B.shape[0]:
        raise ValueError(f"shape mismatch {A.shape} x {B.shape}")
    M, K = A.shape
    N = B.shape[1]
    C = np.zeros((M, N), dtype=np.int64)
    worst = ctypes.c_int64(0)
    if M and N:
        _load().qxo_gemm_i64(M, N, K, _ptr(A), K, _ptr(B), N, _ptr(C), N,
                             ctypes.byref(worst))
    return C, int(worst.value)


def gemm_f64(A, B):
    A = _as_f64(A)
    B = _as_f64(B)
    if A.ndim != 2 or B.ndim != 2 or A.shape[1] != B.shape[0]:
        raise ValueError(f"shape mismatch {A.shape} x {B.shape}")
    M, K = A.shape
    N = B.shape[1]
    C = np.zeros((M, N), dtype=np.float64)
    if M and N:
        _load().qxo_gemm_f64(M, N, K, _ptr(A), K, _ptr(B), N, _ptr(C), N)
    return C


def gemm_absref(A, B):
    """Per-element sum_k |A[i][k]| |B[k][j]| in float64."""
    return gemm_f64(np.abs(_as_f64(A)), np.abs(_as_f64(B)))


# --------------------------------------------------------------------- Conv
def _conv_shapes(x, w, stride, pad):
    if x.ndim != 4 or w.ndim != 4 or x.shape[1] != w.shape[1]:
        raise ValueError(f"conv shapes {x.shape} {w.shape}")
    if stride < 1 or pad < 0:
        raise ValueError("stride >= 1 and pad >= 0 required")
    n, c, h, wd = x.shape
    k, _, r, s = w.shape
    P = (h + 2 * pad - r) // stride + 1
    Q = (wd + 2 * pad - s) // stride + 1
    if P < 1 or Q < 1:
        raise ValueError("empty output")
    return n, c, h, wd, k, r, s, P, Q


def conv2d(x, w, stride: int = 1, pad: int = 0):
    """Exact direct convolution (int64), NCHW x KCRS -> N K P Q."""
    x = _as_i32(x)
    w = _as_i32(w)
    n, c, h, wd, k, r, s, P, Q = _conv_shapes(x, w, stride, pad)
    y = np.zeros((n, k, P, Q), dtype=np.int64)
    _load().qxo_conv2d_i64(n, c, h, wd, k, r, s, stride, pad, _ptr(x), _ptr(w), _ptr(y))
    return y


def conv2d_f64(x, w, stride: int = 1, pad: int = 0):
    x = _as_f64(x)
    w = _as_f64(w)
    n, c, h, wd, k, r, s, P, Q = _conv_shapes(x, w, stride, pad)
    y = np.zeros((n, k, P, Q), dtype=np.float64)
    _load().qxo_conv2d_f64(n, c, h, wd, k, r, s, stride, pad, _ptr(x), _ptr(w), _ptr(y))
    return y


def conv2d_absref(x, w, stride: int = 1, pad: int = 0):
    return conv2d_f64(np.abs(_as_f64(x)), np.abs(_as_f64(w)), stride, pad)


# ---------------------------------------------------------------- Attention
def _attn_shapes(Q, K, V):
    if Q.ndim != 2 or Q.shape != K.shape or Q.shape != V.shape:
        raise ValueError(f"attention shapes {Q.shape} {K.shape} {V.shape}")
    return Q.shape


def _per_head(fn, Q, K, V):
    """Batched cores: ``fn`` on every head of (heads, L, d) operands; the
    results are stacked along a new leading axis (scalars: the maximum)."""
    Q, K, V = _np(Q), _np(K), _np(V)
    if Q.ndim != 3 or Q.shape != K.shape or Q.shape != V.shape:
        raise ValueError(f"attention shapes {Q.shape} {K.shape} {V.shape}")
    outs = [fn(Q[h], K[h], V[h]) for h in range(Q.shape[0])]
    return tuple(max(col) if isinstance(col[0], int) else np.stack(col) for col in zip(*outs))


def attn(Q, K, V):
    """Exact O = (Q K^T) V as written.  Returns ``(O, S, max_abs_S)``.
    (heads, L, d) operands give (heads, L, d) O, (heads, L, L) S and the
    largest |S| over all heads."""
    if _np(Q).ndim == 3:
        return _per_head(attn, Q, K, V)
    Q = _as_i32(Q)
    K = _as_i32(K)
    V = _as_i32(V)
    L, d = _attn_shapes(Q, K, V)
    S = np.zeros((L, L), dtype=np.int64)
    O = np.zeros((L, d), dtype=np.int64)
    worst = ctypes.c_int64(0)
    _load().qxo_attn_i64(L, d, _ptr(Q), _ptr(K), _ptr(V), _ptr(S), _ptr(O),
                         ctypes.byref(worst))
    return O, S, int(worst.value)


def attn_f64(Q, K, V):
    if _np(Q).ndim == 3:
        return _per_head(attn_f64, Q, K, V)
    Q = _as_f64(Q)
    K = _as_f64(K)
    V = _as_f64(V)
    L, d = _attn_shapes(Q, K, V)
    S = np.zeros((L, L), dtype=np.float64)
    O = np.zeros((L, d), dtype=np.float64)
    _load().qxo_attn_f64(L, d, _ptr(Q), _ptr(K), _ptr(V), _ptr(S), _ptr(O))
    return O, S


def attn_absref(Q, K, V):
    """(|Q| |K|^T) |V| in float64: the magnitude the FP32 attention error is
    measured against (it carries the first product's error into the second)."""
    O, _ = attn_f64(np.abs(_as_f64(Q)), np.abs(_as_f64(K)), np.abs(_as_f64(V)))
    return O


# ------------------------------------------------ memory-bound operators
def minmax(x):
    """(min, max) of all elements: exact for integers, float64 for floats."""
    a = _np(x).reshape(-1)
    if a.size == 0:
        raise ValueError("empty input")
    if a.dtype.kind in "iu":
        a = _as_i32(a)
        lo, hi = ctypes.c_int64(0), ctypes.c_int64(0)
        _load().qxo_minmax_i64(a.size, _ptr(a), ctypes.byref(lo), ctypes.byref(hi))
        return int(lo.value), int(hi.value)
    a = _as_f64(a)
    lo, hi = ctypes.c_double(0), ctypes.c_double(0)
    _load().qxo_minmax_f64(a.size, _ptr(a), ctypes.byref(lo), ctypes.byref(hi))
    return float(lo.value), float(hi.value)


def pool2d(x, kh: int = 2, kw: int = 2, stride: int = 2, mode: str = "max"):
    """NCHW pooling, no padding.  Integers: int64 result (average = floor);
    floats: float64 result."""
    a = _np(x)
    if a.ndim != 4 or kh < 1 or kw < 1 or stride < 1 or mode not in ("max", "avg"):
        raise ValueError("bad pooling arguments")
    n, c, h, w = a.shape
    if h < kh or w < kw:
        raise ValueError("window larger than the image")
    P, Q = (h - kh) // stride + 1, (w - kw) // stride + 1
    is_max = 1 if mode == "max" else 0
    if a.dtype.kind in "iu":
        a = _as_i32(a)
        y = np.zeros((n, c, P, Q), dtype=np.int64)
        _load().qxo_pool2d_i64(n, c, h, w, kh, kw, stride, is_max, _ptr(a), _ptr(y))
    else:
        a = _as_f64(a)
        y = np.zeros((n, c, P, Q), dtype=np.float64)
        _load().qxo_pool2d_f64(n, c, h, w, kh, kw, stride, is_max, _ptr(a), _ptr(y))
    return y


# ------------------------------------------------------ integer pipeline
def requant(acc, shift: int, hi: int):
    """ReLU, arithmetic right shift by `shift`, clamp to `hi` (int64)."""
    a = np.asarray(_np(acc), dtype=np.int64)
    return np.minimum(np.maximum(a, 0) >> shift, hi)


LENET_SHAPES = {            # classic LeNet-5 layer shapes (the paper names only "LeNet")
    "x": (1, 32, 32), "w1": (6, 1, 5, 5), "w2": (16, 6, 5, 5),
    "w3": (400, 120), "w4": (120, 84), "w5": (84, 10),
}


def lenet(x, w1, w2, w3, w4, w5, shifts, act_hi: int, pool: str = "max"):
    """LeNet-shaped INT32 pipeline on N x 1 x 32 x 32 images:
    conv 6@5x5 -> requant -> pool 2x2/2 -> conv 16@5x5 -> requant -> pool 2x2/2
    -> flatten (NCHW order, 400) -> fc 120 -> requant -> fc 84 -> requant
    -> fc 10 (raw int32 logits).  `shifts` are the four requantizing shifts."""
    x = _np(x)
    a = requant(conv2d(x, w1), shifts[0], act_hi)
    a = pool2d(a, 2, 2, 2, pool)
    a = requant(conv2d(a, w2), shifts[1], act_hi)
    a = pool2d(a, 2, 2, 2, pool)
    a = a.reshape(a.shape[0], -1)
    a = requant(gemm(a, w3)[0], shifts[2], act_hi)
    a = requant(gemm(a, w4)[0], shifts[3], act_hi)
    return gemm(a, w5)[0]
