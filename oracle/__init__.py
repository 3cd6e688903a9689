"""ORACLE -- test infrastructure only.

A plain, slow, obviously-correct CPU implementation (binary64 C loops over
binary16 inputs) of what the pure-FP16 ResNet-50 training step computes.  It
exists to check the CUDA library; it shares no code with it.  Only the tests,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it.  The product path (``paper_1911_07384_gb300``) never does.

Every function takes numpy ``uint16`` arrays holding binary16 bit patterns
(NHWC activations, KRSC weights) and returns binary64 results, except the SGD
step, which is the bit-exact binary16 emulation.

Paper passages followed (arXiv 1911.07384):
  * Sec. 3 (IEEE-754 binary16 format and ops)            -> f16 codec, h_* ops
  * Sec. 5.1 / 5.2 (ResNet-50, all storage and arithmetic
    in FP16, no master copy; PyTorch ImageNet recipe)     -> conv_*, sgd_update
  * Eq. 1, Eq. 2 and the x0.25 scaling of Sec. 4.2        -> bn_fwd, bn_bwd
  * Sec. 5.1 (rest of the ResNet-50 training step)        -> maxpool, avgpool,
                                                             softmax_xent
  * Sec. 5.1 / 5.2 (data-parallel gradient average, FP16)  -> allreduce_combine
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = ["orc_fp16.c", "orc_ops.c"]
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle's C sources into ``oracle/_build/liboracle.so``."""
    srcs = [os.path.join(_HERE, s) for s in _SRCS] + [os.path.join(_HERE, "oracle.h")]
    if not force and os.path.exists(_LIB_PATH):
        newest = max(os.path.getmtime(s) for s in srcs)
        if os.path.getmtime(_LIB_PATH) >= newest:
            return _LIB_PATH
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", "-o", tmp] + [os.path.join(_HERE, s) for s in _SRCS] + ["-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _L():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u16p = ctypes.POINTER(ctypes.c_uint16)
            f64p = ctypes.POINTER(ctypes.c_double)
            i64p = ctypes.POINTER(ctypes.c_int64)
            i32p = ctypes.POINTER(ctypes.c_int32)
            I = ctypes.c_int
            lib.orc_f16_to_f64.argtypes = [ctypes.c_uint16]
            lib.orc_f16_to_f64.restype = ctypes.c_double
            lib.orc_f64_to_f16.argtypes = [ctypes.c_double]
            lib.orc_f64_to_f16.restype = ctypes.c_uint16
            lib.orc_f16_decode.argtypes = [u16p, f64p, ctypes.c_int64]
            lib.orc_f16_encode.argtypes = [f64p, u16p, ctypes.c_int64]
            for nm in ("orc_h_add", "orc_h_sub", "orc_h_mul"):
                getattr(lib, nm).argtypes = [ctypes.c_uint16, ctypes.c_uint16]
                getattr(lib, nm).restype = ctypes.c_uint16
            lib.orc_num_threads.restype = I
            conv_args = [u16p, u16p] + [I] * 9 + [i64p, ctypes.c_int64, f64p, f64p, i32p]
            for nm in ("orc_conv_fwd", "orc_conv_dgrad", "orc_conv_wgrad"):
                getattr(lib, nm).argtypes = conv_args
            lib.orc_sgd_update.argtypes = [u16p, u16p, u16p, ctypes.c_int64, ctypes.c_uint16,
                                           ctypes.c_uint16, ctypes.c_uint16]
            lib.orc_allreduce_combine.argtypes = [u16p, I, ctypes.c_int64, ctypes.c_int64, ctypes.c_uint16,
                                                  u16p]
            lib.orc_bn_fwd.argtypes = [u16p, u16p, u16p, u16p, ctypes.c_int64, I, ctypes.c_double,
                                       ctypes.c_double, I, f64p, f64p, f64p, f64p]
            lib.orc_bn_bwd.argtypes = [u16p, u16p, u16p, u16p, ctypes.c_int64, I, ctypes.c_double,
                                       ctypes.c_double, I, f64p, f64p, f64p, f64p]
            lib.orc_bn_fwd_swap.argtypes = lib.orc_bn_fwd.argtypes
            lib.orc_bn_bwd_swap.argtypes = [u16p, u16p, u16p, u16p, u16p, ctypes.c_int64, I, ctypes.c_double,
                                            ctypes.c_double, I, f64p, f64p, f64p, f64p]
            lib.orc_maxpool_fwd.argtypes = [u16p, I, I, I, I, f64p]
            lib.orc_maxpool_bwd.argtypes = [u16p, u16p, I, I, I, I, f64p, f64p]
            lib.orc_avgpool_fwd.argtypes = [u16p, I, I, I, f64p]
            lib.orc_avgpool_bwd.argtypes = [u16p, I, I, I, f64p]
            lib.orc_softmax_xent.argtypes = [u16p, u16p, i32p, I, I, f64p, f64p, f64p]
            _lib = lib
    return _lib


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.float16:
        a = a.view(np.uint16)
    assert a.dtype == np.uint16, a.dtype
    return a


def _p(a, ct):
    if a is None:
        return None
    return a.ctypes.data_as(ctypes.POINTER(ct))


def num_threads() -> int:
    return int(_L().orc_num_threads())


# ---------------------------------------------------------------- binary16 codec
def f16_to_f64(bits: np.ndarray) -> np.ndarray:
    b = _u16(bits)
    out = np.empty(b.shape, np.float64)
    _L().orc_f16_decode(_p(b, ctypes.c_uint16), _p(out, ctypes.c_double), b.size)
    return out


def f64_to_f16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, np.uint16)
    _L().orc_f16_encode(_p(x, ctypes.c_double), _p(out, ctypes.c_uint16), x.size)
    return out


def h_add(a: int, b: int) -> int:
    return int(_L().orc_h_add(a, b))


def h_sub(a: int, b: int) -> int:
    return int(_L().orc_h_sub(a, b))


def h_mul(a: int, b: int) -> int:
    return int(_L().orc_h_mul(a, b))


# ---------------------------------------------------------------- convolutions
def conv_out_hw(H, W, R, S, stride, pad):
    return (H + 2 * pad - R) // stride + 1, (W + 2 * pad - S) // stride + 1


def _conv(fn, a, b, dims, idx, out_count):
    a, b = _u16(a), _u16(b)
    if idx is not None:
        idx = np.ascontiguousarray(idx, dtype=np.int64)
        count = idx.size
    else:
        count = out_count
    V = np.empty(count, np.float64)
    A = np.empty(count, np.float64)
    T = np.empty(count, np.int32)
    fn(_p(a, ctypes.c_uint16), _p(b, ctypes.c_uint16), *[int(d) for d in dims],
       _p(idx, ctypes.c_int64) if idx is not None else None, count,
       _p(V, ctypes.c_double), _p(A, ctypes.c_double), _p(T, ctypes.c_int32))
    return V, A, T


def conv_fwd(x, w, N, H, W, C, K, R, S, stride, pad, idx=None):
    """Forward conv.  Returns (V, A, T) per output of y[N,P,Q,K] (flat, or at idx)."""
    P, Q = conv_out_hw(H, W, R, S, stride, pad)
    return _conv(_L().orc_conv_fwd, x, w, (N, H, W, C, K, R, S, stride, pad), idx, N * P * Q * K)


def conv_dgrad(dy, w, N, H, W, C, K, R, S, stride, pad, idx=None):
    """Data gradient.  Returns (V, A, T) per element of dx[N,H,W,C]."""
    return _conv(_L().orc_conv_dgrad, dy, w, (N, H, W, C, K, R, S, stride, pad), idx, N * H * W * C)


def conv_wgrad(x, dy, N, H, W, C, K, R, S, stride, pad, idx=None):
    """Weight gradient.  Returns (V, A, T) per element of dw[K,R,S,C]."""
    return _conv(_L().orc_conv_wgrad, x, dy, (N, H, W, C, K, R, S, stride, pad), idx, K * R * S * C)


# ---------------------------------------------------------------- SGD
def sgd_update(w, v, g, lr_bits: int, momentum_bits: int, wd_bits: int):
    """Bit-exact pure-FP16 SGD step; returns new (w, v) bit arrays."""
    w = _u16(w).copy()
    v = _u16(v).copy()
    g = _u16(g)
    _L().orc_sgd_update(_p(w, ctypes.c_uint16), _p(v, ctypes.c_uint16), _p(g, ctypes.c_uint16),
                        w.size, lr_bits, momentum_bits, wd_bits)
    return w, v


# ---------------------------------------------------------------- data-parallel exchange
def allreduce_combine(planes, scale_bits: int):
    """planes: [world][n] binary16 bits, one plane per rank in rank order.
    Returns the n binary16 bits of the fixed-order FP16 average (Sec. 5.1,
    5.2): a pairwise tree of additions over the ranks, then x scale."""
    planes = _u16(planes)
    world, n = planes.shape
    out = np.empty(n, np.uint16)
    _L().orc_allreduce_combine(_p(planes, ctypes.c_uint16), world, n, n, scale_bits, _p(out, ctypes.c_uint16))
    return out


# ---------------------------------------------------------------- BatchNorm
def bn_fwd_swap(x, gamma, beta, residual, R, C, eps, s, relu):
    """The swap variant (Sec. 4.1): y = gamma*(s*xhat + residual) + beta [, ReLU].
    Returns y[R,C], mean[C], var[C], invstd[C] (all binary64)."""
    x, gamma, beta, residual = _u16(x), _u16(gamma), _u16(beta), _u16(residual)
    y = np.empty(R * C, np.float64)
    mean, var, invstd = (np.empty(C, np.float64) for _ in range(3))
    _L().orc_bn_fwd_swap(_p(x, ctypes.c_uint16), _p(gamma, ctypes.c_uint16), _p(beta, ctypes.c_uint16),
                         _p(residual, ctypes.c_uint16), R, C, float(eps), float(s), int(relu),
                         _p(y, ctypes.c_double), _p(mean, ctypes.c_double), _p(var, ctypes.c_double),
                         _p(invstd, ctypes.c_double))
    return y.reshape(R, C), mean, var, invstd


def bn_bwd_swap(x, gamma, dy, y_saved, residual, R, C, eps, s, relu):
    """Backward of bn_fwd_swap.  Returns dx[R,C], dgamma[C], dbeta[C], dres[R,C] (binary64)."""
    x, gamma, dy, residual = _u16(x), _u16(gamma), _u16(dy), _u16(residual)
    y_saved = _u16(y_saved) if y_saved is not None else np.zeros(1, np.uint16)
    dx = np.empty(R * C, np.float64)
    dres = np.empty(R * C, np.float64)
    dg, db = np.empty(C, np.float64), np.empty(C, np.float64)
    _L().orc_bn_bwd_swap(_p(x, ctypes.c_uint16), _p(gamma, ctypes.c_uint16), _p(dy, ctypes.c_uint16),
                         _p(y_saved, ctypes.c_uint16), _p(residual, ctypes.c_uint16), R, C, float(eps), float(s),
                         int(relu), _p(dx, ctypes.c_double), _p(dg, ctypes.c_double), _p(db, ctypes.c_double),
                         _p(dres, ctypes.c_double))
    return dx.reshape(R, C), dg, db, dres.reshape(R, C)


def bn_fwd(x, gamma, beta, residual, R, C, eps, s, relu):
    """Returns y[R,C], mean[C], var[C], invstd[C] (all binary64)."""
    x, gamma, beta = _u16(x), _u16(gamma), _u16(beta)
    residual = _u16(residual) if residual is not None else None
    y = np.empty(R * C, np.float64)
    mean, var, invstd = (np.empty(C, np.float64) for _ in range(3))
    _L().orc_bn_fwd(_p(x, ctypes.c_uint16), _p(gamma, ctypes.c_uint16), _p(beta, ctypes.c_uint16),
                    _p(residual, ctypes.c_uint16), R, C, float(eps), float(s), int(relu),
                    _p(y, ctypes.c_double), _p(mean, ctypes.c_double), _p(var, ctypes.c_double),
                    _p(invstd, ctypes.c_double))
    return y.reshape(R, C), mean, var, invstd


def bn_bwd(x, gamma, dy, y_saved, R, C, eps, s, relu):
    """Returns dx[R,C], dgamma[C], dbeta[C], dres[R,C] (binary64)."""
    x, gamma, dy = _u16(x), _u16(gamma), _u16(dy)
    y_saved = _u16(y_saved) if y_saved is not None else np.zeros(1, np.uint16)
    dx = np.empty(R * C, np.float64)
    dres = np.empty(R * C, np.float64)
    dg, db = np.empty(C, np.float64), np.empty(C, np.float64)
    _L().orc_bn_bwd(_p(x, ctypes.c_uint16), _p(gamma, ctypes.c_uint16), _p(dy, ctypes.c_uint16),
                    _p(y_saved, ctypes.c_uint16), R, C, float(eps), float(s), int(relu),
                    _p(dx, ctypes.c_double), _p(dg, ctypes.c_double), _p(db, ctypes.c_double),
                    _p(dres, ctypes.c_double))
    return dx.reshape(R, C), dg, db, dres.reshape(R, C)


# ---------------------------------------------------------------- pools, loss
def maxpool_fwd(x, N, H, W, C):
    P, Q = conv_out_hw(H, W, 3, 3, 2, 1)
    x = _u16(x)
    y = np.empty(N * P * Q * C, np.float64)
    _L().orc_maxpool_fwd(_p(x, ctypes.c_uint16), N, H, W, C, _p(y, ctypes.c_double))
    return y


def maxpool_bwd(x, dy, N, H, W, C):
    x, dy = _u16(x), _u16(dy)
    dx = np.empty(N * H * W * C, np.float64)
    A = np.empty(N * H * W * C, np.float64)
    _L().orc_maxpool_bwd(_p(x, ctypes.c_uint16), _p(dy, ctypes.c_uint16), N, H, W, C,
                         _p(dx, ctypes.c_double), _p(A, ctypes.c_double))
    return dx, A


def avgpool_fwd(x, N, HW, C):
    x = _u16(x)
    y = np.empty(N * C, np.float64)
    _L().orc_avgpool_fwd(_p(x, ctypes.c_uint16), N, HW, C, _p(y, ctypes.c_double))
    return y


def avgpool_bwd(dy, N, HW, C):
    dy = _u16(dy)
    dx = np.empty(N * HW * C, np.float64)
    _L().orc_avgpool_bwd(_p(dy, ctypes.c_uint16), N, HW, C, _p(dx, ctypes.c_double))
    return dx


def softmax_xent(logits, bias, labels, B, K):
    logits = _u16(logits)
    bias = _u16(bias) if bias is not None else None
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    loss = np.zeros(1, np.float64)
    dl = np.empty(B * K, np.float64)
    db = np.empty(K, np.float64)
    _L().orc_softmax_xent(_p(logits, ctypes.c_uint16), _p(bias, ctypes.c_uint16),
                          _p(labels, ctypes.c_int32), B, K, _p(loss, ctypes.c_double),
                          _p(dl, ctypes.c_double), _p(db, ctypes.c_double))
    return float(loss[0]), dl, db
