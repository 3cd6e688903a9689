"""Thin ctypes binding of libpf16 (include/pf16.h): the same entry points,
argument marshalling only.  Tensors are torch CUDA tensors (any 2-byte dtype;
the bits are binary16); every computation happens in the library's kernels.
A non-zero status raises PF16Error.  If the library cannot be built or
loaded, importing the entry points raises: there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

PF16_OK = 0
PF16_ERR_NULL = -1
PF16_ERR_ALIGN = -2
PF16_ERR_SHAPE = -3
PF16_ERR_UNSUPPORTED = -4
PF16_ERR_WORKSPACE = -5
PF16_ERR_CUDA = -6
PF16_ERR_TIMEOUT = -7
PF16_ERR_ARG = -8

PF16_ACCUMULATE = 0x1
PF16_F32_ACCUM = 0x4
PF16_BN_RELU = 0x1
PF16_BN_RESIDUAL = 0x2
PF16_BN_SWAP = 0x4
PF16_PASS_FWD, PF16_PASS_DGRAD, PF16_PASS_WGRAD = 0, 1, 2

EXPORTS = [
    "pf16_conv_workspace_size", "pf16_conv_fwd", "pf16_conv_dgrad", "pf16_conv_wgrad",
    "pf16_sgd_update", "pf16_allreduce_combine", "pf16_bn_workspace_size", "pf16_bn_fwd_bwd", "pf16_maxpool_fwd",
    "pf16_maxpool_bwd", "pf16_avgpool_fwd", "pf16_avgpool_bwd",
    "pf16_softmax_xent_workspace_size", "pf16_softmax_xent", "pf16_sync_status",
    "pf16_status_string", "pf16_device_arch", "pf16_conv_wgrad_noalloc",
    "pf16_kernel_launches", "pf16_maxpool_fwd_argmax", "pf16_maxpool_bwd_argmax",
    "pf16_conv_bnstats_size", "pf16_conv_fwd_bnstats", "pf16_conv_dgrad_bnstats_size",
    "pf16_conv_dgrad_bnstats", "pf16_conv_dgrad_bnstats_add", "pf16_tc_rate", "pf16_wait_flag",
    "pf16_conv_fwd_bnin", "pf16_conv_wgrad_bnin", "pf16_bn_relu_maxpool_fwd",
]


class PF16Error(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: pf16 status {code} ({status_string(code)})")


class ConvDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n", "h", "w", "c", "k", "r", "s", "stride", "pad")]

    def out_hw(self):
        return ((self.h + 2 * self.pad - self.r) // self.stride + 1,
                (self.w + 2 * self.pad - self.s) // self.stride + 1)


class BnSource(ctypes.Structure):
    """pf16_bn_source: the BatchNorm whose output gradient a data gradient is."""
    _fields_ = [(n, ctypes.c_void_p) for n in ("x", "relu_mask", "mean", "invstd")]


class BnOperand(ctypes.Structure):
    """pf16_bn_operand: a BatchNorm applied in a conv's operand path."""
    _fields_ = [("mean", ctypes.c_void_p), ("invstd", ctypes.c_void_p), ("gamma", ctypes.c_void_p),
                ("beta", ctypes.c_void_p), ("post_scale", ctypes.c_uint16), ("flags", ctypes.c_uint32),
                ("relu_mask", ctypes.c_void_p)]


class BnDesc(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("h", ctypes.c_int32), ("w", ctypes.c_int32),
                ("c", ctypes.c_int32), ("eps", ctypes.c_uint16), ("post_scale", ctypes.c_uint16),
                ("flags", ctypes.c_uint32)]


_BN_T = ("x", "gamma", "beta", "residual", "dy", "y_saved", "y", "mean", "invstd", "dx", "dgamma",
         "dbeta", "dresidual", "relu_mask", "conv_stats")


class BnTensors(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in _BN_T]


_lock = threading.Lock()
_lib = None


def lib():
    """Load (building first if needed) libpf16.so."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            L = ctypes.CDLL(path)
            vp, sz, u16, u32, i32, I = (ctypes.c_void_p, ctypes.c_size_t, ctypes.c_uint16,
                                       ctypes.c_uint32, ctypes.c_int32, ctypes.c_int)
            cdp = ctypes.POINTER(ConvDesc)
            L.pf16_conv_workspace_size.argtypes = [cdp, I]
            L.pf16_conv_workspace_size.restype = sz
            for nm in ("pf16_conv_fwd", "pf16_conv_dgrad", "pf16_conv_wgrad"):
                getattr(L, nm).argtypes = [cdp, vp, vp, vp, vp, sz, u32, vp]
                getattr(L, nm).restype = I
            L.pf16_conv_bnstats_size.argtypes = [cdp]
            L.pf16_conv_bnstats_size.restype = sz
            L.pf16_conv_fwd_bnstats.argtypes = [cdp, vp, vp, vp, vp, sz, vp, sz, vp]
            bop = ctypes.POINTER(BnOperand)
            L.pf16_conv_fwd_bnin.argtypes = [cdp, vp, bop, vp, vp, vp, sz, vp]
            L.pf16_conv_fwd_bnin.restype = I
            L.pf16_conv_wgrad_bnin.argtypes = [cdp, vp, bop, vp, vp, vp, sz, vp]
            L.pf16_conv_wgrad_bnin.restype = I
            L.pf16_conv_fwd_bnstats.restype = I
            L.pf16_conv_dgrad_bnstats_size.argtypes = [cdp]
            L.pf16_conv_dgrad_bnstats_size.restype = sz
            L.pf16_conv_dgrad_bnstats.argtypes = [cdp, vp, vp, vp, vp, sz, ctypes.POINTER(BnSource), vp, sz,
                                                  vp]
            L.pf16_conv_dgrad_bnstats.restype = I
            L.pf16_conv_dgrad_bnstats_add.argtypes = [cdp, vp, vp, vp, vp, sz, ctypes.POINTER(BnSource), vp, vp,
                                                      vp, sz, vp]
            L.pf16_conv_dgrad_bnstats_add.restype = I
            L.pf16_conv_wgrad_noalloc.argtypes = [cdp, vp, vp, vp, u32, vp]
            L.pf16_conv_wgrad_noalloc.restype = I
            L.pf16_sgd_update.argtypes = [vp, vp, vp, sz, u16, u16, u16, u32, vp]
            L.pf16_sgd_update.restype = I
            L.pf16_allreduce_combine.argtypes = [vp, i32, sz, sz, u16, vp, vp]
            L.pf16_allreduce_combine.restype = I
            L.pf16_bn_workspace_size.argtypes = [ctypes.POINTER(BnDesc)]
            L.pf16_bn_workspace_size.restype = sz
            L.pf16_bn_fwd_bwd.argtypes = [ctypes.POINTER(BnDesc), I, ctypes.POINTER(BnTensors), vp,
                                          sz, vp]
            L.pf16_bn_fwd_bwd.restype = I
            L.pf16_bn_relu_maxpool_fwd.argtypes = [ctypes.POINTER(BnDesc), ctypes.POINTER(BnTensors), vp, vp,
                                                   vp, sz, vp]
            L.pf16_bn_relu_maxpool_fwd.restype = I
            L.pf16_maxpool_fwd.argtypes = [vp, vp, i32, i32, i32, i32, vp]
            L.pf16_maxpool_bwd.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp]
            L.pf16_maxpool_fwd_argmax.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp]
            L.pf16_maxpool_bwd_argmax.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp]
            L.pf16_avgpool_fwd.argtypes = [vp, vp, i32, i32, i32, vp]
            L.pf16_avgpool_bwd.argtypes = [vp, vp, i32, i32, i32, vp]
            for nm in ("pf16_maxpool_fwd", "pf16_maxpool_bwd", "pf16_avgpool_fwd", "pf16_avgpool_bwd",
                       "pf16_maxpool_fwd_argmax", "pf16_maxpool_bwd_argmax"):
                getattr(L, nm).restype = I
            L.pf16_softmax_xent_workspace_size.argtypes = [i32, i32]
            L.pf16_softmax_xent_workspace_size.restype = sz
            L.pf16_softmax_xent.argtypes = [vp, vp, vp, i32, i32, vp, vp, vp, vp, sz, vp]
            L.pf16_softmax_xent.restype = I
            L.pf16_sync_status.argtypes = [vp]
            L.pf16_sync_status.restype = I
            L.pf16_status_string.argtypes = [I]
            L.pf16_status_string.restype = ctypes.c_char_p
            L.pf16_tc_rate.argtypes = [i32, i32, i32, i32, ctypes.POINTER(ctypes.c_double), vp]
            L.pf16_tc_rate.restype = I
            L.pf16_wait_flag.argtypes = [vp, ctypes.c_uint32, ctypes.c_uint64, vp]
            L.pf16_wait_flag.restype = I
            L.pf16_device_arch.argtypes = []
            L.pf16_device_arch.restype = I
            L.pf16_kernel_launches.argtypes = []
            L.pf16_kernel_launches.restype = ctypes.c_uint64
            _lib = L
    return _lib


def status_string(code: int) -> str:
    return lib().pf16_status_string(int(code)).decode()


def _check(rc: int, where: str) -> None:
    if rc != PF16_OK:
        raise PF16Error(rc, where)


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch

        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def conv_desc(n, h, w, c, k, r, s, stride, pad) -> ConvDesc:
    return ConvDesc(n, h, w, c, k, r, s, stride, pad)


def conv_workspace_size(d: ConvDesc, pass_: int) -> int:
    return int(lib().pf16_conv_workspace_size(ctypes.byref(d), pass_))


def conv_fwd(d, x, w, y, ws=None, flags=0, stream=None):
    _check(lib().pf16_conv_fwd(ctypes.byref(d), _ptr(x), _ptr(w), _ptr(y), _ptr(ws), _nbytes(ws),
                               flags, _stream(stream)), "pf16_conv_fwd")


def conv_bnstats_size(d) -> int:
    return int(lib().pf16_conv_bnstats_size(ctypes.byref(d)))


def conv_fwd_bnstats(d, x, w, y, stats, ws=None, stream=None):
    """Forward conv that also writes the BatchNorm statistics of y into `stats`
    (a device buffer of conv_bnstats_size(d) bytes) for bn_fwd_bwd(conv_stats=)."""
    _check(lib().pf16_conv_fwd_bnstats(ctypes.byref(d), _ptr(x), _ptr(w), _ptr(y), _ptr(ws), _nbytes(ws),
                                       _ptr(stats), _nbytes(stats), _stream(stream)), "pf16_conv_fwd_bnstats")


def bn_operand(mean, invstd, gamma, beta, post_scale_bits, relu, relu_mask=None) -> BnOperand:
    return BnOperand(_ptr(mean), _ptr(invstd), _ptr(gamma), _ptr(beta), post_scale_bits,
                     PF16_BN_RELU if relu else 0, _ptr(relu_mask))


def conv_fwd_bnin(d, x, bn: BnOperand, w, y, stats=None, stream=None):
    """Forward conv of BN(x): x is the BatchNorm's input; the BatchNorm is
    applied to each operand tile (and its ReLU decisions written to
    bn.relu_mask when given); optional statistics of y as conv_fwd_bnstats."""
    _check(lib().pf16_conv_fwd_bnin(ctypes.byref(d), _ptr(x), ctypes.byref(bn), _ptr(w), _ptr(y), _ptr(stats),
                                    _nbytes(stats), _stream(stream)), "pf16_conv_fwd_bnin")


def conv_wgrad_bnin(d, x, bn: BnOperand, dy, dw, ws=None, stream=None):
    """Weight gradient with input BN(x), applied in the operand path."""
    _check(lib().pf16_conv_wgrad_bnin(ctypes.byref(d), _ptr(x), ctypes.byref(bn), _ptr(dy), _ptr(dw), _ptr(ws),
                                      _nbytes(ws), _stream(stream)), "pf16_conv_wgrad_bnin")


def conv_dgrad(d, dy, w, dx, ws=None, flags=0, stream=None):
    _check(lib().pf16_conv_dgrad(ctypes.byref(d), _ptr(dy), _ptr(w), _ptr(dx), _ptr(ws),
                                 _nbytes(ws), flags, _stream(stream)), "pf16_conv_dgrad")


def conv_dgrad_bnstats_size(d) -> int:
    return int(lib().pf16_conv_dgrad_bnstats_size(ctypes.byref(d)))


def conv_dgrad_bnstats(d, dy, w, dx, x, relu_mask, mean, invstd, stats, ws=None, stream=None):
    """Data gradient that also writes the backward statistics of the BatchNorm
    whose output gradient dx is (input x, ReLU mask or None, saved mean and
    invstd) into `stats` (conv_dgrad_bnstats_size(d) bytes) for
    bn_fwd_bwd(phase 1, conv_stats=)."""
    src = BnSource(_ptr(x), _ptr(relu_mask), _ptr(mean), _ptr(invstd))
    _check(lib().pf16_conv_dgrad_bnstats(ctypes.byref(d), _ptr(dy), _ptr(w), _ptr(dx), _ptr(ws),
                                         _nbytes(ws), ctypes.byref(src), _ptr(stats), _nbytes(stats),
                                         _stream(stream)), "pf16_conv_dgrad_bnstats")


def conv_dgrad_bnstats_add(d, dy, w, dx, x, relu_mask, mean, invstd, add, add_mask, stats, ws=None,
                           stream=None):
    """conv_dgrad_bnstats with dx = rn(data gradient + add where add_mask's bit
    is set); add_mask None: the whole of add."""
    src = BnSource(_ptr(x), _ptr(relu_mask), _ptr(mean), _ptr(invstd))
    _check(lib().pf16_conv_dgrad_bnstats_add(ctypes.byref(d), _ptr(dy), _ptr(w), _ptr(dx), _ptr(ws),
                                             _nbytes(ws), ctypes.byref(src), _ptr(add), _ptr(add_mask),
                                             _ptr(stats), _nbytes(stats), _stream(stream)),
           "pf16_conv_dgrad_bnstats_add")


def conv_wgrad(d, x, dy, dw, ws=None, flags=0, stream=None):
    _check(lib().pf16_conv_wgrad(ctypes.byref(d), _ptr(x), _ptr(dy), _ptr(dw), _ptr(ws),
                                 _nbytes(ws), flags, _stream(stream)), "pf16_conv_wgrad")


def conv_wgrad_noalloc(d, x, dy, dw, flags=0, stream=None):
    """Weight gradient with the library's fixed internal scratch instead of a
    caller workspace (for callers that cannot provide device memory)."""
    _check(lib().pf16_conv_wgrad_noalloc(ctypes.byref(d), _ptr(x), _ptr(dy), _ptr(dw), flags,
                                         _stream(stream)), "pf16_conv_wgrad_noalloc")


WGRAD_NOALLOC_SCRATCH_BYTES = 32 << 20


def sgd_update(w, v, g, lr_bits, momentum_bits, wd_bits, flags=0, stream=None):
    _check(lib().pf16_sgd_update(_ptr(w), _ptr(v), _ptr(g), w.numel(), lr_bits, momentum_bits,
                                 wd_bits, flags, _stream(stream)), "pf16_sgd_update")


def allreduce_combine(planes, world, n, plane_stride, scale_bits, out, stream=None):
    """planes: a device tensor holding `world` planes of n binary16 values,
    plane r at element offset r * plane_stride; out: n values (may be planes)."""
    _check(lib().pf16_allreduce_combine(_ptr(planes), world, n, plane_stride, scale_bits, _ptr(out),
                                        _stream(stream)), "pf16_allreduce_combine")


def bn_desc(n, h, w, c, eps_bits=0x00A8, post_scale_bits=0x3400, flags=0) -> BnDesc:
    return BnDesc(n, h, w, c, eps_bits, post_scale_bits, flags)


def bn_workspace_size(d: BnDesc) -> int:
    return int(lib().pf16_bn_workspace_size(ctypes.byref(d)))


def bn_fwd_bwd(d, phase, ws, stream=None, **tensors):
    t = BnTensors(**{k: (v.data_ptr() if v is not None else None) for k, v in tensors.items()})
    _check(lib().pf16_bn_fwd_bwd(ctypes.byref(d), phase, ctypes.byref(t), _ptr(ws), _nbytes(ws),
                                 _stream(stream)), "pf16_bn_fwd_bwd")


def bn_relu_maxpool_fwd(d, ws, pooled, argmax, stream=None, **tensors):
    """The stem's BatchNorm (phase 0, ReLU) with its output max-pooled at once;
    y is not stored (pass no y).  tensors as bn_fwd_bwd's."""
    t = BnTensors(**{k: (v.data_ptr() if v is not None else None) for k, v in tensors.items()})
    _check(lib().pf16_bn_relu_maxpool_fwd(ctypes.byref(d), ctypes.byref(t), _ptr(pooled), _ptr(argmax), _ptr(ws),
                                          _nbytes(ws), _stream(stream)), "pf16_bn_relu_maxpool_fwd")


def maxpool_fwd(x, y, n, h, w, c, stream=None):
    _check(lib().pf16_maxpool_fwd(_ptr(x), _ptr(y), n, h, w, c, _stream(stream)), "pf16_maxpool_fwd")


def maxpool_bwd(x, dy, dx, n, h, w, c, stream=None):
    _check(lib().pf16_maxpool_bwd(_ptr(x), _ptr(dy), _ptr(dx), n, h, w, c, _stream(stream)),
           "pf16_maxpool_bwd")


def maxpool_fwd_argmax(x, y, argmax, n, h, w, c, stream=None):
    _check(lib().pf16_maxpool_fwd_argmax(_ptr(x), _ptr(y), _ptr(argmax), n, h, w, c, _stream(stream)),
           "pf16_maxpool_fwd_argmax")


def maxpool_bwd_argmax(argmax, dy, dx, n, h, w, c, stream=None):
    _check(lib().pf16_maxpool_bwd_argmax(_ptr(argmax), _ptr(dy), _ptr(dx), n, h, w, c, _stream(stream)),
           "pf16_maxpool_bwd_argmax")


def avgpool_fwd(x, y, n, hw, c, stream=None):
    _check(lib().pf16_avgpool_fwd(_ptr(x), _ptr(y), n, hw, c, _stream(stream)), "pf16_avgpool_fwd")


def avgpool_bwd(dy, dx, n, hw, c, stream=None):
    _check(lib().pf16_avgpool_bwd(_ptr(dy), _ptr(dx), n, hw, c, _stream(stream)), "pf16_avgpool_bwd")


def softmax_xent_workspace_size(b, k) -> int:
    return int(lib().pf16_softmax_xent_workspace_size(b, k))


def softmax_xent(logits, bias, labels, b, k, loss, dlogits, dbias, ws, stream=None):
    _check(lib().pf16_softmax_xent(_ptr(logits), _ptr(bias), _ptr(labels), b, k, _ptr(loss),
                                   _ptr(dlogits), _ptr(dbias), _ptr(ws), _nbytes(ws),
                                   _stream(stream)), "pf16_softmax_xent")


def sync_status(stream=None) -> int:
    return int(lib().pf16_sync_status(_stream(stream)))


def device_arch() -> int:
    return int(lib().pf16_device_arch())


def kernel_launches() -> int:
    """Kernels libpf16 has enqueued in this process (graph-captured ones once)."""
    return int(lib().pf16_kernel_launches())


def loaded_path() -> str:
    return os.path.abspath(_build.LIB)


def tc_rate(n, f32_accum=False, chains=1, reps=20000, stream=None) -> float:
    """TFLOP/s of the library's MMA-only probe (pf16_tc_rate): kind::f16
    tcgen05 MMAs of M = 128, N = n from shared memory, on every SM."""
    out = ctypes.c_double(0.0)
    _check(lib().pf16_tc_rate(int(n), 1 if f32_accum else 0, int(chains), int(reps), ctypes.byref(out),
                              _stream(stream)), "pf16_tc_rate")
    return out.value


def wait_flag(flag, value, timeout_ns, stream=None):
    """Enqueue a bounded wait until the int32 device word `flag` equals `value`
    (pf16_wait_flag); an expired wait shows up in sync_status() as
    PF16_ERR_TIMEOUT."""
    _check(lib().pf16_wait_flag(_ptr(flag), int(value) & 0xFFFFFFFF, int(timeout_ns), _stream(stream)),
           "pf16_wait_flag")
