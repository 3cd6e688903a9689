"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
entry point include/pf16.h declares, and rejects invalid calls on the host
with the documented status codes before touching the device."""
import ctypes
import os
import re

import pytest

from paper_1911_07384_gb300 import pf16

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "pf16.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pf16_[a-z0-9_]+)\s*\(", src)))


def test_header_and_binding_agree():
    assert declared_functions() == sorted(pf16.EXPORTS)


def test_library_exports_every_declared_symbol():
    L = pf16.lib()
    for name in declared_functions():
        assert hasattr(L, name), name
        assert ctypes.cast(getattr(L, name), ctypes.c_void_p).value


def test_status_strings():
    for code in range(-8, 1):
        assert pf16.status_string(code) != "unknown status"
    assert pf16.status_string(-99) == "unknown status"


FAKE = ctypes.c_void_p(0x10000)      # aligned, never dereferenced: validation fails first
FAKE_MIS = ctypes.c_void_p(0x10002)  # misaligned


def test_conv_validation_errors():
    L = pf16.lib()
    good = pf16.conv_desc(2, 8, 8, 64, 64, 3, 3, 1, 1)
    assert L.pf16_conv_fwd(None, FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_NULL
    bad = pf16.conv_desc(2, 8, 8, 64, 64, 3, 3, 1, 1)
    bad.h = 0
    assert L.pf16_conv_fwd(ctypes.byref(bad), FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_SHAPE
    odd = pf16.conv_desc(2, 8, 8, 48, 64, 3, 3, 1, 1)
    assert L.pf16_conv_fwd(ctypes.byref(odd), FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_UNSUPPORTED
    s3 = pf16.conv_desc(2, 8, 8, 64, 64, 3, 3, 3, 1)
    assert L.pf16_conv_fwd(ctypes.byref(s3), FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_UNSUPPORTED
    assert L.pf16_conv_fwd(ctypes.byref(good), None, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_NULL
    assert L.pf16_conv_fwd(ctypes.byref(good), FAKE_MIS, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_ALIGN
    assert L.pf16_conv_fwd(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, 0x80, None) == pf16.PF16_ERR_ARG
    assert L.pf16_conv_wgrad(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, 1, None) == pf16.PF16_ERR_ARG
    stem = pf16.conv_desc(2, 32, 32, 3, 64, 7, 7, 2, 3)
    assert L.pf16_conv_dgrad(ctypes.byref(stem), FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_UNSUPPORTED
    # stem forward needs its patch workspace
    assert L.pf16_conv_fwd(ctypes.byref(stem), FAKE, FAKE, FAKE, None, 0, 0, None) == pf16.PF16_ERR_WORKSPACE
    # data gradient with BatchNorm backward statistics
    src = pf16.BnSource(FAKE, None, FAKE, FAKE)
    sz = pf16.conv_dgrad_bnstats_size(good)
    assert sz > 0
    dg = L.pf16_conv_dgrad_bnstats
    assert dg(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, None, FAKE, sz, None) == pf16.PF16_ERR_NULL
    assert dg(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), None, sz, None) == pf16.PF16_ERR_NULL
    assert dg(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), FAKE, sz - 1,
              None) == pf16.PF16_ERR_WORKSPACE
    assert dg(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), FAKE_MIS, sz,
              None) == pf16.PF16_ERR_ALIGN
    nox = pf16.BnSource(None, None, FAKE, FAKE)
    assert dg(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, ctypes.byref(nox), FAKE, sz, None) == pf16.PF16_ERR_NULL
    # stride 2: the four stride phases must share their grid (even sizes with 3x3 / pad 1)
    assert pf16.conv_dgrad_bnstats_size(pf16.conv_desc(2, 8, 8, 64, 64, 3, 3, 2, 1)) == sz
    for s2 in (pf16.conv_desc(2, 9, 9, 64, 64, 3, 3, 2, 1), pf16.conv_desc(2, 8, 9, 64, 64, 3, 3, 2, 1),
               pf16.conv_desc(2, 8, 8, 64, 64, 1, 1, 2, 0)):
        assert pf16.conv_dgrad_bnstats_size(s2) == 0
        assert dg(ctypes.byref(s2), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), FAKE, sz,
                  None) == pf16.PF16_ERR_UNSUPPORTED
    # ... plus a masked addend: 1x1 stride 1 only, no overlap with dx
    da = L.pf16_conv_dgrad_bnstats_add
    one = pf16.conv_desc(2, 8, 8, 256, 64, 1, 1, 1, 0)
    sz1 = pf16.conv_dgrad_bnstats_size(one)
    far = ctypes.c_void_p(0x1000000)  # past dx's 2*8*8*256*2 bytes at FAKE
    assert da(ctypes.byref(one), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), None, None, FAKE, sz1,
              None) == pf16.PF16_ERR_NULL
    assert da(ctypes.byref(good), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), far, None, FAKE, sz,
              None) == pf16.PF16_ERR_UNSUPPORTED  # 3x3
    assert da(ctypes.byref(one), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), FAKE, None, FAKE, sz1,
              None) == pf16.PF16_ERR_ARG  # add is dx
    assert da(ctypes.byref(one), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), ctypes.c_void_p(0x10100), None,
              FAKE, sz1, None) == pf16.PF16_ERR_ARG  # add overlaps dx
    assert da(ctypes.byref(one), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), ctypes.c_void_p(0x1000008), None,
              FAKE, sz1, None) == pf16.PF16_ERR_ALIGN
    assert da(ctypes.byref(one), FAKE, FAKE, FAKE, None, 0, ctypes.byref(src), far, ctypes.c_void_p(0x2000004),
              FAKE, sz1, None) == pf16.PF16_ERR_ALIGN  # mask not 8-byte aligned


def test_tc_rate_validation_errors():
    L = pf16.lib()
    out = ctypes.c_double(0.0)
    assert L.pf16_tc_rate(256, 0, 1, 100, None, None) == pf16.PF16_ERR_NULL
    for n, f32, chains, reps in [(96, 0, 1, 100), (256, 2, 1, 100), (256, 0, 3, 100), (256, 0, 1, 0),
                                 (64, 0, 1, (1 << 20) + 1)]:
        assert L.pf16_tc_rate(n, f32, chains, reps, ctypes.byref(out), None) == pf16.PF16_ERR_ARG


def test_workspace_sizes_are_host_computable():
    cfg3 = pf16.conv_desc(256, 56, 56, 256, 64, 1, 1, 1, 0)
    assert pf16.conv_workspace_size(cfg3, pf16.PF16_PASS_FWD) == 0
    assert pf16.conv_workspace_size(cfg3, pf16.PF16_PASS_DGRAD) == 0
    w = pf16.conv_workspace_size(cfg3, pf16.PF16_PASS_WGRAD)
    assert w > 0 and w % 256 == 0
    stem = pf16.conv_desc(256, 224, 224, 3, 64, 7, 7, 2, 3)
    assert pf16.conv_workspace_size(stem, pf16.PF16_PASS_FWD) >= 256 * 112 * 112 * 147 * 2
    bad = pf16.conv_desc(0, 56, 56, 256, 64, 1, 1, 1, 0)
    assert pf16.conv_workspace_size(bad, pf16.PF16_PASS_WGRAD) == 0


def test_other_validation_errors():
    L = pf16.lib()
    assert L.pf16_sgd_update(FAKE, FAKE, FAKE, 16, 0, 0, 0, 1, None) == pf16.PF16_ERR_ARG
    assert L.pf16_sgd_update(None, FAKE, FAKE, 16, 0, 0, 0, 0, None) == pf16.PF16_ERR_NULL
    assert L.pf16_sgd_update(FAKE_MIS, FAKE, FAKE, 16, 0, 0, 0, 0, None) == pf16.PF16_ERR_ALIGN
    assert L.pf16_sgd_update(None, None, None, 0, 0, 0, 0, 0, None) == pf16.PF16_OK  # n = 0: no-op
    d = pf16.bn_desc(2, 4, 4, 12)
    assert L.pf16_bn_fwd_bwd(ctypes.byref(d), 0, None, FAKE, 1 << 20, None) == pf16.PF16_ERR_UNSUPPORTED
    d = pf16.bn_desc(2, 4, 4, 64)
    t = pf16.BnTensors()
    assert L.pf16_bn_fwd_bwd(ctypes.byref(d), 2, ctypes.byref(t), FAKE, 1 << 20, None) == pf16.PF16_ERR_ARG
    assert L.pf16_bn_fwd_bwd(ctypes.byref(d), 0, ctypes.byref(t), FAKE, 1 << 20, None) == pf16.PF16_ERR_NULL
    assert L.pf16_bn_fwd_bwd(ctypes.byref(d), 0, ctypes.byref(t), FAKE, 1, None) == pf16.PF16_ERR_WORKSPACE
    # the swap variant is defined with a residual input only, and needs two more partial buffers
    ds = pf16.bn_desc(2, 4, 4, 64, 0x00A8, 0x3400, pf16.PF16_BN_SWAP)
    assert L.pf16_bn_fwd_bwd(ctypes.byref(ds), 0, ctypes.byref(t), FAKE, 1 << 20, None) == pf16.PF16_ERR_ARG
    assert pf16.bn_workspace_size(ds) == 0
    dr = pf16.bn_desc(2, 4, 4, 64, 0x00A8, 0x3400, pf16.PF16_BN_RESIDUAL)
    dsr = pf16.bn_desc(2, 4, 4, 64, 0x00A8, 0x3400, pf16.PF16_BN_RESIDUAL | pf16.PF16_BN_SWAP)
    assert pf16.bn_workspace_size(dsr) > pf16.bn_workspace_size(dr) > 0
    assert L.pf16_maxpool_fwd(FAKE, FAKE, 1, 8, 8, 12, None) == pf16.PF16_ERR_UNSUPPORTED
    assert L.pf16_maxpool_fwd_argmax(FAKE, FAKE, None, 1, 8, 8, 16, None) == pf16.PF16_ERR_NULL
    assert L.pf16_maxpool_fwd_argmax(FAKE, FAKE, ctypes.c_void_p(0x10004), 1, 8, 8, 16,
                                     None) == pf16.PF16_ERR_ALIGN
    assert L.pf16_maxpool_bwd_argmax(None, FAKE, FAKE, 1, 8, 8, 16, None) == pf16.PF16_ERR_NULL
    assert L.pf16_maxpool_bwd_argmax(FAKE, FAKE, FAKE, 1, 8, 8, 12, None) == pf16.PF16_ERR_UNSUPPORTED
    assert L.pf16_avgpool_fwd(FAKE, None, 1, 49, 64, None) == pf16.PF16_ERR_NULL
    assert L.pf16_softmax_xent(FAKE, None, FAKE, 4, 5000, FAKE, FAKE, None, FAKE, 1 << 20,
                               None) == pf16.PF16_ERR_UNSUPPORTED


def test_wait_flag_validation_errors():
    L = pf16.lib()
    assert L.pf16_wait_flag(None, 1, 1000, None) == pf16.PF16_ERR_NULL
    assert L.pf16_wait_flag(FAKE_MIS, 1, 1000, None) == pf16.PF16_ERR_ALIGN
    assert L.pf16_wait_flag(FAKE, 1, 10_000_000_001, None) == pf16.PF16_ERR_ARG


def test_launch_plan_agrees_with_the_library():
    """bench.py counts one data-gradient launch for a stride-2 filter when the
    library runs its four stride phases as one GEMM -- exactly the layers for
    which the library also offers the fused backward statistics."""
    import bench

    seen = set()
    for h, w in [(8, 8), (9, 9), (12, 10), (13, 14), (56, 56), (7, 7)]:
        for r in (1, 3, 5, 7):
            for pad in range(r):
                if (h + 2 * pad - r) < 0 or (w + 2 * pad - r) < 0:
                    continue
                d = pf16.conv_desc(2, h, w, 64, 64, r, r, 2, pad)
                one = bench.one_phase_launch(d)
                assert one == (pf16.conv_dgrad_bnstats_size(d) > 0), (h, w, r, pad)
                seen.add(one)
    assert seen == {True, False}
