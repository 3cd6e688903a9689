"""pf16_conv_wgrad_noalloc: the weight gradient for callers that cannot give
the library scratch memory (hosts that plan every byte of device memory
themselves, deployments that forbid allocation after set-up, bindings with no
CUDA allocator).  It must agree with pf16_conv_wgrad, which takes a caller
workspace, on consecutive calls that share the library's fixed scratch, and it
must refuse layers whose scratch would not fit.

Kept in the last file pytest collects, so a stop-at-first-failure run has
already run every other test before this one."""
import ctypes

import numpy as np
import pytest

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import conv_bound, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

# 3x3 config-1 layer (49 split-K partial planes) and a 1x1 N=32 GEMM layer
SHAPES = [(4, 56, 56, 64, 64, 3, 3, 1, 1), (32, 28, 28, 512, 128, 1, 1, 1, 0)]


def call_noalloc(d, x, dy, dw):
    """Through the C-ABI directly: no workspace argument exists."""
    import torch

    rc = pf16.lib().pf16_conv_wgrad_noalloc(ctypes.byref(d), ctypes.c_void_p(x.data_ptr()),
                                            ctypes.c_void_p(dy.data_ptr()), ctypes.c_void_p(dw.data_ptr()),
                                            0, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == pf16.PF16_OK, pf16.status_string(rc)


def test_noalloc_matches_workspace_entry_point(orc):
    for i, shape in enumerate(SHAPES):
        N, H, W, C, K, R, S, st, pd = shape
        P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
        d = pf16.conv_desc(*shape)
        need = pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)
        assert 0 < need <= pf16.WGRAD_NOALLOC_SCRATCH_BYTES
        # two calls in a row with different inputs: the second reuses the shared scratch
        for call in range(2):
            x = syn.normal_f16(syn.seed_for(1, "x", 10 * i + call), (N, H, W, C))
            dy = syn.normal_f16(syn.seed_for(1, "dy", 10 * i + call), (N, P, Q, K), 0.01)
            tx, tdy = dev(x), dev(dy)
            ref = empty16(K * R * S * C)
            pf16.conv_wgrad(d, tx, tdy, ref, workspace(need))
            got = empty16(K * R * S * C)
            call_noalloc(d, tx, tdy, got)
            assert pf16.sync_status() == 0
            # same tolerance as the parity tests, with sum|terms| from the oracle
            idx = np.arange(0, K * R * S * C, 7)
            _, A, _ = orc.conv_wgrad(x, dy, *shape, idx=idx)
            a, b = f64(host(got))[idx], f64(host(ref))[idx]
            assert np.all(np.abs(a - b) <= conv_bound(A, N * P * Q))
            assert np.array_equal(host(got), host(ref))  # same plan, deterministic kernels


def test_noalloc_rejects_layers_that_do_not_fit():
    stem = pf16.conv_desc(256, 224, 224, 3, 64, 7, 7, 2, 3)
    assert pf16.conv_workspace_size(stem, pf16.PF16_PASS_WGRAD) > pf16.WGRAD_NOALLOC_SCRATCH_BYTES
    x, dy, dw = empty16(8), empty16(8), empty16(8)  # never touched: rejected before any launch
    rc = pf16.lib().pf16_conv_wgrad_noalloc(ctypes.byref(stem), ctypes.c_void_p(x.data_ptr()),
                                            ctypes.c_void_p(dy.data_ptr()), ctypes.c_void_p(dw.data_ptr()),
                                            0, None)
    assert rc == pf16.PF16_ERR_WORKSPACE
