"""The stem's BatchNorm + ReLU + max pooling forward as one call
(pf16_bn_relu_maxpool_fwd): bit for bit the separate calls it replaces
(pf16_bn_fwd_bwd phase 0, then pf16_maxpool_fwd_argmax on its y), whose
parity with the oracle tests/test_gpu_bn.py and tests/test_gpu_glue.py check.  Shapes: the stem's own
112 x 112 x 64 at small batch, odd and even sizes (padding rows and columns,
the last window row or column with a single cell), one and eight channel
groups, and statistics from the stem conv's epilogue."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev, empty16, f64, workspace

pytestmark = pytest.mark.gpu

EPS = 0x00A8
SHAPES = [(2, 112, 112, 64), (3, 15, 17, 64), (2, 9, 8, 16), (1, 4, 5, 8), (2, 1, 3, 8), (5, 6, 6, 24)]


def ids(s):
    return "N{}_{}x{}_C{}".format(*s)


def bn_inputs(shape, seed):
    N, H, W, C = shape
    x = syn.normal_f16(syn.seed_for(seed, "x"), (N * H * W, C))
    gamma = (1.0 + 0.1 * f64(syn.normal_f16(syn.seed_for(seed, 6), (C,)))).astype(np.float16).view(np.uint16)
    beta = (0.1 * f64(syn.normal_f16(syn.seed_for(seed, 7), (C,)))).astype(np.float16).view(np.uint16)
    return x, gamma, beta


def u8(n):
    return torch.empty(n, dtype=torch.uint8, device="cuda")


def separate_fwd(d, bws, tx, tg, tb, conv_stats, N, H, W, C):
    rows = N * H * W
    P, Q = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    ty, tm, ti, tmask = empty16(rows * C), empty16(C), empty16(C), u8(rows * C // 8)
    pf16.bn_fwd_bwd(d, 0, bws, x=tx, gamma=tg, beta=tb, y=ty, mean=tm, invstd=ti, relu_mask=tmask,
                    conv_stats=conv_stats)
    tp, targ = empty16(N * P * Q * C), u8(N * P * Q * C)
    pf16.maxpool_fwd_argmax(ty, tp, targ, N, H, W, C)
    assert pf16.sync_status() == 0
    return tm, ti, tmask, tp, targ


def fused_fwd(d, bws, tx, tg, tb, conv_stats, N, H, W, C):
    rows = N * H * W
    P, Q = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    tm, ti, tmask = empty16(C), empty16(C), u8(rows * C // 8)
    tp, targ = empty16(N * P * Q * C), u8(N * P * Q * C)
    pf16.bn_relu_maxpool_fwd(d, bws, tp, targ, x=tx, gamma=tg, beta=tb, mean=tm, invstd=ti, relu_mask=tmask,
                             conv_stats=conv_stats)
    assert pf16.sync_status() == 0
    return tm, ti, tmask, tp, targ


def check_fwd_same(a, b):
    for name, ta, tb_ in zip(("mean", "invstd", "relu_mask", "pooled", "argmax"), a, b):
        assert np.array_equal(ta.cpu().numpy(), tb_.cpu().numpy()), name


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_bn_relu_maxpool_fwd_bit_identical(shape):
    N, H, W, C = shape
    x, gamma, beta = bn_inputs(shape, 31)
    d = pf16.bn_desc(N, H, W, C, EPS, 0x3C00, pf16.PF16_BN_RELU)
    bws = workspace(pf16.bn_workspace_size(d))
    tx, tg, tb = dev(x), dev(gamma), dev(beta)
    check_fwd_same(separate_fwd(d, bws, tx, tg, tb, None, N, H, W, C),
                   fused_fwd(d, bws, tx, tg, tb, None, N, H, W, C))


def test_bn_relu_maxpool_fwd_from_conv_stats():
    """The step's form: the statistics come from the stem conv's epilogue."""
    cshape = (2, 64, 64, 3, 64, 7, 7, 2, 3)
    cd = pf16.conv_desc(*cshape)
    P, Q = cd.out_hw()
    N, C = 2, 64
    xin = syn.normal_f16(syn.seed_for(32, "x"), (N, 64, 64, 3))
    w = syn.he_normal_f16(syn.seed_for(32, "w"), 64, 7, 7, 3)
    ty = empty16(N * P * Q * C)
    st = torch.empty(pf16.conv_bnstats_size(cd), dtype=torch.uint8, device="cuda")
    pf16.conv_fwd_bnstats(cd, dev(xin), dev(w), ty, st, workspace(pf16.conv_workspace_size(cd, pf16.PF16_PASS_FWD)))
    _, gamma, beta = bn_inputs((N, P, Q, C), 33)
    d = pf16.bn_desc(N, P, Q, C, EPS, 0x3C00, pf16.PF16_BN_RELU)
    bws = workspace(pf16.bn_workspace_size(d))
    tg, tb = dev(gamma), dev(beta)
    check_fwd_same(separate_fwd(d, bws, ty, tg, tb, st, N, P, Q, C), fused_fwd(d, bws, ty, tg, tb, st, N, P, Q, C))


def test_stem_fused_rejects():
    N, H, W, C = 1, 4, 4, 8
    d_res = pf16.bn_desc(N, H, W, C, EPS, 0x3C00, pf16.PF16_BN_RELU | pf16.PF16_BN_RESIDUAL)
    d = pf16.bn_desc(N, H, W, C, EPS, 0x3C00, pf16.PF16_BN_RELU)
    bws = workspace(pf16.bn_workspace_size(d))
    t = dict(x=empty16(N * H * W * C), gamma=empty16(C), beta=empty16(C), mean=empty16(C), invstd=empty16(C))
    tp, targ = empty16(N * 2 * 2 * C), u8(N * 2 * 2 * C)
    with pytest.raises(pf16.PF16Error) as e:
        pf16.bn_relu_maxpool_fwd(d_res, bws, tp, targ, residual=empty16(N * H * W * C), **t)
    assert e.value.code == -4  # PF16_ERR_UNSUPPORTED: a residual
    with pytest.raises(pf16.PF16Error) as e:
        pf16.bn_relu_maxpool_fwd(d, bws, tp, targ, y=empty16(N * H * W * C), **t)
    assert e.value.code == -8  # PF16_ERR_ARG: y would not be written
