"""BatchNorm applied in the conv's operand path (pf16_conv_fwd_bnin,
pf16_conv_wgrad_bnin; Eq. 1-2 and the x0.25 of Sec. 4.2 fused into the next
convolution): the conv of BN(x), taking the BatchNorm's input x and
transforming each operand tile in shared memory, must be bit-identical to
pf16_bn_fwd_bwd phase 0 (which stores BN(x)) followed by the plain conv --
the output, its fused statistics, the ReLU bit mask, and the weight
gradient.  The BatchNorm's stored output is itself checked against the
oracle in tests/test_gpu_bn.py, and the plain convs in tests/test_gpu_conv.py.
Also: phase 0 with y = NULL computes the same mean / invstd as the full call."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

EPS = 0x00A8

SHAPES = [
    # N, H, W, C, K (1x1, stride 1), post_scale bits, relu
    (4, 14, 14, 64, 256, 0x3400, True),     # a stage-1 style 64 -> 256 expansion, one n-tile
    (2, 28, 28, 128, 512, 0x3400, True),    # two n-tiles: each A tile transformed twice, mask once
    (3, 7, 7, 512, 2048, 0x3400, True),     # eight n-tiles, 147 rows (a partial M tile)
    (2, 9, 11, 192, 64, 0x3C00, False),     # three channel chunks, 198 rows, no ReLU, scale 1
    (1, 56, 56, 64, 256, 0x3400, True),     # 3,136 rows: many tiles per CTA
]


def ids(c):
    return "N{}_{}x{}_C{}_K{}_s{:04x}_relu{}".format(*c)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


@pytest.mark.parametrize("case", SHAPES, ids=ids)
def test_bn_in_operand_path_bit_identical(case):
    N, H, W, C, K, sbits, relu = case
    R = N * H * W
    x = f16(2.0 * f64(syn.normal_f16(31, (R, C))) + 0.5)
    gamma = f16(1.0 + 0.3 * f64(syn.normal_f16(32, (C,))))
    beta = f16(0.2 * f64(syn.normal_f16(33, (C,))))
    w = syn.he_normal_f16(syn.seed_for(6, "w", C + K), K, 1, 1, C)
    dy = syn.normal_f16(syn.seed_for(6, "dy", C + K), (R, K), 0.01)
    tx, tg, tb, tw, tdy = dev(x), dev(gamma), dev(beta), dev(w), dev(dy)

    # the unfused pair: the BatchNorm stores its output, the conv reads it
    bd = pf16.bn_desc(N, H, W, C, EPS, sbits, pf16.PF16_BN_RELU if relu else 0)
    bws = workspace(pf16.bn_workspace_size(bd))
    ybn, tm, ti = empty16(R * C), empty16(C), empty16(C)
    mask = torch.zeros(R * C // 8, dtype=torch.uint8, device="cuda") if relu else None
    pf16.bn_fwd_bwd(bd, 0, bws, x=tx, gamma=tg, beta=tb, y=ybn, mean=tm, invstd=ti, relu_mask=mask)
    # statistics only: the same mean and invstd
    tm2, ti2 = empty16(C), empty16(C)
    pf16.bn_fwd_bwd(bd, 0, bws, x=tx, mean=tm2, invstd=ti2)
    d = pf16.conv_desc(N, H, W, C, K, 1, 1, 1, 0)
    ssz = pf16.conv_bnstats_size(d)
    y_ref = empty16(R * K)
    st_ref = torch.zeros(ssz, dtype=torch.uint8, device="cuda")
    pf16.conv_fwd_bnstats(d, ybn, tw, y_ref, st_ref)
    dw_ref = empty16(K * C)
    wws = workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD))
    pf16.conv_wgrad(d, ybn, tdy, dw_ref, wws)
    assert pf16.sync_status() == 0
    assert np.array_equal(host(tm2), host(tm)) and np.array_equal(host(ti2), host(ti))

    # fused: the conv takes x and applies the BatchNorm to each operand tile
    mask2 = torch.full((R * C // 8,), 0xA5, dtype=torch.uint8, device="cuda") if relu else None
    op = pf16.bn_operand(tm, ti, tg, tb, sbits, relu, mask2)
    y = empty16(R * K)
    st = torch.zeros(ssz, dtype=torch.uint8, device="cuda")
    pf16.conv_fwd_bnin(d, tx, op, tw, y, st)
    dw = empty16(K * C)
    pf16.conv_wgrad_bnin(d, tx, pf16.bn_operand(tm, ti, tg, tb, sbits, relu), tdy, dw, wws)
    assert pf16.sync_status() == 0
    assert np.array_equal(host(y), host(y_ref))
    assert np.array_equal(host(dw), host(dw_ref))
    if relu:
        assert torch.equal(mask2, mask)
    # the output's statistics: the BatchNorm computed from them is the same
    k_bd = pf16.bn_desc(N, H, W, K, EPS, 0x3400, 0)
    k_ws = workspace(pf16.bn_workspace_size(k_bd))
    outs = []
    for stats in (st_ref, st):
        m, i = empty16(K), empty16(K)
        pf16.bn_fwd_bwd(k_bd, 0, k_ws, x=y_ref, mean=m, invstd=i, conv_stats=stats)
        outs.append((host(m), host(i)))
    assert pf16.sync_status() == 0
    assert np.array_equal(outs[0][0], outs[1][0]) and np.array_equal(outs[0][1], outs[1][1])


def test_bn_in_rejects_other_shapes_and_arguments():
    C, K = 64, 64
    t = empty16(1 << 16)
    m = empty16(C)
    op = pf16.bn_operand(m, m, m, m, 0x3400, True)
    with pytest.raises(pf16.PF16Error):  # a 3x3 conv is not covered
        pf16.conv_fwd_bnin(pf16.conv_desc(1, 8, 8, C, K, 3, 3, 1, 1), t, op, t, t)
    with pytest.raises(pf16.PF16Error):  # a strided 1x1 neither
        pf16.conv_wgrad_bnin(pf16.conv_desc(1, 8, 8, C, K, 1, 1, 2, 0), t, op, t, t)
    with pytest.raises(pf16.PF16Error):  # a mask without ReLU
        pf16.conv_fwd_bnin(pf16.conv_desc(1, 8, 8, C, K, 1, 1, 1, 0), t,
                           pf16.bn_operand(m, m, m, m, 0x3400, False, torch.empty(64, dtype=torch.uint8,
                                                                                   device="cuda")), t, t)
    with pytest.raises(pf16.PF16Error):  # no mask from the weight gradient
        pf16.conv_wgrad_bnin(pf16.conv_desc(1, 8, 8, C, K, 1, 1, 1, 0), t,
                             pf16.bn_operand(m, m, m, m, 0x3400, True, torch.empty(64, dtype=torch.uint8,
                                                                                   device="cuda")), t, t,
                             workspace(1 << 20))
    assert pf16.sync_status() == 0
