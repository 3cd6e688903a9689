"""GPU parity of the fused BatchNorm forward statistics (pf16_conv_fwd_bnstats
feeding pf16_bn_fwd_bwd through conv_stats; Eq. 1, Eq. 2 and Sec. 4.2).

The conv output must be bit-identical to pf16_conv_fwd's.  The BatchNorm
computed from the partial statistics is checked against the oracle's binary64
BatchNorm of that same output, with the tolerance of tests/test_gpu_bn.py:
per element (4L + 8) u (s (|gamma| (|xhat| + 1) + |beta|) + |residual|) + 2^-24,
L = ceil(log2 R) -- the statistics are a different tree of the same FP16
node operations, of depth below L + 6."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import U, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

EPS = 0x00A8
EPS_F = float(np.uint16(EPS).view(np.float16))

SHAPES = [
    # N, H, W, C, K, R, S, stride, pad
    (2, 28, 28, 64, 64, 3, 3, 1, 1),     # halo engine (padded rows of 32)
    (2, 56, 56, 64, 64, 3, 3, 1, 1),     # halo engine (padded rows of 64, columns 56..63 dropped)
    (1, 7, 7, 64, 64, 3, 3, 1, 1),       # im2col, a single partial M tile (49 rows)
    (2, 14, 14, 256, 64, 1, 1, 1, 0),    # dense 1x1
    (2, 13, 13, 128, 256, 3, 3, 2, 1),   # strided 3x3, 4 n-chunks in a tile
    (2, 7, 7, 256, 512, 1, 1, 1, 0),     # two n-tiles (BN = 256)
    (3, 7, 7, 512, 1024, 1, 1, 1, 0),    # four n-tiles
    (2, 28, 28, 128, 128, 3, 3, 1, 1),   # wide halo engine, one image per padded row of 32
    (4, 14, 14, 256, 256, 3, 3, 1, 1),   # wide halo engine, four images per padded row (non-prefix rows)
    (2, 32, 32, 3, 64, 7, 7, 2, 3),      # stem, space-to-depth halo (rows of 32)
    (1, 30, 30, 3, 64, 7, 7, 2, 3),      # stem, s2d halo (rows of 128, columns 15..127 dropped)
    (2, 20, 20, 3, 128, 7, 7, 2, 3),     # stem with 128 outputs (patch matrix)
]


def ids(s):
    return "N{}_{}x{}_C{}_K{}_{}x{}_s{}p{}".format(*s)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_conv_fwd_bnstats_then_bn(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    rows = N * P * Q
    x = syn.normal_f16(syn.seed_for(6, "x"), (N, H, W, C))
    w = syn.he_normal_f16(syn.seed_for(6, "w"), K, R, S, C)
    d = pf16.conv_desc(*shape)
    ws = workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_FWD))
    tx, tw = dev(x), dev(w)
    y_ref, y = empty16(rows * K), empty16(rows * K)
    pf16.conv_fwd(d, tx, tw, y_ref, ws)
    stats = torch.empty(pf16.conv_bnstats_size(d), dtype=torch.uint8, device="cuda")
    pf16.conv_fwd_bnstats(d, tx, tw, y, stats, ws)
    assert pf16.sync_status() == 0
    yb = host(y)
    assert np.array_equal(yb, host(y_ref))  # the statistics do not touch the output

    gamma = f16(1.0 + 0.1 * f64(syn.normal_f16(12, (K,))))
    beta = f16(0.1 * f64(syn.normal_f16(13, (K,))))
    resid = syn.normal_f16(14, (rows, K))
    s = 0.25
    bd = pf16.bn_desc(N, P, Q, K, EPS, int(f16([s])[0]), pf16.PF16_BN_RELU | pf16.PF16_BN_RESIDUAL)
    bws = workspace(pf16.bn_workspace_size(bd))
    tz, tm, ti = empty16(rows * K), empty16(K), empty16(K)
    pf16.bn_fwd_bwd(bd, 0, bws, x=y, gamma=dev(gamma), beta=dev(beta), residual=dev(resid), y=tz, mean=tm,
                    invstd=ti, conv_stats=stats)
    assert pf16.sync_status() == 0
    L = int(np.ceil(np.log2(rows)))
    zo, mean, var, invstd = orc.bn_fwd(yb, gamma, beta, resid, rows, K, EPS_F, s, True)
    xv = f64(yb).reshape(rows, K)
    xhat = (xv - mean) * invstd
    scale = s * (np.abs(f64(gamma)) * (np.abs(xhat) + 1) + np.abs(f64(beta))) + np.abs(f64(resid).reshape(rows, K))
    tol = (4 * L + 8) * U * scale + 2.0 ** -24
    err = np.abs(f64(host(tz)).reshape(rows, K) - zo)
    assert np.all(err <= tol), float(np.max(err / tol))
    assert np.all(np.abs(f64(host(tm)) - mean) <= (L + 8) * U * np.abs(xv).max(0))
    assert np.all(np.abs(f64(host(ti)) - invstd) <= (2 * L + 16) * U * invstd)


BWD_SHAPES = [
    # conv (N, H, W, C, K, R, S, stride, pad) whose data gradient is the BatchNorm's dy; relu
    ((2, 14, 14, 256, 64, 1, 1, 1, 0), True),    # dense 1x1, 256 channels: one 256-wide n-tile
    ((2, 14, 14, 64, 256, 1, 1, 1, 0), True),    # dense 1x1, 64 channels
    ((3, 7, 7, 512, 256, 1, 1, 1, 0), False),    # two n-tiles, no ReLU (no mask)
    ((2, 28, 28, 64, 64, 3, 3, 1, 1), True),     # halo engine, padded rows of 32
    ((2, 56, 56, 64, 64, 3, 3, 1, 1), True),     # halo engine, padded rows of 64 (columns 56..63 dropped)
    ((2, 14, 14, 128, 128, 3, 3, 1, 1), True),   # stride-1 im2col data gradient, 128-wide n-tile
    ((2, 28, 28, 128, 128, 3, 3, 1, 1), True),   # the shape whose forward takes the wide halo engine
    ((1, 7, 7, 64, 64, 3, 3, 1, 1), True),       # one partial tile (49 rows)
    ((2, 7, 7, 256, 1024, 1, 1, 1, 0), True),    # long reduction (16 K-blocks): register-fed epilogue
    ((4, 14, 14, 256, 128, 1, 1, 1, 0), True),   # short reduction, many tiles per CTA: TMA-fed epilogue
    ((3, 14, 14, 128, 128, 3, 3, 2, 1), True),   # strided 3x3, even size: the four stride phases in one
                                                 # launch, scattered rows, ragged last tile of each phase
    ((2, 10, 12, 64, 64, 3, 3, 2, 1), False),    # the same with H != W and no ReLU
    ((2, 14, 14, 512, 512, 3, 3, 2, 1), True),   # the same with two n-tiles
]


def bwd_ids(c):
    return ids(c[0]) + ("_relu" if c[1] else "")


@pytest.mark.parametrize("case", BWD_SHAPES, ids=bwd_ids)
def test_conv_dgrad_bnstats_then_bn_bwd(orc, case):
    """pf16_conv_dgrad_bnstats: dx bit-identical to pf16_conv_dgrad's; the
    BatchNorm backward from its statistics within the BN backward bound of
    tests/test_gpu_bn.py against the oracle on the same dy = dx."""
    shape, relu = case
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    rows = N * H * W
    w = syn.he_normal_f16(syn.seed_for(7, "w"), K, R, S, C)
    dyc = syn.normal_f16(syn.seed_for(7, "dy"), (N, P, Q, K), 0.05)
    xb = syn.normal_f16(syn.seed_for(7, "x"), (rows, C))     # the BatchNorm's input
    gamma = f16(1.0 + 0.1 * f64(syn.normal_f16(15, (C,))))
    beta = f16(0.1 * f64(syn.normal_f16(16, (C,))))
    s = 0.25
    bd = pf16.bn_desc(N, H, W, C, EPS, int(f16([s])[0]), pf16.PF16_BN_RELU if relu else 0)
    bws = workspace(pf16.bn_workspace_size(bd))
    tx, tg, tb = dev(xb), dev(gamma), dev(beta)
    ty, tm, ti = empty16(rows * C), empty16(C), empty16(C)
    tmask = torch.empty(rows * C // 8, dtype=torch.uint8, device="cuda") if relu else None
    pf16.bn_fwd_bwd(bd, 0, bws, x=tx, gamma=tg, beta=tb, y=ty, mean=tm, invstd=ti, relu_mask=tmask)
    assert pf16.sync_status() == 0

    d = pf16.conv_desc(*shape)
    size = pf16.conv_dgrad_bnstats_size(d)
    assert size > 0
    stats = torch.empty(size, dtype=torch.uint8, device="cuda")
    tdyc, tw = dev(dyc), dev(w)
    dx_ref, dx = empty16(rows * C), empty16(rows * C)
    pf16.conv_dgrad(d, tdyc, tw, dx_ref)
    pf16.conv_dgrad_bnstats(d, tdyc, tw, dx, tx, tmask, tm, ti, stats)
    assert pf16.sync_status() == 0
    g = host(dx)
    assert np.array_equal(g, host(dx_ref))  # the statistics do not touch the data gradient
    check_bn_bwd_from_stats(orc, bd, bws, tx, tg, tm, ti, ty, tmask, dx, stats, xb, gamma, beta, N * H * W, C,
                            s, relu)


def check_bn_bwd_from_stats(orc, bd, bws, tx, tg, tm, ti, ty, tmask, dx, stats, xb, gamma, beta, rows, C, s,
                            relu):
    """The BatchNorm backward (phase 1) from the fused statistics in `stats`
    against the oracle's on the same dy = dx."""
    g = host(dx)
    tdx, tdg, tdb = empty16(rows * C), empty16(C), empty16(C)
    pf16.bn_fwd_bwd(bd, 1, bws, x=tx, gamma=tg, mean=tm, invstd=ti, dy=dx, y_saved=ty, relu_mask=tmask,
                    dx=tdx, dgamma=tdg, dbeta=tdb, conv_stats=stats)
    assert pf16.sync_status() == 0
    L = int(np.ceil(np.log2(rows)))
    yb = host(ty)
    dxo, dgo, dbo, dro = orc.bn_bwd(xb, gamma, g, yb, rows, C, EPS_F, s, relu)
    _, mean, var, invstd = orc.bn_fwd(xb, gamma, beta, None, rows, C, EPS_F, s, relu)
    xhat = (f64(xb).reshape(rows, C) - mean) * invstd
    dyp = np.abs(dro)
    k = np.abs(s * f64(gamma) * invstd)
    tol = (4 * L + 8) * U * k * (dyp + dyp.max(0) * (np.abs(xhat) + 1)) + 2.0 ** -24
    err = np.abs(f64(host(tdx)).reshape(rows, C) - dxo)
    assert np.all(err <= tol), float(np.max(err / tol))
    tol_b = (4 * L + 8) * U * s * dyp.sum(0) + 2.0 ** -24
    tol_g = (4 * L + 8) * U * s * (dyp * (np.abs(xhat) + 1)).sum(0) + 2.0 ** -24
    assert np.all(np.abs(f64(host(tdb)) - dbo) <= tol_b), float(np.max(np.abs(f64(host(tdb)) - dbo) / tol_b))
    assert np.all(np.abs(f64(host(tdg)) - dgo) <= tol_g), float(np.max(np.abs(f64(host(tdg)) - dgo) / tol_g))


@pytest.mark.parametrize("shape", [(2, 13, 13, 64, 64, 3, 3, 2, 1),    # odd size: unequal stride phases
                                   (2, 14, 14, 64, 64, 1, 1, 2, 0)],   # strided 1x1: positions no tap reaches
                         ids=ids)
def test_conv_dgrad_bnstats_rejects_strided(shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    d = pf16.conv_desc(*shape)
    assert pf16.conv_dgrad_bnstats_size(d) == 0
    stats = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    t = empty16(N * H * W * C)
    with pytest.raises(pf16.PF16Error):
        pf16.conv_dgrad_bnstats(d, empty16(N * P * Q * K), empty16(K * R * S * C), t, t, None, empty16(C),
                                empty16(C), stats)


ADD_SHAPES = [
    # 1x1 stride-1 data gradients whose dx also takes a masked addend
    (2, 14, 14, 256, 64, 1, 1, 1, 0),    # one n-tile of 256
    (3, 7, 7, 512, 128, 1, 1, 1, 0),     # two n-tiles, 147 rows (a partial M tile)
    (1, 7, 7, 64, 64, 1, 1, 1, 0),       # 64-wide tile, one partial M tile
]


@pytest.mark.parametrize("shape", ADD_SHAPES, ids=ids)
@pytest.mark.parametrize("masked", [True, False], ids=["mask", "nomask"])
def test_conv_dgrad_bnstats_add(orc, shape, masked):
    """pf16_conv_dgrad_bnstats_add: dx bit-identical to the masked addend
    followed by pf16_conv_dgrad with PF16_ACCUMULATE (Sec. 4.2's identity
    shortcut: dresidual plus the first convolution's data gradient); the
    BatchNorm backward from its statistics within the bound of the test
    above."""
    N, H, W, C, K, R, S, st, pd = shape
    rows = N * H * W
    w = syn.he_normal_f16(syn.seed_for(9, "w"), K, R, S, C)
    dyc = syn.normal_f16(syn.seed_for(9, "dy"), (N, H, W, K), 0.05)
    add = syn.normal_f16(syn.seed_for(9, 6), (rows, C), 0.05)
    gate = syn.normal_f16(syn.seed_for(9, 7), (rows, C))     # the addend's ReLU decisions
    on = f64(gate).reshape(rows, C) > 0
    add_mask = np.packbits(on, axis=1, bitorder="little").reshape(-1)
    xb = syn.normal_f16(syn.seed_for(9, "x"), (rows, C))
    gamma = f16(1.0 + 0.1 * f64(syn.normal_f16(17, (C,))))
    beta = f16(0.1 * f64(syn.normal_f16(18, (C,))))
    s = 0.25
    bd = pf16.bn_desc(N, H, W, C, EPS, int(f16([s])[0]), pf16.PF16_BN_RELU)
    bws = workspace(pf16.bn_workspace_size(bd))
    tx, tg, tb = dev(xb), dev(gamma), dev(beta)
    ty, tm, ti = empty16(rows * C), empty16(C), empty16(C)
    tmask = torch.empty(rows * C // 8, dtype=torch.uint8, device="cuda")
    pf16.bn_fwd_bwd(bd, 0, bws, x=tx, gamma=tg, beta=tb, y=ty, mean=tm, invstd=ti, relu_mask=tmask)
    assert pf16.sync_status() == 0

    d = pf16.conv_desc(*shape)
    stats = torch.empty(pf16.conv_dgrad_bnstats_size(d), dtype=torch.uint8, device="cuda")
    tdyc, tw, tadd = dev(dyc), dev(w), dev(add)
    tam = torch.from_numpy(add_mask).to("cuda") if masked else None
    # the two-call path: the masked addend (exact), then the accumulating data gradient
    a_eff = add.reshape(rows, C).copy()
    if masked:
        a_eff[~on] = 0
    dx_ref = dev(a_eff.reshape(-1))
    pf16.conv_dgrad(d, tdyc, tw, dx_ref, None, pf16.PF16_ACCUMULATE)
    dx = empty16(rows * C)
    pf16.conv_dgrad_bnstats_add(d, tdyc, tw, dx, tx, tmask, tm, ti, tadd, tam, stats)
    assert pf16.sync_status() == 0
    assert np.array_equal(host(dx), host(dx_ref))
    check_bn_bwd_from_stats(orc, bd, bws, tx, tg, tm, ti, ty, tmask, dx, stats, xb, gamma, beta, rows, C, s,
                            True)
