"""GPU parity of pf16_bn_fwd_bwd (Eq. 1, Eq. 2, x post_scale, residual, ReLU)
against the oracle's binary64 BatchNorm on the same binary16 inputs.

Tolerance (no bound is given by the paper; derived from the FP16 schedule):
the statistics are halving trees of depth L = ceil(log2 R) (one rounding per
level), the normalisation and affine steps add a fixed number of roundings.
Per element of the forward output
    |err| <= (4 L + 8) u * (s (|gamma| (|xhat| + 1) + |beta|) + |residual|) + 2^-24
and of the data gradient
    |err| <= (4 L + 8) u * |s gamma invstd| * (|dy'| + max|dy'| (|xhat| + 1)) + 2^-24,
u = 2^-11; dgamma / dbeta within (4 L + 8) u * s * sum|terms| + 2^-24."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import U, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

EPS = 0x00A8
EPS_F = float(np.uint16(EPS).view(np.float16))


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


CASES = [
    # N, H, W, C, post_scale, relu, residual
    (4, 14, 14, 64, 0.25, True, True),
    (2, 7, 7, 2048, 0.25, False, False),
    (8, 56, 56, 64, 1.0, True, False),
    (3, 5, 7, 24, 0.25, True, True),      # C not a power of two, ragged rows
    (256, 14, 14, 256, 0.25, True, True),  # R = 50,176: two chunks on some statistics CTAs
    # R = 9,990,500 rows of 8 channels: 39,026 statistics chunks of 256 rows,
    # more than 152 backward CTAs take at 256 chunks each (that grid grows to
    # 153, most CTAs closing a full 256-chunk tree); the last chunk is partial
    # and owned by an inner CTA
    (1, 1, 9990500, 8, 0.25, True, False),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "N{}_{}x{}_C{}_s{}_relu{}_res{}".format(*c))
def test_bn_fwd_bwd(orc, case):
    N, H, W, C, s, relu, res = case
    R = N * H * W
    L = int(np.ceil(np.log2(R)))
    x = f16(f64(syn.normal_f16(11, (R, C), 2.0)) + 0.5)
    gamma = f16(1.0 + 0.1 * f64(syn.normal_f16(12, (C,))))
    beta = f16(0.1 * f64(syn.normal_f16(13, (C,))))
    resid = syn.normal_f16(14, (R, C)) if res else None
    dy = syn.normal_f16(15, (R, C), 0.01)
    flags = (pf16.PF16_BN_RELU if relu else 0) | (pf16.PF16_BN_RESIDUAL if res else 0)
    sbits = int(f16([s])[0])
    d = pf16.bn_desc(N, H, W, C, EPS, sbits, flags)
    ws = workspace(pf16.bn_workspace_size(d))
    tx, tg, tb = dev(x), dev(gamma), dev(beta)
    ty, tm, ti = empty16(R * C), empty16(C), empty16(C)
    tmask = torch.empty(R * C // 8, dtype=torch.uint8, device="cuda") if relu else None
    pf16.bn_fwd_bwd(d, 0, ws, x=tx, gamma=tg, beta=tb, residual=dev(resid) if res else None, y=ty,
                    mean=tm, invstd=ti, relu_mask=tmask)
    assert pf16.sync_status() == 0
    y = host(ty)
    if relu:  # the bit mask holds exactly the decisions y > 0
        bits = np.unpackbits(tmask.cpu().numpy(), bitorder="little").reshape(R, C)
        assert np.array_equal(bits.astype(bool), f64(y).reshape(R, C) > 0)
    yo, mean, var, invstd = orc.bn_fwd(x, gamma, beta, resid, R, C, EPS_F, s, relu)
    xhat = (f64(x).reshape(R, C) - mean) * invstd
    gf, bf = f64(gamma), f64(beta)
    scale = s * (np.abs(gf) * (np.abs(xhat) + 1) + np.abs(bf))
    if res:
        scale = scale + np.abs(f64(resid).reshape(R, C))
    tol = (4 * L + 8) * U * scale + 2.0 ** -24
    err = np.abs(f64(y).reshape(R, C) - yo)
    assert np.all(err <= tol), float(np.max(err / tol))
    # saved statistics
    assert np.all(np.abs(f64(host(tm)) - mean) <= (L + 2) * U * np.abs(f64(x).reshape(R, C)).max(0))
    assert np.all(np.abs(f64(host(ti)) - invstd) <= (2 * L + 8) * U * invstd)

    # backward, teacher-forced on the GPU's own saved output and statistics
    tdx, tdg, tdb, tdr = empty16(R * C), empty16(C), empty16(C), empty16(R * C)
    pf16.bn_fwd_bwd(d, 1, ws, x=tx, gamma=tg, mean=tm, invstd=ti, dy=dev(dy), y_saved=ty, dx=tdx,
                    dgamma=tdg, dbeta=tdb, dresidual=tdr)
    assert pf16.sync_status() == 0
    dxo, dgo, dbo, dro = orc.bn_bwd(x, gamma, dy, y, R, C, EPS_F, s, relu)
    assert np.array_equal(f64(host(tdr)).reshape(R, C), dro)  # masking is exact
    dyp = np.abs(dro)
    k = np.abs(s * gf * invstd)
    tol = (4 * L + 8) * U * k * (dyp + dyp.max(0) * (np.abs(xhat) + 1)) + 2.0 ** -24
    err = np.abs(f64(host(tdx)).reshape(R, C) - dxo)
    assert np.all(err <= tol), float(np.max(err / tol))
    tol_b = (4 * L + 8) * U * s * dyp.sum(0) + 2.0 ** -24
    tol_g = (4 * L + 8) * U * s * (dyp * (np.abs(xhat) + 1)).sum(0) + 2.0 ** -24
    assert np.all(np.abs(f64(host(tdb)) - dbo) <= tol_b)
    assert np.all(np.abs(f64(host(tdg)) - dgo) <= tol_g)
    if relu:  # the same backward reading the bit mask instead of y: bit-identical
        mdx, mdg, mdb, mdr = empty16(R * C), empty16(C), empty16(C), empty16(R * C)
        pf16.bn_fwd_bwd(d, 1, ws, x=tx, gamma=tg, mean=tm, invstd=ti, dy=dev(dy), relu_mask=tmask,
                        dx=mdx, dgamma=mdg, dbeta=mdb, dresidual=mdr)
        assert pf16.sync_status() == 0
        for a, b in ((mdx, tdx), (mdg, tdg), (mdb, tdb), (mdr, tdr)):
            assert np.array_equal(host(a), host(b))


def test_bn_constant_channel_and_zero_gamma(orc):
    """Closed forms: a constant channel normalises to 0 so y = s*beta; gamma = 0
    gives y = s*beta exactly too."""
    N, H, W, C = 2, 8, 8, 16
    R = N * H * W
    x = f16(np.tile(np.linspace(-3, 3, C), (R, 1)))
    gamma = f16(np.where(np.arange(C) % 2 == 0, 0.0, 1.5))
    beta = f16(np.linspace(-1, 1, C))
    d = pf16.bn_desc(N, H, W, C, EPS, 0x3400, 0)
    ws = workspace(pf16.bn_workspace_size(d))
    ty = empty16(R * C)
    pf16.bn_fwd_bwd(d, 0, ws, x=dev(x), gamma=dev(gamma), beta=dev(beta), y=ty, mean=empty16(C),
                    invstd=empty16(C))
    y = f64(host(ty)).reshape(R, C)
    assert np.array_equal(y, np.tile(0.25 * f64(beta), (R, 1)))


SWAP_CASES = [
    # N, H, W, C, relu
    (4, 14, 14, 256, True),
    (3, 5, 7, 24, False),        # ragged rows, no ReLU
    (256, 7, 7, 2048, True),     # a stage-4 block's last BatchNorm at batch 256
]


@pytest.mark.parametrize("case", SWAP_CASES, ids=lambda c: "N{}_{}x{}_C{}_relu{}".format(*c))
def test_bn_swap_fwd_bwd(orc, case):
    """PF16_BN_SWAP (Sec. 4.1's switch) against the oracle's swap BatchNorm.
    Forward bound (4L+8) u (|gamma| (s (|xhat|+1) + |r|) + |beta|) + 2^-24; the
    data gradient has the plain form; dresidual = rn(gamma dy') to one rounding;
    dbeta = sum dy', dgamma = s sum dy' xhat + sum dy' r within (4L+8) u sum|terms|."""
    N, H, W, C, relu = case
    R = N * H * W
    L = int(np.ceil(np.log2(R)))
    s = 0.25
    x = f16(f64(syn.normal_f16(31, (R, C), 2.0)) + 0.5)
    gamma = f16(1.0 + 0.1 * f64(syn.normal_f16(32, (C,))))
    beta = f16(0.1 * f64(syn.normal_f16(33, (C,))))
    resid = syn.normal_f16(34, (R, C))
    dy = syn.normal_f16(35, (R, C), 0.01)
    flags = pf16.PF16_BN_RESIDUAL | pf16.PF16_BN_SWAP | (pf16.PF16_BN_RELU if relu else 0)
    d = pf16.bn_desc(N, H, W, C, EPS, int(f16([s])[0]), flags)
    ws = workspace(pf16.bn_workspace_size(d))
    tx, tg, tb, tr = dev(x), dev(gamma), dev(beta), dev(resid)
    ty, tm, ti = empty16(R * C), empty16(C), empty16(C)
    tmask = torch.empty(R * C // 8, dtype=torch.uint8, device="cuda") if relu else None
    pf16.bn_fwd_bwd(d, 0, ws, x=tx, gamma=tg, beta=tb, residual=tr, y=ty, mean=tm, invstd=ti, relu_mask=tmask)
    assert pf16.sync_status() == 0
    y = host(ty)
    yo, mean, var, invstd = orc.bn_fwd_swap(x, gamma, beta, resid, R, C, EPS_F, s, relu)
    xhat = (f64(x).reshape(R, C) - mean) * invstd
    gf, bf, rf = f64(gamma), f64(beta), f64(resid).reshape(R, C)
    tol = (4 * L + 8) * U * (np.abs(gf) * (s * (np.abs(xhat) + 1) + np.abs(rf)) + np.abs(bf)) + 2.0 ** -24
    err = np.abs(f64(y).reshape(R, C) - yo)
    assert np.all(err <= tol), float(np.max(err / tol))

    tdx, tdg, tdb, tdr = empty16(R * C), empty16(C), empty16(C), empty16(R * C)
    pf16.bn_fwd_bwd(d, 1, ws, x=tx, gamma=tg, mean=tm, invstd=ti, dy=dev(dy), y_saved=ty, residual=tr,
                    relu_mask=tmask, dx=tdx, dgamma=tdg, dbeta=tdb, dresidual=tdr)
    assert pf16.sync_status() == 0
    dxo, dgo, dbo, dro = orc.bn_bwd_swap(x, gamma, dy, y, resid, R, C, EPS_F, s, relu)
    dz = np.abs(dro / np.where(gf == 0, 1, gf))  # |dy'|
    k = np.abs(s * gf * invstd)
    tol = (4 * L + 8) * U * k * (dz + dz.max(0) * (np.abs(xhat) + 1)) + 2.0 ** -24
    e = np.abs(f64(host(tdx)).reshape(R, C) - dxo)
    assert np.all(e <= tol), float(np.max(e / tol))
    e = np.abs(f64(host(tdr)).reshape(R, C) - dro)
    assert np.all(e <= U * np.abs(dro) + 2.0 ** -24), float(np.max(e))
    tol_b = (4 * L + 8) * U * dz.sum(0) + 2.0 ** -24
    tol_g = (4 * L + 8) * U * (s * (dz * (np.abs(xhat) + 1)).sum(0) + (dz * np.abs(rf)).sum(0)) + 2.0 ** -24
    assert np.all(np.abs(f64(host(tdb)) - dbo) <= tol_b), float(np.max(np.abs(f64(host(tdb)) - dbo) / tol_b))
    assert np.all(np.abs(f64(host(tdg)) - dgo) <= tol_g), float(np.max(np.abs(f64(host(tdg)) - dgo) / tol_g))
