"""Pins for the oracle's BatchNorm (Eq. 1, Eq. 2, batch statistics) with the
x0.25 output scaling inside residual blocks (Sec. 4.2), residual add and ReLU.

Checks: closed forms (constant channel, gamma = 0), the normalisation
invariants (mean(xhat) = 0, var(xhat) = var/(var+eps)), the backward
invariants (sum dx = 0; sum dx*xhat = gamma*invstd*dgamma*eps/(var+eps), which
is 0 for eps = 0), and a central finite-difference
check of the backward against the forward on inputs whose perturbations are
exact in binary16.  The swap variant of a block's last BatchNorm (Sec. 4.1,
gamma * (s * xhat + r) + beta) is pinned by its reduction to the plain one at
gamma = 1, beta = 0, its closed forms (constant channel, gamma = 0) and the
same finite-difference check, which also covers the residual gradient."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import synthetic as syn

EPS = float(np.uint16(0x00A8).view(np.float16))  # 1e-5 rounded to binary16 (subnormal)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


def test_eps_constant():
    assert EPS == 168 * 2.0 ** -24


def test_constant_channel_gives_s_beta(orc):
    R, C = 64, 3
    x = f16(np.tile([1.5, -2.0, 0.0], (R, 1)))
    gamma, beta = f16([2.0, -1.0, 0.5]), f16([0.25, -0.75, 1.0])
    y, mean, var, invstd = orc.bn_fwd(x, gamma, beta, None, R, C, EPS, 0.25, False)
    assert np.array_equal(var, np.zeros(C))
    assert np.allclose(y, np.tile(0.25 * np.array([0.25, -0.75, 1.0]), (R, 1)), rtol=0, atol=0)
    assert np.allclose(invstd, 1 / np.sqrt(EPS))


def test_gamma_zero_gives_s_beta(orc):
    R, C = 100, 4
    x = syn.normal_f16(3, (R, C))
    gamma, beta = f16([0, 0, 0, 0]), f16([1.0, -2.0, 0.5, 0.0])
    y, *_ = orc.bn_fwd(x, gamma, beta, None, R, C, EPS, 0.25, False)
    assert np.array_equal(y, np.tile(0.25 * np.array([1.0, -2.0, 0.5, 0.0]), (R, 1)))


def test_normalisation_invariants(orc):
    R, C = 777, 5
    x = syn.normal_f16(4, (R, C), 3.0)
    ones, zeros = f16(np.ones(C)), f16(np.zeros(C))
    xhat, mean, var, invstd = orc.bn_fwd(x, ones, zeros, None, R, C, EPS, 1.0, False)
    xf = x.view(np.float16).astype(np.float64)
    assert np.allclose(mean, xf.mean(0), rtol=1e-14, atol=1e-14)
    assert np.allclose(var, xf.var(0), rtol=1e-13)
    assert np.allclose(xhat.mean(0), 0, atol=1e-13)
    assert np.allclose(xhat.var(0), var / (var + EPS), rtol=1e-12)


def test_residual_and_relu(orc):
    R, C = 50, 2
    x = syn.normal_f16(5, (R, C))
    res = syn.normal_f16(6, (R, C))
    g, b = f16([1.0, 0.5]), f16([0.0, 0.25])
    y0, *_ = orc.bn_fwd(x, g, b, None, R, C, EPS, 0.25, False)
    y1, *_ = orc.bn_fwd(x, g, b, res, R, C, EPS, 0.25, True)
    rf = res.view(np.float16).astype(np.float64).reshape(R, C)
    assert np.allclose(y1, np.maximum(y0 + rf, 0.0), rtol=0, atol=1e-15)


def _grid_x(seed, R, C):
    # values k * 2^-6 in [-1, 1): x +- 2^-10 is exact in binary16
    k = np.floor(syn.uniform(seed, R * C) * 128).astype(np.int64) - 64
    return f16(k * 2.0 ** -6).reshape(R, C)


@pytest.mark.parametrize("s", [1.0, 0.25])
def test_backward_matches_finite_differences(orc, s):
    R, C = 24, 3
    x = _grid_x(7, R, C)
    gamma, beta = f16([1.0, 0.75, 1.25]), f16([0.5, -0.25, 0.0])
    u = syn.normal_f16(8, (R, C), 1.0)  # dL/dy
    uf = u.view(np.float16).astype(np.float64)

    def L(xb, gb=gamma, bb=beta):
        y, *_ = orc.bn_fwd(xb, gb, bb, None, R, C, EPS, s, False)
        return float(np.sum(y * uf))

    dx, dg, db, _ = orc.bn_bwd(x, gamma, u, None, R, C, EPS, s, False)
    h = 2.0 ** -10
    xf = x.view(np.float16).astype(np.float64)
    for i in [0, 5, 17, 40, 71]:
        r, c = divmod(i, C)
        xp, xm = xf.copy(), xf.copy()
        xp[r, c] += h
        xm[r, c] -= h
        fd = (L(f16(xp)) - L(f16(xm))) / (2 * h)
        assert abs(fd - dx[r, c]) <= 2e-4 * (np.abs(dx).max() + 1e-30), (i, fd, dx[r, c])
    gf = gamma.view(np.float16).astype(np.float64)
    bf = beta.view(np.float16).astype(np.float64)
    for c in range(C):
        gp, gm, bp, bm = gf.copy(), gf.copy(), bf.copy(), bf.copy()
        gp[c] += h
        gm[c] -= h
        bp[c] += h
        bm[c] -= h
        fdg = (L(x, f16(gp), beta) - L(x, f16(gm), beta)) / (2 * h)
        fdb = (L(x, gamma, f16(bp)) - L(x, gamma, f16(bm))) / (2 * h)
        assert abs(fdg - dg[c]) <= 1e-6 * (abs(dg[c]) + 1), (c, fdg, dg[c])
        assert abs(fdb - db[c]) <= 1e-9 * (abs(db[c]) + 1), (c, fdb, db[c])


def test_backward_invariants(orc):
    R, C = 513, 4
    x = syn.normal_f16(9, (R, C), 2.0)
    dy = syn.normal_f16(10, (R, C), 0.01)
    gamma, _ = f16([1.0, -0.5, 2.0, 0.25]), None
    gf = gamma.view(np.float16).astype(np.float64)
    for eps in (EPS, 0.0):
        dx, dg, db, _ = orc.bn_bwd(x, gamma, dy, None, R, C, eps, 0.25, False)
        xhat, _, var, invstd = orc.bn_fwd(x, f16(np.ones(C)), f16(np.zeros(C)), None, R, C, eps, 1.0,
                                          False)
        scale = np.abs(dx).sum(0)
        assert np.all(np.abs(dx.sum(0)) <= 1e-12 * scale)
        # sum dx*xhat = gamma*invstd*dgamma * eps/(var+eps): zero exactly when eps = 0
        lhs = (dx * xhat).sum(0)
        rhs = gf * invstd * dg * eps / (var + eps)
        assert np.all(np.abs(lhs - rhs) <= 1e-12 * np.abs(dx * xhat).sum(0))


def test_relu_mask_and_residual_gradient(orc):
    R, C = 40, 2
    x = syn.normal_f16(11, (R, C))
    dy = syn.normal_f16(12, (R, C))
    y_saved = f16(np.where(np.arange(R * C).reshape(R, C) % 3 == 0, 0.0, 1.0))
    g = f16([1.0, 1.0])
    dx_m, dg_m, db_m, dres = orc.bn_bwd(x, g, dy, y_saved, R, C, EPS, 0.25, True)
    mask = y_saved.view(np.float16).astype(np.float64) > 0
    dyf = dy.view(np.float16).astype(np.float64)
    assert np.array_equal(dres, np.where(mask, dyf, 0.0))
    dy_masked = f16(np.where(mask, dyf, 0.0))
    dx_r, dg_r, db_r, _ = orc.bn_bwd(x, g, dy_masked, None, R, C, EPS, 0.25, False)
    assert np.array_equal(dx_m, dx_r) and np.array_equal(dg_m, dg_r) and np.array_equal(db_m, db_r)


# ------------------------------------------------------------ swap variant
def test_swap_with_unit_gamma_zero_beta_is_the_plain_batchnorm(orc):
    """gamma = 1, beta = 0: gamma*(s*xhat + r) + beta = s*(gamma*xhat + beta) + r, so the
    swap forward, dx and dres equal the plain ones, and dbeta = plain dbeta / s."""
    R, C, s = 96, 3, 0.25
    x = syn.normal_f16(21, (R, C))
    res = syn.normal_f16(22, (R, C))
    dy = syn.normal_f16(23, (R, C), 0.1)
    g, b = f16(np.ones(C)), f16(np.zeros(C))
    y0, *_ = orc.bn_fwd(x, g, b, res, R, C, EPS, s, True)
    y1, *_ = orc.bn_fwd_swap(x, g, b, res, R, C, EPS, s, True)
    assert np.array_equal(y0, y1)
    ys = f16(y0)
    dx0, dg0, db0, dr0 = orc.bn_bwd(x, g, dy, ys, R, C, EPS, s, True)
    dx1, dg1, db1, dr1 = orc.bn_bwd_swap(x, g, dy, ys, res, R, C, EPS, s, True)
    assert np.array_equal(dx0, dx1) and np.array_equal(dr0, dr1)
    assert np.allclose(db1, db0 / s, rtol=1e-15, atol=0)


def test_swap_constant_channel_and_zero_gamma(orc):
    """A constant channel has xhat = 0, so y = gamma*r + beta; gamma = 0 gives y = beta
    whatever x and r are (with the zero-gamma initialisation the block output is beta)."""
    R, C = 40, 2
    x = f16(np.tile([1.5, -2.0], (R, 1)))
    res = syn.normal_f16(24, (R, C))
    rf = res.view(np.float16).astype(np.float64).reshape(R, C)
    g, b = f16([2.0, -0.5]), f16([0.25, 1.0])
    y, *_ = orc.bn_fwd_swap(x, g, b, res, R, C, EPS, 0.25, False)
    assert np.allclose(y, rf * np.array([2.0, -0.5]) + np.array([0.25, 1.0]), rtol=0, atol=1e-15)
    x2 = syn.normal_f16(25, (R, C))
    y2, *_ = orc.bn_fwd_swap(x2, f16([0.0, 0.0]), b, res, R, C, EPS, 0.25, False)
    assert np.array_equal(y2, np.tile([0.25, 1.0], (R, 1)))


@pytest.mark.parametrize("s", [1.0, 0.25])
def test_swap_backward_matches_finite_differences(orc, s):
    R, C = 24, 3
    x = _grid_x(27, R, C)
    res = _grid_x(28, R, C)
    gamma, beta = f16([1.0, 0.75, 1.25]), f16([0.5, -0.25, 0.0])
    u = syn.normal_f16(29, (R, C), 1.0)
    uf = u.view(np.float16).astype(np.float64)

    def L(xb, gb=gamma, bb=beta, rb=res):
        y, *_ = orc.bn_fwd_swap(xb, gb, bb, rb, R, C, EPS, s, False)
        return float(np.sum(y * uf))

    dx, dg, db, dr = orc.bn_bwd_swap(x, gamma, u, None, res, R, C, EPS, s, False)
    h = 2.0 ** -10
    xf = x.view(np.float16).astype(np.float64)
    rf = res.view(np.float16).astype(np.float64)
    for i in [0, 5, 17, 40, 71]:
        r, c = divmod(i, C)
        xp, xm = xf.copy(), xf.copy()
        xp[r, c] += h
        xm[r, c] -= h
        fd = (L(f16(xp)) - L(f16(xm))) / (2 * h)
        assert abs(fd - dx[r, c]) <= 2e-4 * (np.abs(dx).max() + 1e-30), (i, fd, dx[r, c])
        rp, rm = rf.copy(), rf.copy()
        rp[r, c] += h
        rm[r, c] -= h
        fdr = (L(x, rb=f16(rp)) - L(x, rb=f16(rm))) / (2 * h)
        assert abs(fdr - dr[r, c]) <= 1e-9 * (abs(dr[r, c]) + 1), (i, fdr, dr[r, c])
    gf = gamma.view(np.float16).astype(np.float64)
    bf = beta.view(np.float16).astype(np.float64)
    for c in range(C):
        gp, gm, bp, bm = gf.copy(), gf.copy(), bf.copy(), bf.copy()
        gp[c] += h
        gm[c] -= h
        bp[c] += h
        bm[c] -= h
        fdg = (L(x, f16(gp), beta) - L(x, f16(gm), beta)) / (2 * h)
        fdb = (L(x, gamma, f16(bp)) - L(x, gamma, f16(bm))) / (2 * h)
        assert abs(fdg - dg[c]) <= 1e-6 * (abs(dg[c]) + 1), (c, fdg, dg[c])
        assert abs(fdb - db[c]) <= 1e-9 * (abs(db[c]) + 1), (c, fdb, db[c])
