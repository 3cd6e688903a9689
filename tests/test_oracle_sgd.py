"""Pins for the oracle's pure-FP16 SGD step (PyTorch ImageNet recipe adopted in
paper Sec. 5.1: momentum, coupled weight decay, no dampening, no Nesterov; no
master copy and FP16 arithmetic throughout, Sec. 5.2; the small-update
stagnation of Sec. 2).  Checked against numpy's independent float16
arithmetic and against hand-worked cases."""
import numpy as np

LR, MOM, WD = 0x2E66, 0x3B33, 0x068E  # 0.1, 0.9, 1e-4 rounded to binary16


def _np_step(w, v, g, lr, mom, wd):
    f = lambda b: np.asarray(b, np.uint16).view(np.float16)
    w16, v16, g16 = f(w), f(v), f(g)
    lr16, mom16, wd16 = f(np.uint16(lr)), f(np.uint16(mom)), f(np.uint16(wd))
    with np.errstate(all="ignore"):
        if wd != 0:
            g16 = g16 + wd16 * w16
        v2 = mom16 * v16 + g16
        w2 = w16 - lr16 * v2
    return w2.view(np.uint16), v2.view(np.uint16)


def _same(a, b):
    fa, fb = a.view(np.float16), b.view(np.float16)
    nan = np.isnan(fa)
    return np.array_equal(nan, np.isnan(fb)) and np.array_equal(a[~nan], b[~nan])


def test_matches_numpy_float16_random(orc):
    rng = np.random.default_rng(5)
    n = 200_000
    w = (rng.standard_normal(n) * 0.05).astype(np.float16).view(np.uint16)
    v = (rng.standard_normal(n) * 0.01).astype(np.float16).view(np.uint16)
    g = (rng.standard_normal(n) * np.exp2(rng.uniform(-26, 2, n))).astype(np.float16).view(np.uint16)
    for wd in (WD, 0x0000):
        ow, ov = orc.sgd_update(w, v, g, LR, MOM, wd)
        rw, rv = _np_step(w, v, g, LR, MOM, wd)
        assert _same(ow, rw) and _same(ov, rv)


def test_multi_step_sequence(orc):
    rng = np.random.default_rng(6)
    n = 4096
    w = (1.0 + rng.integers(-8, 9, n) * 2.0 ** -10).astype(np.float16).view(np.uint16)
    v = np.zeros(n, np.uint16)
    ow, ov, rw, rv = w, v, w, v
    for step in range(10):
        g = (np.where(rng.random(n) < 0.5, -1, 1) * np.exp2(rng.uniform(-24, 4, n))).astype(
            np.float16).view(np.uint16)
        ow, ov = orc.sgd_update(ow, ov, g, LR, MOM, WD)
        rw, rv = _np_step(rw, rv, g, LR, MOM, WD)
        assert _same(ow, rw) and _same(ov, rv), step


def test_stagnation_below_half_ulp(orc):
    # w = 1: the ulp above 1 is 2^-10, so |lr*v'| < 2^-12 (half the ulp below 1) leaves w unchanged
    w = np.array([0x3C00] * 3, np.uint16)
    v = np.zeros(3, np.uint16)
    g = np.float16([2.0 ** -12, -2.0 ** -12, 2.0 ** -20]).view(np.uint16)
    ow, ov = orc.sgd_update(w, v, g, LR, MOM, 0)
    assert np.array_equal(ow, w)
    assert np.array_equal(ov, g)  # v' = 0.9*0 + g


def test_weight_decay_zero_is_skipped(orc):
    # wd = +0 must not form 0*w: with w = inf that product would be NaN
    w = np.float16([np.inf]).view(np.uint16)
    v = np.zeros(1, np.uint16)
    g = np.float16([0.5]).view(np.uint16)
    ow, ov = orc.sgd_update(w, v, g, LR, MOM, 0)
    assert ov[0] == np.float16(0.5).view(np.uint16)
    assert ow[0] == 0x7C00


def test_inf_nan_propagate(orc):
    w = np.float16([1.0, 1.0, 1.0]).view(np.uint16)
    v = np.zeros(3, np.uint16)
    g = np.float16([np.inf, -np.inf, np.nan]).view(np.uint16)
    ow, ov = orc.sgd_update(w, v, g, LR, MOM, WD)
    f = ow.view(np.float16)
    assert f[0] == -np.inf and f[1] == np.inf and np.isnan(f[2])


def test_signed_zero_cases(orc):
    w = np.array([0x8000, 0x0000, 0x8000], np.uint16)   # -0, +0, -0
    v = np.array([0x0000, 0x8000, 0x8000], np.uint16)
    g = np.array([0x0000, 0x8000, 0x8000], np.uint16)
    ow, ov = orc.sgd_update(w, v, g, LR, MOM, 0)
    # v' = mom*v + g: +0+(+0)=+0; -0+(-0)=-0; -0+(-0)=-0
    assert list(ov) == [0x0000, 0x8000, 0x8000]
    # w' = w - lr*v': -0 - (+0) = -0; +0 - (-0) = +0; -0 - (-0) = +0
    assert list(ow) == [0x8000, 0x0000, 0x0000]


def test_hand_worked_single_element(orc):
    # w=0.5, v=0.25, g=0.125, lr=0x2E66, mom=0x3B33, wd=0x068E (each product rounded once)
    w, v, g = np.float16([0.5]).view(np.uint16), np.float16([0.25]).view(np.uint16), np.float16([0.125]).view(np.uint16)
    ow, ov = orc.sgd_update(w, v, g, LR, MOM, WD)
    mom = 0.89990234375
    lr = 0.0999755859375
    wd = np.float16(np.uint16(WD).view(np.float16)).astype(np.float64)
    t1 = float(np.float16(wd * 0.5))
    g2 = float(np.float16(0.125 + t1))
    t2 = float(np.float16(mom * 0.25))
    v2 = float(np.float16(t2 + g2))
    t3 = float(np.float16(lr * v2))
    w2 = float(np.float16(0.5 - t3))
    assert ov.view(np.float16)[0] == v2 and ow.view(np.float16)[0] == w2
    # worked by hand in exact rationals: v2 = 1434 * 2^-12 (tie 1433.5 -> even), w2 = 1905 * 2^-12
    assert v2 == 0.35009765625 and w2 == 0.465087890625
