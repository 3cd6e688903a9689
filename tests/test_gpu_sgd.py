"""GPU parity of pf16_sgd_update: bit-exact against the oracle's FP16
emulation (NaNs compared as NaN), including the config-1 weights, the
underflow-stress sequence and ragged tails."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev, host

pytestmark = pytest.mark.gpu

LR, MOM, WD = 0x2E66, 0x3B33, 0x068E


def same(a, b):
    fa, fb = a.view(np.float16), b.view(np.float16)
    nan = np.isnan(fa)
    return np.array_equal(nan, np.isnan(fb)) and np.array_equal(a[~nan], b[~nan])


@pytest.mark.parametrize("n", [36864, 1, 7, 8, 9, 4099, 1_000_003])
@pytest.mark.parametrize("wd", [WD, 0x0000])
def test_sgd_bit_exact(orc, n, wd):
    w = syn.he_normal_f16(syn.seed_for(1, "w"), 1, 1, 1, n).ravel()
    v = syn.normal_f16(syn.seed_for(1, "v"), (n,), 0.01)
    g = syn.normal_f16(syn.seed_for(1, "dy"), (n,), 0.05)
    ew, ev = orc.sgd_update(w, v, g, LR, MOM, wd)
    tw, tv, tg = dev(w), dev(v), dev(g)
    pf16.sgd_update(tw, tv, tg, LR, MOM, wd)
    assert pf16.sync_status() == 0
    assert same(host(tw), ew) and same(host(tv), ev)


def test_sgd_stress_sequence(orc):
    """Config 5: weights near 1, log-uniform gradients over [2^-24, 2^4],
    ten steps; many updates fall below half an ulp and must stagnate."""
    n = 1 << 16
    w = syn.near_one_f16(syn.seed_for(5, "w"), (n,))
    v = np.zeros(n, np.uint16)
    tw, tv = dev(w), dev(v)
    ew, ev = w, v
    for step in range(10):
        g = syn.loguniform_pm_f16(syn.seed_for(5, "dy", step), (n,))
        ew, ev = orc.sgd_update(ew, ev, g, LR, MOM, WD)
        pf16.sgd_update(tw, tv, dev(g), LR, MOM, WD)
        assert same(host(tw), ew) and same(host(tv), ev), step
    assert pf16.sync_status() == 0


def test_sgd_specials(orc):
    w = np.float16([1.0, -0.0, 0.0, np.inf, 65504, 6e-8, -1.0, 0.5]).view(np.uint16)
    v = np.float16([0.0, -0.0, 1.0, 0.0, 65504, -6e-8, np.nan, 0.25]).view(np.uint16)
    g = np.float16([np.inf, -0.0, -0.0, 1.0, 65504, 6e-8, 1.0, 0.125]).view(np.uint16)
    for wd in (WD, 0):
        ew, ev = orc.sgd_update(w, v, g, LR, MOM, wd)
        tw, tv = dev(w), dev(v)
        pf16.sgd_update(tw, tv, dev(g), LR, MOM, wd)
        assert same(host(tw), ew) and same(host(tv), ev)
