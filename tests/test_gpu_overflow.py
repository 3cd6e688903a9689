"""Overflow in the FP16 accumulation (the paper keeps IEEE binary16 arithmetic
throughout, Sec. 3, where a result beyond the largest finite value rounds to
infinity): inputs whose exact sums exceed the binary16 range by far more than
any accumulation order's rounding can hide must give infinities of the right
sign in every conv pass, as the oracle's exact sums rounded to binary16 do.
NaN inputs reach exactly the outputs whose terms include them."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import pf16
from gpu_util import dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

SHAPES = [(1, 8, 8, 64, 64, 3, 3, 1, 1),     # halo engine
          (1, 8, 8, 128, 128, 3, 3, 1, 1),   # im2col GEMM, 128-wide N tile
          (2, 7, 7, 256, 64, 1, 1, 1, 0)]    # dense 1x1

BIG = np.float16(64.0).view(np.uint16)      # products 4096; >= 64 terms per output here


def ids(s):
    return "N{}_{}x{}_C{}_K{}_{}x{}_s{}p{}".format(*s)


def passes(shape, x, w, dy):
    N, H, W, C, K, R, S, st, pd = shape
    d = pf16.conv_desc(*shape)
    P, Q = d.out_hw()
    y, dx, dw = empty16(N * P * Q * K), empty16(N * H * W * C), empty16(K * R * S * C)
    pf16.conv_fwd(d, dev(x), dev(w), y, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_FWD)))
    pf16.conv_dgrad(d, dev(dy), dev(w), dx)
    pf16.conv_wgrad(d, dev(x), dev(dy), dw, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)))
    assert pf16.sync_status() == 0
    return f64(host(y)), f64(host(dx)), f64(host(dw))


@pytest.mark.parametrize("sign", [1, -1], ids=["pos", "neg"])
@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_overflow_gives_signed_infinity(orc, shape, sign):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    big = BIG if sign > 0 else BIG | 0x8000
    x = np.full((N, H, W, C), big, np.uint16)
    w = np.full((K, R, S, C), BIG, np.uint16)
    dy = np.full((N, P, Q, K), BIG, np.uint16)
    got = passes(shape, x, w, dy)
    exact = (orc.conv_fwd(x, w, *shape)[0], orc.conv_dgrad(dy, w, *shape)[0], orc.conv_wgrad(x, dy, *shape)[0])
    # An FP16 sum of n same-sign terms, in any order, is at least exact / (1 + u)^n
    # (u = 2^-11); every exact sum here stays at or above 65520 (the smallest
    # value that rounds to infinity) after that factor, so every pass must overflow.
    for g, V, n, what in zip(got, exact, (C * R * S, K * R * S, N * P * Q), ("fwd", "dgrad", "wgrad")):
        assert np.all(np.abs(V) >= 65520.0 * (1 + 2.0 ** -11) ** n), what
        want = np.sign(V) * np.inf
        assert np.array_equal(g.ravel(), want.ravel()), (what, g.ravel()[:4])


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_nan_reaches_exactly_its_outputs(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    one = np.float16(1.0).view(np.uint16)
    x = np.full((N, H, W, C), one, np.uint16)
    x[0, H // 2, W // 2, 5] = 0x7E00  # one quiet NaN
    w = np.full((K, R, S, C), np.float16(2.0 ** -6).view(np.uint16), np.uint16)
    dy = np.full((N, P, Q, K), np.float16(2.0 ** -6).view(np.uint16), np.uint16)
    y, _, dw = passes(shape, x, w, dy)
    # forward: NaN exactly at outputs whose window covers pixel (H/2, W/2), every channel
    Vy = orc.conv_fwd(x, w, *shape)[0]
    assert np.array_equal(np.isnan(y.ravel()), np.isnan(Vy)), "fwd"
    Vw = orc.conv_wgrad(x, dy, *shape)[0]
    assert np.array_equal(np.isnan(dw.ravel()), np.isnan(Vw)), "wgrad"
    assert np.isnan(Vy).any() and (~np.isnan(Vy)).any()
