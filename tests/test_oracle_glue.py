"""Pins for the oracle's pooling and loss (the rest of the ResNet-50 training
step, paper Sec. 5.1): numpy sliding-window max, adjoint identities,
closed forms (uniform logits give ln K) and finite differences."""
import numpy as np

from paper_1911_07384_gb300 import synthetic as syn


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


def test_maxpool_fwd_matches_numpy_windows(orc):
    N, H, W, C = 2, 11, 8, 5
    x = syn.normal_f16(1, (N, H, W, C))
    y = orc.maxpool_fwd(x, N, H, W, C)
    xf = x.view(np.float16).astype(np.float64)
    pad = np.pad(xf, ((0, 0), (1, 1), (1, 1), (0, 0)), constant_values=-np.inf)
    win = np.lib.stride_tricks.sliding_window_view(pad, (3, 3), axis=(1, 2))[:, ::2, ::2]
    assert np.array_equal(y, win.max(axis=(-1, -2)).ravel())


def test_maxpool_bwd_adjoint_and_ties(orc):
    N, H, W, C = 2, 9, 10, 3
    x = syn.normal_f16(2, (N, H, W, C))
    P, Q = orc.conv_out_hw(H, W, 3, 3, 2, 1)
    dy = syn.normal_f16(3, (N, P, Q, C))
    y = orc.maxpool_fwd(x, N, H, W, C)
    dx, A = orc.maxpool_bwd(x, dy, N, H, W, C)
    f = lambda a: a.view(np.float16).astype(np.float64).ravel()
    assert abs(np.dot(f(dy), y) - np.dot(dx, f(x))) <= 1e-12 * np.dot(np.abs(f(dy)), np.abs(y))
    # all-equal input: each window's gradient goes to its first (top-left) valid cell
    xe = f16(np.ones((1, 5, 5, 1)))
    dye = f16(np.ones((1, 3, 3, 1)))
    dxe, _ = orc.maxpool_bwd(xe, dye, 1, 5, 5, 1)
    ref = np.zeros((5, 5))
    for p in range(3):
        for q in range(3):
            ref[max(2 * p - 1, 0), max(2 * q - 1, 0)] += 1
    assert np.array_equal(dxe.reshape(5, 5), ref)


def test_avgpool(orc):
    N, HW, C = 3, 49, 6
    x = syn.normal_f16(4, (N, HW, C))
    dy = syn.normal_f16(5, (N, C))
    y = orc.avgpool_fwd(x, N, HW, C)
    dx = orc.avgpool_bwd(dy, N, HW, C)
    f = lambda a: a.view(np.float16).astype(np.float64).ravel()
    assert np.allclose(y, f(x).reshape(N, HW, C).mean(1).ravel(), rtol=1e-14)
    assert abs(np.dot(f(dy), y) - np.dot(dx, f(x))) <= 1e-12 * np.dot(np.abs(f(dy)), np.abs(y))
    const = f16(np.full((1, HW, 2), 0.375))
    assert np.array_equal(orc.avgpool_fwd(const, 1, HW, 2), [0.375, 0.375])


def test_softmax_xent_uniform_logits(orc):
    B, K = 4, 1000
    loss, dl, db = orc.softmax_xent(np.zeros(B * K, np.uint16), np.zeros(K, np.uint16),
                                    np.array([0, 5, 999, 17]), B, K)
    assert abs(loss - np.log(K)) < 1e-14
    dl = dl.reshape(B, K)
    assert np.allclose(dl.sum(1), 0, atol=1e-15)
    assert abs(dl[0, 0] - (1 / K - 1) / B) < 1e-16 and abs(dl[0, 1] - 1 / K / B) < 1e-18
    assert np.allclose(db, dl.sum(0), rtol=0, atol=1e-16)


def test_softmax_xent_finite_differences(orc):
    B, K = 3, 10
    k = np.floor(syn.uniform(6, B * K) * 64).astype(np.int64) - 32
    logits = f16(k * 2.0 ** -4)            # |l| <= 2: l +- 2^-8 exact
    bias = f16(np.linspace(-0.5, 0.5, K))
    labels = np.array([3, 0, 9])
    loss, dl, db = orc.softmax_xent(logits, bias, labels, B, K)
    lf = logits.view(np.float16).astype(np.float64)
    h = 2.0 ** -8
    for i in [0, 4, 13, 29]:
        lp, lm = lf.copy(), lf.copy()
        lp[i] += h
        lm[i] -= h
        fd = (orc.softmax_xent(f16(lp), bias, labels, B, K)[0] -
              orc.softmax_xent(f16(lm), bias, labels, B, K)[0]) / (2 * h)
        assert abs(fd - dl[i]) < 1e-5, (i, fd, dl[i])
