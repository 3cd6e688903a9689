"""Pins for the oracle's convolutions (forward, data gradient, weight gradient
of the ResNet-50 layers, paper Sec. 5.1; FP16 values, Sec. 5.2).

Independent checks, none of which re-types the oracle's loops:
  * exact integer brute force: a binary16 value is an integer times 2^-24, so
    every product is an integer times 2^-48 and the sums are exact Python ints;
  * a delta kernel makes the forward pass a pure shift of x;
  * the adjoint identity <dy, fwd(x,w)> = <dgrad(dy,w), x> = <wgrad(x,dy), w>;
  * a 1x1 stride-1 convolution is a matrix product (numpy);
  * linearity in x for inputs with disjoint support.
"""
import itertools

import numpy as np
import pytest

from paper_1911_07384_gb300 import synthetic as syn


def _rand_f16(seed, shape, std=1.0):
    return syn.normal_f16(seed, shape, std)


def _ints(bits):
    """binary16 bits -> exact integers in units of 2^-24 (Python ints)."""
    v = bits.view(np.float16).astype(np.float64)
    return np.array([int(round(t * 2 ** 24)) for t in v.ravel()], dtype=object).reshape(bits.shape)


def _brute_fwd(xi, wi, stride, pad):
    N, H, W, C = xi.shape
    K, R, S, _ = wi.shape
    P, Q = (H + 2 * pad - R) // stride + 1, (W + 2 * pad - S) // stride + 1
    y = np.zeros((N, P, Q, K), dtype=object)
    a = np.zeros((N, P, Q, K), dtype=object)
    for n, p, q, k in itertools.product(range(N), range(P), range(Q), range(K)):
        acc = 0
        ab = 0
        for r, s, c in itertools.product(range(R), range(S), range(C)):
            h, w = p * stride + r - pad, q * stride + s - pad
            if 0 <= h < H and 0 <= w < W:
                t = xi[n, h, w, c] * wi[k, r, s, c]
                acc += t
                ab += abs(t)
        y[n, p, q, k] = acc
        a[n, p, q, k] = ab
    return y, a


def _brute_dgrad(dyi, wi, H, W, stride, pad):
    N, P, Q, K = dyi.shape
    _, R, S, C = wi.shape
    dx = np.zeros((N, H, W, C), dtype=object)
    # scatter form: every forward term x[n,h,w,c]*w[k,r,s,c] feeding y[n,p,q,k]
    for n, p, q, k in itertools.product(range(N), range(P), range(Q), range(K)):
        for r, s in itertools.product(range(R), range(S)):
            h, w = p * stride + r - pad, q * stride + s - pad
            if 0 <= h < H and 0 <= w < W:
                for c in range(C):
                    dx[n, h, w, c] += dyi[n, p, q, k] * wi[k, r, s, c]
    return dx


def _brute_wgrad(xi, dyi, R, S, stride, pad):
    N, H, W, C = xi.shape
    _, P, Q, K = dyi.shape
    dw = np.zeros((K, R, S, C), dtype=object)
    for n, p, q, k in itertools.product(range(N), range(P), range(Q), range(K)):
        for r, s in itertools.product(range(R), range(S)):
            h, w = p * stride + r - pad, q * stride + s - pad
            if 0 <= h < H and 0 <= w < W:
                for c in range(C):
                    dw[k, r, s, c] += dyi[n, p, q, k] * xi[n, h, w, c]
    return dw


def _close_exact(V, A, exact_int):
    exact = np.array([float(e) * 2.0 ** -48 for e in exact_int.ravel()])
    # binary64 summation error bound for the oracle's sequential sums
    bound = 64 * 2.0 ** -53 * np.maximum(A, 1e-300) + 1e-300
    assert np.all(np.abs(V - exact) <= bound), np.max(np.abs(V - exact) / bound)


SHAPES = [
    # N, H, W, C, K, R, S, stride, pad
    (1, 5, 4, 3, 2, 3, 3, 1, 1),
    (2, 5, 6, 2, 3, 3, 3, 2, 1),
    (1, 4, 4, 3, 2, 1, 1, 2, 0),
    (1, 7, 6, 2, 2, 7, 7, 2, 3),
    (2, 3, 3, 4, 3, 1, 1, 1, 0),
]


@pytest.mark.parametrize("shape", SHAPES)
def test_conv_fwd_exact_bruteforce(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x = _rand_f16(11, (N, H, W, C))
    w = _rand_f16(12, (K, R, S, C), 0.5)
    V, A, T = orc.conv_fwd(x, w, N, H, W, C, K, R, S, st, pd)
    yi, ai = _brute_fwd(_ints(x), _ints(w), st, pd)
    _close_exact(V, A, yi)
    assert np.allclose(A, np.array([float(t) * 2.0 ** -48 for t in ai.ravel()]), rtol=1e-14, atol=0)


@pytest.mark.parametrize("shape", SHAPES)
def test_conv_dgrad_exact_bruteforce(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = orc.conv_out_hw(H, W, R, S, st, pd)
    dy = _rand_f16(13, (N, P, Q, K))
    w = _rand_f16(14, (K, R, S, C), 0.5)
    V, A, T = orc.conv_dgrad(dy, w, N, H, W, C, K, R, S, st, pd)
    _close_exact(V, A, _brute_dgrad(_ints(dy), _ints(w), H, W, st, pd))


@pytest.mark.parametrize("shape", SHAPES)
def test_conv_wgrad_exact_bruteforce(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = orc.conv_out_hw(H, W, R, S, st, pd)
    x = _rand_f16(15, (N, H, W, C))
    dy = _rand_f16(16, (N, P, Q, K))
    V, A, T = orc.conv_wgrad(x, dy, N, H, W, C, K, R, S, st, pd)
    _close_exact(V, A, _brute_wgrad(_ints(x), _ints(dy), R, S, st, pd))
    # every (n,p,q) counts once per output, in range or not
    assert np.all(T <= N * P * Q)


def test_sampled_outputs_equal_full(orc):
    N, H, W, C, K, R, S, st, pd = 2, 9, 7, 16, 8, 3, 3, 2, 1
    P, Q = orc.conv_out_hw(H, W, R, S, st, pd)
    x = _rand_f16(21, (N, H, W, C))
    w = _rand_f16(22, (K, R, S, C))
    dy = _rand_f16(23, (N, P, Q, K))
    rng = np.random.default_rng(0)
    for fn, a, b, total in ((orc.conv_fwd, x, w, N * P * Q * K), (orc.conv_dgrad, dy, w, N * H * W * C),
                            (orc.conv_wgrad, x, dy, K * R * S * C)):
        Vf, Af, Tf = fn(a, b, N, H, W, C, K, R, S, st, pd)
        idx = rng.integers(0, total, 50)
        Vs, As, Ts = fn(a, b, N, H, W, C, K, R, S, st, pd, idx=idx)
        assert np.array_equal(Vs, Vf[idx]) and np.array_equal(As, Af[idx]) and np.array_equal(Ts, Tf[idx])


@pytest.mark.parametrize("r0,s0", [(0, 0), (1, 1), (2, 0), (0, 2)])
def test_delta_kernel_is_shift(orc, r0, s0):
    N, H, W, C = 2, 6, 5, 8
    K, R, S, pad = C, 3, 3, 1
    x = _rand_f16(31, (N, H, W, C))
    w = np.zeros((K, R, S, C), np.float16)
    for k in range(K):
        w[k, r0, s0, k] = 1.0
    V, _, _ = orc.conv_fwd(x, w.view(np.uint16), N, H, W, C, K, R, S, 1, pad)
    y = V.reshape(N, H, W, K)
    xf = x.view(np.float16).astype(np.float64)
    ref = np.zeros_like(y)
    for h in range(H):
        for ww in range(W):
            hh, wq = h + r0 - pad, ww + s0 - pad
            if 0 <= hh < H and 0 <= wq < W:
                ref[:, h, ww, :] = xf[:, hh, wq, :]
    assert np.array_equal(y, ref)


@pytest.mark.parametrize("shape", [(2, 9, 9, 16, 24, 3, 3, 1, 1), (2, 10, 10, 16, 8, 3, 3, 2, 1),
                                   (1, 8, 8, 32, 16, 1, 1, 2, 0), (1, 15, 15, 3, 8, 7, 7, 2, 3)])
def test_adjoint_identity(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = orc.conv_out_hw(H, W, R, S, st, pd)
    x = _rand_f16(41, (N, H, W, C))
    w = _rand_f16(42, (K, R, S, C))
    dy = _rand_f16(43, (N, P, Q, K))
    f = lambda a: a.view(np.float16).astype(np.float64).ravel()
    y, _, _ = orc.conv_fwd(x, w, N, H, W, C, K, R, S, st, pd)
    dx, _, _ = orc.conv_dgrad(dy, w, N, H, W, C, K, R, S, st, pd)
    dw, _, _ = orc.conv_wgrad(x, dy, N, H, W, C, K, R, S, st, pd)
    a1 = np.dot(f(dy), y)
    a2 = np.dot(dx, f(x))
    a3 = np.dot(dw, f(w))
    scale = np.dot(np.abs(f(dy)), np.abs(y)) + 1e-300
    assert abs(a1 - a2) / scale < 1e-12
    assert abs(a1 - a3) / scale < 1e-12


def test_1x1_conv_is_matmul(orc):
    N, H, W, C, K = 2, 7, 5, 24, 40
    x = _rand_f16(51, (N, H, W, C))
    w = _rand_f16(52, (K, 1, 1, C))
    V, A, T = orc.conv_fwd(x, w, N, H, W, C, K, 1, 1, 1, 0)
    xf = x.view(np.float16).astype(np.float64).reshape(-1, C)
    wf = w.view(np.float16).astype(np.float64).reshape(K, C)
    assert np.allclose(V, (xf @ wf.T).ravel(), rtol=0, atol=1e-12)
    assert np.allclose(A, (np.abs(xf) @ np.abs(wf).T).ravel(), rtol=1e-13)
    assert np.all(T == C)


def test_linearity_in_x(orc):
    N, H, W, C, K, R, S = 1, 6, 6, 8, 8, 3, 3
    x = _rand_f16(61, (N, H, W, C))
    w = _rand_f16(62, (K, R, S, C))
    mask = (np.arange(x.size).reshape(x.shape) % 3) == 0
    x1 = np.where(mask, x, np.uint16(0))
    x2 = np.where(mask, np.uint16(0), x)
    y, _, _ = orc.conv_fwd(x, w, N, H, W, C, K, R, S, 1, 1)
    y1, _, _ = orc.conv_fwd(x1, w, N, H, W, C, K, R, S, 1, 1)
    y2, _, _ = orc.conv_fwd(x2, w, N, H, W, C, K, R, S, 1, 1)
    assert np.allclose(y, y1 + y2, rtol=0, atol=1e-12)


def test_dgrad_term_counts(orc):
    # 3x3 stride 2 pad 1: interior rows of dx get 1 or 2 taps per axis
    N, H, W, C, K, R, S, st, pd = 1, 8, 8, 8, 8, 3, 3, 2, 1
    P, Q = orc.conv_out_hw(H, W, R, S, st, pd)
    dy = _rand_f16(71, (N, P, Q, K))
    w = _rand_f16(72, (K, R, S, C))
    _, _, T = orc.conv_dgrad(dy, w, N, H, W, C, K, R, S, st, pd)
    T = T.reshape(N, H, W, C)[0, :, :, 0]
    taps = lambda h: sum(1 for r in range(R) if (h + pd - r) % st == 0 and 0 <= (h + pd - r) // st < P)
    ref = np.array([[taps(h) * taps(w) * K for w in range(W)] for h in range(H)])
    assert np.array_equal(T, ref)
