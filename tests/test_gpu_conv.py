"""GPU parity of the tcgen05 convolutions (forward, data gradient, weight
gradient) against the oracle on the same seeded binary16 inputs.

Bound (the contract): |gpu - oracle| <= 4 * sqrt(R) * 2^-11 * sum|terms| per
element, R = the reduction length (C*R*S forward, the number of contributing
(k, r, s) terms for the data gradient, N*P*Q for the weight gradient).
Single-term cases (delta kernel, delta gradient) must be bit-exact."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import U, assert_conv_close, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

SHAPES = [
    # N, H, W, C, K, R, S, stride, pad
    (4, 56, 56, 64, 64, 3, 3, 1, 1),     # config 1 (halo engine: padded rows of 64)
    (2, 28, 28, 64, 64, 3, 3, 1, 1),     # halo engine, padded rows of 32
    (3, 16, 30, 64, 64, 3, 3, 1, 1),     # halo engine, W + 2 = 32 exactly
    (1, 7, 7, 64, 64, 3, 3, 1, 1),       # one partial M tile
    (2, 9, 9, 64, 128, 3, 3, 2, 1),      # strided 3x3, odd size: unequal stride phases
    (3, 14, 14, 128, 128, 3, 3, 2, 1),   # strided 3x3, even size: the four phases in one launch, ragged M tile
    (2, 10, 12, 192, 64, 3, 3, 2, 1),    # the same with H != W and a partial N tile
    (2, 14, 14, 256, 64, 1, 1, 1, 0),    # 1x1 GEMM
    (2, 14, 14, 64, 256, 1, 1, 1, 0),
    (2, 13, 13, 128, 256, 1, 1, 2, 0),   # strided 1x1 projection, odd size
    (3, 10, 10, 192, 320, 3, 3, 1, 1),   # 3 channel chunks, partial N tile
    (2, 32, 32, 3, 64, 7, 7, 2, 3),      # stem, space-to-depth halo (rows of 32)
    (3, 30, 30, 3, 64, 7, 7, 2, 3),      # stem, s2d halo, odd P = 15 (rows of 128)
    (2, 100, 98, 3, 64, 7, 7, 2, 3),     # stem, s2d halo (rows of 64), H != W
    (2, 31, 29, 3, 64, 7, 7, 2, 3),      # stem, odd H and W
    (2, 20, 20, 3, 128, 7, 7, 2, 3),     # stem with 128 outputs: patch GEMM
    (2, 16, 16, 3, 64, 3, 3, 1, 1),      # c = 3, 3x3: patch GEMM
    (16, 1, 1, 2048, 1000, 1, 1, 1, 0),  # fully connected layer
    (2, 28, 28, 128, 128, 3, 3, 1, 1),   # wide halo forward, one image per padded row of 32
    (4, 14, 14, 256, 256, 3, 3, 1, 1),   # wide halo forward, four images per padded row of 64
    (4, 12, 12, 128, 256, 3, 3, 1, 1),   # wide halo forward, four images, W = 12, C != K
    (2, 12, 24, 192, 128, 3, 3, 1, 1),   # wide halo forward, W = 24 of 32, three input chunks
]


def ids(s):
    return "N{}_{}x{}_C{}_K{}_{}x{}_s{}p{}".format(*s)


def inputs(shape, seed_cfg=1):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    x = syn.normal_f16(syn.seed_for(seed_cfg, "x"), (N, H, W, C))
    w = syn.he_normal_f16(syn.seed_for(seed_cfg, "w"), K, R, S, C)
    dy = syn.normal_f16(syn.seed_for(seed_cfg, "dy"), (N, P, Q, K), 0.01)
    return x, w, dy, P, Q


def run_fwd(d, x, w, flags=0, y0=None):
    y = dev(y0) if y0 is not None else empty16(d.n * d.out_hw()[0] * d.out_hw()[1] * d.k)
    ws = workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_FWD))
    pf16.conv_fwd(d, dev(x), dev(w), y, ws, flags)
    assert pf16.sync_status() == 0
    return host(y)


def run_dgrad(d, dy, w, flags=0, dx0=None):
    dx = dev(dx0) if dx0 is not None else empty16(d.n * d.h * d.w * d.c)
    pf16.conv_dgrad(d, dev(dy), dev(w), dx, None, flags)
    assert pf16.sync_status() == 0
    return host(dx)


def run_wgrad(d, x, dy):
    dw = empty16(d.k * d.r * d.s * d.c)
    ws = workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD))
    pf16.conv_wgrad(d, dev(x), dev(dy), dw, ws)
    assert pf16.sync_status() == 0
    return host(dw)


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_conv_fwd(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape)
    d = pf16.conv_desc(*shape)
    y = run_fwd(d, x, w)
    V, A, T = orc.conv_fwd(x, w, *shape)
    rel = assert_conv_close(y, V, A, C * R * S, "fwd")
    assert rel < 2.0 ** -7, rel


@pytest.mark.parametrize("shape", [s for s in SHAPES if s[3] != 3], ids=ids)
def test_conv_dgrad(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape)
    d = pf16.conv_desc(*shape)
    dx = run_dgrad(d, dy, w)
    V, A, T = orc.conv_dgrad(dy, w, *shape)
    rel = assert_conv_close(dx, V, A, np.maximum(T, 1), "dgrad")
    assert rel < 2.0 ** -7, rel


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_conv_wgrad(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape)
    d = pf16.conv_desc(*shape)
    dw = run_wgrad(d, x, dy)
    V, A, T = orc.conv_wgrad(x, dy, *shape)
    rel = assert_conv_close(dw, V, A, N * P * Q, "wgrad")
    assert rel < 2.0 ** -6, rel


def test_stem_full_width_sampled(orc):
    """The batch-256 stem's row width (224 -> 112 outputs, padded rows of 128)
    on one image: every output against the oracle."""
    shape = (1, 224, 224, 3, 64, 7, 7, 2, 3)
    x, w, dy, P, Q = inputs(shape, seed_cfg=4)
    d = pf16.conv_desc(*shape)
    y = run_fwd(d, x, w)
    V, A, _ = orc.conv_fwd(x, w, *shape)
    rel = assert_conv_close(y, V, A, 147, "fwd")
    assert rel < 2.0 ** -7, rel


@pytest.mark.parametrize("shape", [(2, 9, 9, 64, 128, 3, 3, 1, 1), (2, 10, 10, 64, 64, 1, 1, 2, 0),
                                   (2, 11, 11, 64, 64, 3, 3, 2, 1), (2, 12, 10, 64, 64, 3, 3, 1, 1),
                                   (2, 12, 12, 64, 64, 3, 3, 2, 1),
                                   (2, 32, 32, 3, 64, 7, 7, 2, 3)],
                         ids=ids)
def test_accumulate_flag(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape)
    d = pf16.conv_desc(*shape)
    y0 = syn.normal_f16(77, (N * P * Q * K,))
    y = run_fwd(d, x, w, pf16.PF16_ACCUMULATE, y0)
    V, A, _ = orc.conv_fwd(x, w, *shape)
    assert_conv_close(y, V, A, C * R * S, "fwd+acc", prev=y0)
    if C == 3:
        return  # the stem has no data gradient
    dx0 = syn.normal_f16(78, (N * H * W * C,))
    dx = run_dgrad(d, dy, w, pf16.PF16_ACCUMULATE, dx0)
    V, A, T = orc.conv_dgrad(dy, w, *shape)
    assert_conv_close(dx, V, A, np.maximum(T, 1), "dgrad+acc", prev=dx0)
    # positions no tap reaches keep their previous value exactly
    assert np.array_equal(dx[T == 0], dx0[T == 0])


@pytest.mark.parametrize("r0,s0", [(0, 0), (1, 1), (2, 1)])
@pytest.mark.parametrize("st", [1, 2])
def test_delta_kernel_bit_exact(orc, r0, s0, st):
    """w[k,r,s,c] = [k = c][r = r0][s = s0]: one term per output, so the FP16
    forward and data gradient are exact shifts."""
    N, H, W, C = 2, 12, 10, 64
    shape = (N, H, W, C, C, 3, 3, st, 1)
    x, _, _, P, Q = inputs(shape, seed_cfg=2)
    w = np.zeros((C, 3, 3, C), np.float16)
    for k in range(C):
        w[k, r0, s0, k] = 1.0
    w = w.view(np.uint16)
    d = pf16.conv_desc(*shape)
    y = run_fwd(d, x, w)
    V, _, _ = orc.conv_fwd(x, w, *shape)
    assert np.array_equal(f64(y), V)
    dy = syn.normal_f16(9, (N, P, Q, C))
    dx = run_dgrad(d, dy, w)
    V, _, _ = orc.conv_dgrad(dy, w, *shape)
    assert np.array_equal(f64(dx), V)


@pytest.mark.parametrize("shape", [(4, 12, 12, 128, 128, 3, 3, 1, 1),   # wide halo, four images per padded row
                                   (2, 8, 28, 256, 256, 3, 3, 1, 1)],   # wide halo, one image per padded row
                         ids=ids)
@pytest.mark.parametrize("tap", [0, 4, 8])
def test_delta_kernel_wide_halo_bit_exact(orc, shape, tap):
    """The delta kernel through the wide halo engine: each tap window of the
    input box is an exact shift (and so is the data gradient)."""
    N, H, W, C, K, R, S, st, pd = shape
    x, _, _, P, Q = inputs(shape, seed_cfg=2)
    w = np.zeros((K, 3, 3, C), np.float16)
    for k in range(K):
        w[k, tap // 3, tap % 3, k % C] = 1.0
    w = w.view(np.uint16)
    d = pf16.conv_desc(*shape)
    y = run_fwd(d, x, w)
    V, _, _ = orc.conv_fwd(x, w, *shape)
    assert np.array_equal(f64(y), V)
    dy = syn.normal_f16(9, (N, P, Q, K))
    dx = run_dgrad(d, dy, w)
    V, _, _ = orc.conv_dgrad(dy, w, *shape)
    assert np.array_equal(f64(dx), V)


@pytest.mark.parametrize("shape", [(2, 8, 8, 64, 192, 3, 3, 1, 1),    # im2col GEMM
                                   (2, 9, 12, 64, 64, 3, 3, 1, 1),    # halo weight gradient, odd P
                                   (2, 8, 8, 64, 128, 3, 3, 1, 1),    # wide halo weight gradient
                                   (3, 5, 15, 128, 256, 3, 3, 1, 1)],  # wide, three images per box
                         ids=ids)
def test_delta_gradient_wgrad_bit_exact(orc, shape):
    """dy nonzero (= 1) at a single pixel per channel: every dw element is one
    product x * 1, exact in FP16."""
    N, H, W, C, K, R, S, st, pd = shape
    x, _, _, P, Q = inputs(shape, seed_cfg=3)
    dyf = np.zeros((N, P, Q, K), np.float16)
    for k in range(K):
        dyf[k % N, (3 * k) % P, (5 * k) % Q, k] = 1.0
    dy = dyf.view(np.uint16)
    d = pf16.conv_desc(*shape)
    dw = run_wgrad(d, x, dy)
    V, _, _ = orc.conv_wgrad(x, dy, *shape)
    assert np.array_equal(f64(dw), V)


# The wide halo weight gradient (K a multiple of 128, 3x3 stride 1): boxes of
# nb images of W + 1 columns, chunked FP16 accumulations and the split-K tree.
WGRAD_WIDE = [
    (2, 7, 7, 512, 512, 3, 3, 1, 1),     # 7x7: 8-column images, four output-channel tiles
    (17, 2, 7, 64, 128, 3, 3, 1, 1),     # 16 images per box, the second box one image
    (1, 3, 127, 64, 128, 3, 3, 1, 1),    # W + 1 = 128: windows read the zero tail
    (1, 4, 60, 64, 128, 3, 3, 1, 1),     # one image of 61 columns per box
    (8, 28, 28, 128, 128, 3, 3, 1, 1),   # several tiles per chunk, several chunks
    (3, 5, 9, 128, 384, 3, 3, 1, 1),     # three output-channel tiles
]


@pytest.mark.parametrize("shape", WGRAD_WIDE, ids=ids)
def test_conv_wgrad_wide(orc, shape):
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape, seed_cfg=6)
    d = pf16.conv_desc(*shape)
    dw = run_wgrad(d, x, dy)
    V, A, T = orc.conv_wgrad(x, dy, *shape)
    rel = assert_conv_close(dw, V, A, N * P * Q, "wgrad")
    assert rel < 2.0 ** -6, rel


CFG3 = [(256, 56, 56, 256, 64, 1, 1, 1, 0), (256, 28, 28, 512, 128, 1, 1, 1, 0),
        (256, 14, 14, 1024, 256, 1, 1, 1, 0), (256, 7, 7, 512, 2048, 1, 1, 1, 0),
        (256, 56, 56, 64, 64, 3, 3, 1, 1),  # the 3x3 64-channel layer: halo engines, 802,816-pixel weight gradient
        (256, 14, 14, 256, 256, 3, 3, 1, 1)]  # wide halo engines: forward, 50,176-pixel weight gradient


@pytest.mark.parametrize("shape", CFG3, ids=ids)
def test_full_size_sampled(orc, shape):
    """The N=256 pure-GEMM 1x1 layers and the 56x56 3x3 64-channel layer at
    full size, checked on sampled outputs (wgrad reductions of 802,816 pixels)."""
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape, seed_cfg=3)
    d = pf16.conv_desc(*shape)
    rng = np.random.default_rng(3)
    y = run_fwd(d, x, w).ravel()
    idx = rng.integers(0, y.size, 2048)
    V, A, _ = orc.conv_fwd(x, w, *shape, idx=idx)
    assert_conv_close(y[idx], V, A, C, "fwd")
    dx = run_dgrad(d, dy, w).ravel()
    idx = rng.integers(0, dx.size, 2048)
    V, A, T = orc.conv_dgrad(dy, w, *shape, idx=idx)
    assert_conv_close(dx[idx], V, A, np.maximum(T, 1), "dgrad")
    dw = run_wgrad(d, x, dy).ravel()
    idx = rng.integers(0, dw.size, 256)
    V, A, _ = orc.conv_wgrad(x, dy, *shape, idx=idx)
    rel = assert_conv_close(dw[idx], V, A, N * P * Q, "wgrad")
    assert rel < 2.0 ** -5, rel


F32_SHAPES = [
    (2, 14, 14, 256, 256, 3, 3, 1, 1),   # im2col forward, reduction 2,304, 256-wide N tiles
    (4, 14, 14, 256, 256, 3, 3, 1, 1),   # wide halo engine, four images per padded row
    (2, 28, 28, 64, 64, 3, 3, 1, 1),     # halo engine
    (2, 32, 32, 3, 64, 7, 7, 2, 3),      # stem: space-to-depth halo forward, stem weight gradient
    (2, 14, 14, 64, 256, 1, 1, 1, 0),    # dense 1x1
    (2, 12, 12, 128, 128, 3, 3, 2, 1),   # strided 3x3: the four stride phases in one launch, scattered rows
    (2, 9, 9, 64, 128, 3, 3, 2, 1),      # strided 3x3, odd size: one launch per phase
]


@pytest.mark.parametrize("shape", F32_SHAPES, ids=ids)
def test_f32_accumulate_contrast(orc, shape):
    """PF16_F32_ACCUM: FP32 accumulation inside the tensor core and one
    rounding to FP16 per output (per partial for the weight gradient).  The
    forward and the data gradient are then within half an FP16 ulp of the exact
    value plus an FP32 accumulation term, the weight gradient within the
    contract bound, and on average none is farther from the exact value than
    the pure-FP16 result."""
    N, H, W, C, K, R, S, st, pd = shape
    x, w, dy, P, Q = inputs(shape, seed_cfg=5)
    d = pf16.conv_desc(*shape)
    f32 = pf16.PF16_F32_ACCUM

    def check(g32, g16, V, A, Rn, what):
        e32 = np.abs(f64(g32).ravel() - V)
        e16 = np.abs(f64(g16).ravel() - V)
        bound = U * np.abs(V) + Rn * 2.0 ** -22 * A + 2.0 ** -24
        assert np.all(e32 <= bound), (what, float(np.max(e32 / bound)))
        assert e32.mean() <= e16.mean(), (what, e32.mean(), e16.mean())

    V, A, _ = orc.conv_fwd(x, w, *shape)
    check(run_fwd(d, x, w, f32), run_fwd(d, x, w), V, A, C * R * S, "fwd")
    if C != 3:
        V, A, T = orc.conv_dgrad(dy, w, *shape)
        check(run_dgrad(d, dy, w, f32), run_dgrad(d, dy, w), V, A, np.maximum(T, 1), "dgrad")
    dw16 = run_wgrad(d, x, dy)
    dw32 = empty16(d.k * d.r * d.s * d.c)
    pf16.conv_wgrad(d, dev(x), dev(dy), dw32, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)),
                    f32)
    assert pf16.sync_status() == 0
    V, A, _ = orc.conv_wgrad(x, dy, *shape)
    assert_conv_close(host(dw32), V, A, N * P * Q, "wgrad f32")
    assert np.abs(f64(host(dw32)).ravel() - V).mean() <= np.abs(f64(dw16).ravel() - V).mean()
