"""GPU parity over every distinct convolution of ResNet-50 v1.5 at batch 64
(forward, data gradient, weight gradient per layer), and the underflow stress
workload on every distinct 3x3 and 1x1 conv of those at batch 128: log-uniform
output gradients over [2^-24, 2^4] with
random signs against near-one weights, so that products and partial sums run
through the binary16 subnormal range (Sec. 3 keeps gradual underflow).

The tensors are full size, so outputs are checked on seeded samples, each one
against the oracle's exact value for that output.  Inputs are slices of three
seeded pools (normal activations, normal gradients of std 0.01, log-uniform
gradients), drawn once: every slice has the distribution of its workload, and
drawing each layer's tensors separately would take minutes of host time.

Bound (the contract): |gpu - oracle| <= 4 * sqrt(R) * 2^-11 * sum|terms|.  The
stress workload adds an absolute floor of sqrt(R) * 2^-24, the per-addition
error of an FP16 accumulator whose partial sums fall below 2^-14, where a
relative bound no longer describes rounding."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from paper_1911_07384_gb300.resnet50 import conv_shapes
from gpu_util import assert_conv_close, conv_bound, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu

SWEEP_N = 64
STRESS_N = 128


def distinct_shapes(batch):
    seen = []
    for name, s in conv_shapes(batch):
        if s not in seen:
            seen.append(s)
            yield name, s


SWEEP = list(distinct_shapes(SWEEP_N))
# config 5: every distinct 3x3 and 1x1 conv of config 2 (all but the 7x7 stem), at batch 128
STRESS = [s for _, s in distinct_shapes(STRESS_N) if s[5] in (1, 3)]


def ids(s):
    return "N{}_{}x{}_C{}_K{}_{}x{}_s{}p{}".format(*s)


@pytest.fixture(scope="module")
def pools():
    """Seeded binary16 pools, each as large as the largest tensor drawn from it."""
    big = max(s[0] * s[1] * s[2] * max(s[3], s[4]) for s in [s for _, s in SWEEP] + STRESS)
    stress = max(s[0] * s[1] * s[2] * s[4] // (s[7] * s[7]) for s in STRESS)
    return {"x": syn.normal_f16(syn.seed_for(2, "x"), (big,)),
            "dy": syn.normal_f16(syn.seed_for(2, "dy"), (big,), 0.01),
            "dy_log": syn.loguniform_pm_f16(syn.seed_for(5, "dy"), (stress,))}


def take(pool, shape):
    n = int(np.prod(shape))
    assert n <= pool.size
    return pool[:n].reshape(shape)


def check_layer(orc, shape, x, w, dy, rng, fwd=True, floor=False):
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    d = pf16.conv_desc(*shape)
    tx, tw, tdy = dev(x), dev(w), dev(dy)

    def close(got, V, A, Rn, what):
        if not floor:
            return assert_conv_close(got, V, A, Rn, what)
        err = np.abs(f64(got).ravel() - V)
        tol = conv_bound(A, Rn) + np.sqrt(np.asarray(Rn, np.float64)) * 2.0 ** -24
        assert np.all(np.isfinite(f64(got))), what
        assert np.all(err <= tol), (what, int((err > tol).sum()), float(np.max(err / tol)))

    if fwd:
        y = empty16(N * P * Q * K)
        pf16.conv_fwd(d, tx, tw, y, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_FWD)))
        assert pf16.sync_status() == 0
        idx = rng.integers(0, y.numel(), 1024)
        V, A, _ = orc.conv_fwd(x, w, *shape, idx=idx)
        close(host(y)[idx], V, A, C * R * S, f"fwd {shape}")
        del y
    if C != 3:  # the stem's input gradient is never needed
        dx = empty16(N * H * W * C)
        pf16.conv_dgrad(d, tdy, tw, dx, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_DGRAD)))
        assert pf16.sync_status() == 0
        idx = rng.integers(0, dx.numel(), 1024)
        V, A, T = orc.conv_dgrad(dy, w, *shape, idx=idx)
        close(host(dx)[idx], V, A, np.maximum(T, 1), f"dgrad {shape}")
        del dx
    dw = empty16(K * R * S * C)
    pf16.conv_wgrad(d, tx, tdy, dw, workspace(pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)))
    assert pf16.sync_status() == 0
    idx = rng.integers(0, dw.numel(), 256)
    V, A, _ = orc.conv_wgrad(x, dy, *shape, idx=idx)
    close(host(dw)[idx], V, A, N * P * Q, f"wgrad {shape}")


@pytest.mark.parametrize("shape", [s for _, s in SWEEP], ids=ids)
def test_resnet50_layer_sweep_batch64(orc, pools, shape):
    """Every distinct conv of ResNet-50 v1.5 (stem, bottleneck 1x1/3x3/1x1 of
    the four stages, strided 3x3, projection shortcuts, the classifier) at
    batch 64: the kernels and split-K plans this batch selects."""
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    x = take(pools["x"], (N, H, W, C))
    w = syn.he_normal_f16(syn.seed_for(2, "w", sum(shape)), K, R, S, C)
    dy = take(pools["dy"], (N, P, Q, K))
    check_layer(orc, shape, x, w, dy, np.random.default_rng(sum(shape)))


@pytest.mark.parametrize("shape", STRESS, ids=ids)
def test_underflow_stress_batch128(orc, pools, shape):
    """Output gradients of magnitude 2^U(-24, 4) with random signs and weights
    1 + j * 2^-10: data and weight gradients through the subnormal range."""
    N, H, W, C, K, R, S, st, pd = shape
    P, Q = (H + 2 * pd - R) // st + 1, (W + 2 * pd - S) // st + 1
    x = take(pools["x"], (N, H, W, C))
    w = syn.near_one_f16(syn.seed_for(5, "w", sum(shape)), (K, R, S, C))
    dy = take(pools["dy_log"], (N, P, Q, K))
    assert np.any(np.abs(f64(dy)) < 2.0 ** -14)  # subnormal gradients are present
    check_layer(orc, shape, x, w, dy, np.random.default_rng(5 + sum(shape)), fwd=False, floor=True)
