"""GPU parity of the remaining ops of the training step (max pooling, global
average pooling, softmax cross-entropy) against the oracle.

Max pooling forward is exact (a maximum of binary16 values).  The other
bounds follow the FP16 op sequences: a backward cell sums at most 4 window
gradients (3 roundings); the average is a halving tree of depth
L = ceil(log2 hw) and one scaling; the softmax adds the roundings of the
bias add, the exp argument, a pairwise sum over k and the log."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import U, dev, empty16, f64, host, workspace

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape", [(2, 112, 112, 64), (1, 9, 10, 16), (3, 7, 7, 8)])
def test_maxpool(orc, shape):
    N, H, W, C = shape
    P, Q = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    x = syn.normal_f16(21, shape)
    dy = syn.normal_f16(22, (N, P, Q, C), 0.01)
    ty = empty16(N * P * Q * C)
    pf16.maxpool_fwd(dev(x), ty, N, H, W, C)
    assert np.array_equal(f64(host(ty)), orc.maxpool_fwd(x, N, H, W, C))
    tdx = empty16(N * H * W * C)
    pf16.maxpool_bwd(dev(x), dev(dy), tdx, N, H, W, C)
    assert pf16.sync_status() == 0
    dx, A = orc.maxpool_bwd(x, dy, N, H, W, C)
    assert np.all(np.abs(f64(host(tdx)) - dx) <= 3 * U * A)
    # the pair that keeps the maxima's positions: same y, the first-maximum
    # position of every window, and the very same dx
    ty2 = empty16(N * P * Q * C)
    targ = torch.empty(N * P * Q * C, dtype=torch.uint8, device="cuda")
    pf16.maxpool_fwd_argmax(dev(x), ty2, targ, N, H, W, C)
    assert np.array_equal(host(ty2), host(ty))
    assert np.array_equal(targ.cpu().numpy().reshape(N, P, Q, C), first_max_positions(x, N, H, W, C))
    tdx2 = empty16(N * H * W * C)
    pf16.maxpool_bwd_argmax(targ, dev(dy), tdx2, N, H, W, C)
    assert pf16.sync_status() == 0
    assert np.array_equal(host(tdx2), host(tdx))


def first_max_positions(x, N, H, W, C):
    """r*3+s of the first maximum (r then s, padding excluded) of every 3x3 /
    stride-2 / pad-1 window, by a scan over the nine taps in numpy."""
    v = f64(x).reshape(N, H, W, C)
    P, Q = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    best = np.full((N, P, Q, C), -np.inf)
    code = np.full((N, P, Q, C), 255, np.uint8)
    for r in range(3):
        for s_ in range(3):
            hs = 2 * np.arange(P) + r - 1
            ws = 2 * np.arange(Q) + s_ - 1
            okh, okw = (hs >= 0) & (hs < H), (ws >= 0) & (ws < W)
            sub = v[:, np.clip(hs, 0, H - 1)][:, :, np.clip(ws, 0, W - 1)]
            cand = np.where(okh[None, :, None, None] & okw[None, None, :, None], sub, -np.inf)
            better = cand > best
            best = np.where(better, cand, best)
            code = np.where(better, np.uint8(r * 3 + s_), code)
    return code


def test_maxpool_ties_first_cell(orc):
    N, H, W, C = 1, 6, 6, 8
    x = np.zeros((N, H, W, C), np.uint16)  # all equal: first valid cell of each window wins
    dy = syn.normal_f16(23, (N, 3, 3, C))
    tdx = empty16(N * H * W * C)
    pf16.maxpool_bwd(dev(x), dev(dy), tdx, N, H, W, C)
    dx, A = orc.maxpool_bwd(x, dy, N, H, W, C)
    assert np.all(np.abs(f64(host(tdx)) - dx) <= 3 * U * A)
    assert np.array_equal(f64(host(tdx)) != 0, dx != 0)
    targ = torch.empty(N * 3 * 3 * C, dtype=torch.uint8, device="cuda")
    pf16.maxpool_fwd_argmax(dev(x), empty16(N * 3 * 3 * C), targ, N, H, W, C)
    tdx2 = empty16(N * H * W * C)
    pf16.maxpool_bwd_argmax(targ, dev(dy), tdx2, N, H, W, C)
    assert np.array_equal(host(tdx2), host(tdx))


@pytest.mark.parametrize("shape", [(256, 49, 2048), (3, 10, 64)])
def test_avgpool(orc, shape):
    N, HW, C = shape
    L = int(np.ceil(np.log2(HW)))
    x = syn.normal_f16(24, (N, HW, C))
    dy = syn.normal_f16(25, (N, C), 0.01)
    ty = empty16(N * C)
    pf16.avgpool_fwd(dev(x), ty, N, HW, C)
    yo = orc.avgpool_fwd(x, N, HW, C)
    mx = np.abs(f64(x)).reshape(N, HW, C).max(1).ravel()
    assert np.all(np.abs(f64(host(ty)) - yo) <= (L + 3) * U * mx + 2.0 ** -24)
    tdx = empty16(N * HW * C)
    pf16.avgpool_bwd(dev(dy), tdx, N, HW, C)
    assert pf16.sync_status() == 0
    dxo = orc.avgpool_bwd(dy, N, HW, C)
    assert np.all(np.abs(f64(host(tdx)) - dxo) <= 2 * U * np.abs(dxo) + 2.0 ** -24)


@pytest.mark.parametrize("B,K", [(256, 1000), (5, 37), (64, 4096)])
def test_softmax_xent(orc, B, K):
    logits = syn.normal_f16(26, (B, K), 2.0)
    bias = syn.normal_f16(27, (K,), 0.1)
    labels = syn.labels(28, B, K)
    import torch

    tl, tdl, tdb = empty16(1), empty16(B * K), empty16(K)
    ws = workspace(pf16.softmax_xent_workspace_size(B, K))
    pf16.softmax_xent(dev(logits), dev(bias), torch.from_numpy(labels).cuda(), B, K, tl, tdl, tdb, ws)
    assert pf16.sync_status() == 0
    loss, dl, db = orc.softmax_xent(logits, bias, labels, B, K)
    l = (f64(logits).reshape(B, K) + f64(bias))
    lse = np.log(np.exp(l - l.max(1, keepdims=True)).sum(1)) + l.max(1)
    lk = np.log2(K)
    tol_loss = (np.log2(B) + lk + 8) * U * (np.abs(lse).mean() + np.abs(l).max() + 1)
    assert abs(f64(host(tl))[0] - loss) <= tol_loss
    p = np.exp(l - lse[:, None])
    onehot = np.zeros((B, K))
    onehot[np.arange(B), labels] = 1
    tol_d = ((lk + 8) * U * (np.abs(l) + np.abs(lse)[:, None] + 1) * p + 2 * U * np.abs(p - onehot)) / B \
        + 2.0 ** -24
    assert np.all(np.abs(f64(host(tdl)).reshape(B, K) - dl.reshape(B, K)) <= tol_d)
    tol_b = tol_d.sum(0) + (np.log2(B) + 1) * U * np.abs(dl.reshape(B, K)).sum(0) + 2.0 ** -20
    assert np.all(np.abs(f64(host(tdb)) - db) <= tol_b)
