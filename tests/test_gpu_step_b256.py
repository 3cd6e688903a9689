"""Teacher-forced layer-wise parity of the batch-256 ResNet-50 step.

One eager forward and backward of the full workload (batch 256, 224 x 224 x 3,
the calls and kernels the timed step replays: fused BatchNorm statistics in
the conv epilogues, the shortcut gradient added in the data-gradient
epilogue, the stem's space-to-depth engine, the split-K weight gradients) is
run once.  Then every call of it is checked on its own: the oracle is given
the GPU's own binary16 inputs of that call (teacher forcing) and its outputs
are compared element by element under that layer's bound --

* convolutions (forward, data gradient, weight gradient), on sampled outputs
  (1,024 forward / data gradient, 256 weight gradient, each a full
  reduction: up to 3,211,264 pixels for the stem's weight gradient) under
  the contract |err| <= 4 sqrt(R) 2^-11 sum|terms|, plus one rounding where the
  call adds into its output;
* BatchNorms (Eq. 1-2 and Sec. 4.2's x0.25, forward and backward), on every
  row of 8 sampled channels, under the bounds of tests/test_gpu_bn.py; the
  saved mean / invstd and the ReLU bit mask too;
* max pool, average pool, classifier and loss, under the bounds of
  tests/test_gpu_glue.py.

The weights are the initial ones: no update runs, so the arenas still hold
the weights every call used.  Where the step applies a BatchNorm inside the
next conv's operand path (each block's second), the conv is checked against
the oracle on that BatchNorm's output, stored afterwards by the apply pass."""
import zlib

import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from paper_1911_07384_gb300.resnet50 import ResNet50
from gpu_util import U, assert_conv_close, conv_bound, f64, host

pytestmark = pytest.mark.gpu

BATCH, IMAGE = 256, 224
EPS_F = float(np.uint16(0x00A8).view(np.float16))
NS_FWD, NS_WGRAD, NS_CH = 1024, 256, 8


@pytest.fixture(scope="module")
def step():
    torch.cuda.empty_cache()
    net = ResNet50(batch=BATCH, image=IMAGE, seed_cfg=4)
    net.set_batch(syn.images_f16(syn.seed_for(4, "x"), BATCH, IMAGE, IMAGE, 3),
                  syn.labels(syn.seed_for(4, "labels"), BATCH))
    # a non-trivial last BatchNorm in every block (the zero-gamma initialisation
    # would make most of the backward zero)
    g = syn.normal_f16(syn.seed_for(4, 9), (net.nowd.size,))
    gam = (1.0 + 0.2 * f64(g)).astype(np.float16).view(np.int16)
    for b in net.blocks:
        n = b.bn3.c
        b.bn3.gamma.copy_(torch.from_numpy(gam[b.bn3.g_off:b.bn3.g_off + n].copy()))
    net.forward()
    net.backward()
    torch.cuda.synchronize()
    assert pf16.sync_status() == 0
    # A block's second BatchNorm is applied in its last conv's operand path and
    # never stored; store it now (the apply pass, bit-identical to the operand
    # transform: tests/test_gpu_bnin.py) so that the checks below can read it.
    # Its ReLU mask, written by the conv, must come out the same.
    for b in net.blocks:
        if b.fuse_bn2:
            mask = b.bn2.mask.clone()
            b.b2 = torch.empty_like(b.a2)
            b.bn2.fwd(b.a2, b.b2, conv=b.conv2)
            torch.cuda.synchronize()
            assert torch.equal(mask, b.bn2.mask)
    # The stem's BatchNorm + ReLU + max pooling forward runs fused
    # (pf16_bn_relu_maxpool_fwd), which does not store the BatchNorm's output;
    # make it with the separate call, bit-identical to the fused one
    # (tests/test_gpu_stem_fused.py), so that the checks below can read it.
    # The saved mean, invstd and ReLU mask must come out the same.
    if net.stem_fused:
        saved = [net.bn0.mean.clone(), net.bn0.invstd.clone(), net.bn0.mask.clone()]
        net.b0 = torch.empty_like(net.a0)
        net.bn0.fwd(net.a0, net.b0, conv=net.stem)
        torch.cuda.synchronize()
        for a, b in zip(saved, (net.bn0.mean, net.bn0.invstd, net.bn0.mask)):
            assert torch.equal(a, b)
    assert pf16.sync_status() == 0
    yield net
    del net
    torch.cuda.empty_cache()


class Host:
    """Host copies of device tensors, made once per tensor."""

    def __init__(self):
        self.c = {}

    def __call__(self, t):
        k = (t.data_ptr(), t.numel())
        if k not in self.c:
            self.c[k] = host(t)
        return self.c[k]


def _gather(t, idx):
    return host(t.view(-1)[torch.from_numpy(np.asarray(idx, np.int64)).cuda()])


def _dims(conv):
    d = conv.desc
    return d.n, d.h, d.w, d.c, d.k, d.r, d.s, d.stride, d.pad


def _rng(what):
    return np.random.default_rng(zlib.crc32(what.encode()))


def check_fwd(orc, H, conv, x, y, what):
    dims = _dims(conv)
    N, _, _, C, K, R, S, _, _ = dims
    P, Q = conv.desc.out_hw()
    idx = _rng(what).integers(0, N * P * Q * K, NS_FWD)
    V, A, _ = orc.conv_fwd(H(x), H(conv.w), *dims, idx=idx)
    assert_conv_close(_gather(y, idx), V, A, C * R * S, what)


def check_wgrad(orc, H, conv, x, dy, what):
    dims = _dims(conv)
    N, _, _, C, K, R, S, _, _ = dims
    P, Q = conv.desc.out_hw()
    idx = _rng(what).integers(0, K * R * S * C, NS_WGRAD)
    V, A, _ = orc.conv_wgrad(H(x), H(dy), *dims, idx=idx)
    assert_conv_close(_gather(conv.gw, idx), V, A, N * P * Q, what)


def dgrad_ref(orc, H, conv, dy, idx):
    V, A, T = orc.conv_dgrad(H(dy), H(conv.w), *_dims(conv), idx=idx)
    return V, A, np.maximum(T, 1)


def check_dgrad(orc, H, conv, dy, dx, what):
    d = conv.desc
    idx = _rng(what).integers(0, d.n * d.h * d.w * d.c, NS_FWD)
    V, A, T = dgrad_ref(orc, H, conv, dy, idx)
    assert_conv_close(_gather(dx, idx), V, A, T, what)


def _close(g, ref, tol, what):
    err = np.abs(g - ref)
    bad = ~(err <= tol)
    if bad.any():
        i = int(np.argmax(np.where(np.isfinite(err), err - tol, np.inf)))
        raise AssertionError(f"{what}: {int(bad.sum())} of {g.size} outside the bound; worst {i}: gpu {g[i]!r} "
                             f"ref {ref[i]!r} tol {tol[i]!r}")


def mask_at(mask, C, idx):
    """ReLU bits at flat element indices idx of an [R][C] tensor."""
    idx = np.asarray(idx, np.int64)
    byte = (idx // C) * (C // 8) + (idx % C) // 8
    b = host(mask.view(-1)[torch.from_numpy(byte).cuda()]).view(np.uint8)
    return ((b >> (idx % 8).astype(np.uint8)) & 1).astype(bool)


def mask_bits(mask, R, C, ch):
    """ReLU bits of channels ch for every row (bit c % 8 of byte c // 8 of the row)."""
    b = host(mask.view(R, C // 8)[:, torch.from_numpy(ch // 8).cuda()].contiguous()).view(np.uint8)
    return ((b >> (ch % 8).astype(np.uint8)) & 1).astype(bool)


class BnSub:
    """8 sampled channels of one BatchNorm: every row of them, on the host."""

    def __init__(self, bn, what):
        self.bn, self.C = bn, bn.c
        self.R = bn.elems // bn.c
        self.ch = np.sort(_rng(what).choice(self.C, NS_CH, replace=False))
        self.cht = torch.from_numpy(self.ch).cuda()
        self.s = float(np.uint16(bn.desc.post_scale).view(np.float16))
        self.relu = bool(bn.desc.flags & pf16.PF16_BN_RELU)
        self.L = int(np.ceil(np.log2(self.R)))
        self.gamma, self.beta = host(bn.gamma)[self.ch], host(bn.beta)[self.ch]

    def sub(self, t):
        return host(t.view(self.R, self.C)[:, self.cht].contiguous())


def check_bn_fwd(orc, bn, x, y, res, what):
    b = BnSub(bn, what)
    R, L, s = b.R, b.L, b.s
    xs, ys = b.sub(x), b.sub(y)
    rs = b.sub(res) if res is not None else None
    yo, mean, var, invstd = orc.bn_fwd(xs, b.gamma, b.beta, rs, R, NS_CH, EPS_F, s, b.relu)
    xhat = (f64(xs) - mean) * invstd
    scale = s * (np.abs(f64(b.gamma)) * (np.abs(xhat) + 1) + np.abs(f64(b.beta)))
    if rs is not None:
        scale = scale + np.abs(f64(rs))
    _close(f64(ys).ravel(), yo.ravel(), ((4 * L + 8) * U * scale + 2.0 ** -24).ravel(), what + " y")
    _close(f64(host(bn.mean))[b.ch], mean, (L + 8) * U * np.abs(f64(xs)).max(0), what + " mean")
    _close(f64(host(bn.invstd))[b.ch], invstd, (2 * L + 16) * U * invstd, what + " invstd")
    if b.relu:
        assert np.array_equal(mask_bits(bn.mask, R, b.C, b.ch), f64(ys) > 0), what + " mask"


def check_bn_bwd(orc, bn, x, y, dy, dx, dres, what):
    b = BnSub(bn, what)
    R, L, s = b.R, b.L, b.s
    xs, dys, dxs = b.sub(x), b.sub(dy), b.sub(dx)
    ys = b.sub(y) if b.relu else None
    dxo, dgo, dbo, dro = orc.bn_bwd(xs, b.gamma, dys, ys, R, NS_CH, EPS_F, s, b.relu)
    _, mean, var, invstd = orc.bn_fwd(xs, b.gamma, b.beta, None, R, NS_CH, EPS_F, s, b.relu)
    xhat = (f64(xs) - mean) * invstd
    dyp = np.abs(dro)
    k = np.abs(s * f64(b.gamma) * invstd)
    tol = (4 * L + 8) * U * k * (dyp + dyp.max(0) * (np.abs(xhat) + 1)) + 2.0 ** -24
    _close(f64(dxs).ravel(), dxo.ravel(), tol.ravel(), what + " dx")
    tol_b = (4 * L + 8) * U * s * dyp.sum(0) + 2.0 ** -24
    tol_g = (4 * L + 8) * U * s * (dyp * (np.abs(xhat) + 1)).sum(0) + 2.0 ** -24
    _close(f64(host(bn.dbeta))[b.ch], dbo, tol_b, what + " dbeta")
    _close(f64(host(bn.dgamma))[b.ch], dgo, tol_g, what + " dgamma")
    if dres is not None:  # the residual's gradient is dy where the ReLU passed: exact
        assert np.array_equal(f64(b.sub(dres)), dro), what + " dresidual"


def block_dx(net, i):
    """The buffer block i writes the gradient of its input into."""
    return net.blocks[i - 1].dy if i > 0 else net.dp0


def test_stem_forward(orc, step):
    net, H = step, Host()
    check_fwd(orc, H, net.stem, net.x, net.a0, "stem fwd")
    check_bn_fwd(orc, net.bn0, net.a0, net.b0, None, "bn0 fwd")
    # max pool over 4 whole images: a maximum of binary16 values is exact
    n4 = 4
    h0, hp = net.h0, net.hp
    b0 = host(net.b0[: n4 * h0 * h0 * 64])
    assert np.array_equal(f64(host(net.p0[: n4 * hp * hp * 64])), orc.maxpool_fwd(b0, n4, h0, h0, 64))


@pytest.mark.parametrize("i", range(16))
def test_block_forward(orc, step, i):
    net, H = step, Host()
    b = net.blocks[i]
    nm = f"block{i}"
    check_fwd(orc, H, b.conv1, b.x, b.a1, nm + " conv1 fwd")
    check_bn_fwd(orc, b.bn1, b.a1, b.b1, None, nm + " bn1 fwd")
    check_fwd(orc, H, b.conv2, b.b1, b.a2, nm + " conv2 fwd")
    check_bn_fwd(orc, b.bn2, b.a2, b.b2, None, nm + " bn2 fwd")
    check_fwd(orc, H, b.conv3, b.b2, b.a3, nm + " conv3 fwd")
    if b.proj:
        check_fwd(orc, H, b.convp, b.x, b.ap, nm + " proj fwd")
        check_bn_fwd(orc, b.bnp, b.ap, b.bp, None, nm + " bnp fwd")
    check_bn_fwd(orc, b.bn3, b.a3, b.y, b.bp if b.proj else b.x, nm + " bn3 fwd")


def test_head(orc, step):
    """Average pool, classifier, softmax cross-entropy and their backward."""
    net = step
    N, K, HW, C = net.N, net.classes, net.hl * net.hl, net.cl
    last = net.blocks[-1]
    L = int(np.ceil(np.log2(HW)))
    y = host(last.y)
    fo = orc.avgpool_fwd(y, N, HW, C)
    mx = np.abs(f64(y)).reshape(N, HW, C).max(1).ravel()
    _close(f64(host(net.f)), fo, (L + 3) * U * mx + 2.0 ** -24, "avgpool fwd")
    f, w = host(net.f), host(net.fc.w)
    V, A, _ = orc.conv_fwd(f, w, *_dims(net.fc))
    assert_conv_close(host(net.logits), V, A, C, "fc fwd")
    logits, bias = host(net.logits), host(net.bias)
    labels = net.labels.cpu().numpy()
    loss, dl, db = orc.softmax_xent(logits, bias, labels, N, K)
    l = f64(logits).reshape(N, K) + f64(bias)
    lse = np.log(np.exp(l - l.max(1, keepdims=True)).sum(1)) + l.max(1)
    lk = np.log2(K)
    tol_loss = (np.log2(N) + lk + 8) * U * (np.abs(lse).mean() + np.abs(l).max() + 1)
    assert abs(f64(host(net.loss))[0] - loss) <= tol_loss
    p = np.exp(l - lse[:, None])
    onehot = np.zeros((N, K))
    onehot[np.arange(N), labels] = 1
    tol_d = ((lk + 8) * U * (np.abs(l) + np.abs(lse)[:, None] + 1) * p + 2 * U * np.abs(p - onehot)) / N \
        + 2.0 ** -24
    _close(f64(host(net.dlogits)), dl, tol_d.ravel(), "dlogits")
    tol_b = tol_d.sum(0) + (np.log2(N) + 1) * U * np.abs(dl.reshape(N, K)).sum(0) + 2.0 ** -20
    _close(f64(host(net.dbias)), db, tol_b, "dbias")
    # classifier backward, teacher-forced on the GPU's dlogits
    H = Host()
    check_wgrad(orc, H, net.fc, net.f, net.dlogits, "fc wgrad")
    check_dgrad(orc, H, net.fc, net.dlogits, net.df, "fc dgrad")
    dxo = orc.avgpool_bwd(host(net.df), N, HW, C)
    _close(f64(host(last.dy)), dxo, 2 * U * np.abs(dxo) + 2.0 ** -24, "avgpool bwd")


@pytest.mark.parametrize("i", range(15, -1, -1))
def test_block_backward(orc, step, i):
    net, H = step, Host()
    b = net.blocks[i]
    nm = f"block{i}"
    check_bn_bwd(orc, b.bn3, b.a3, b.y, b.dy, b.da3, b.dres if b.proj else None, nm + " bn3 bwd")
    check_wgrad(orc, H, b.conv3, b.b2, b.da3, nm + " conv3 wgrad")
    check_dgrad(orc, H, b.conv3, b.da3, b.db2, nm + " conv3 dgrad")
    check_bn_bwd(orc, b.bn2, b.a2, b.b2, b.db2, b.da2, None, nm + " bn2 bwd")
    check_wgrad(orc, H, b.conv2, b.b1, b.da2, nm + " conv2 wgrad")
    check_dgrad(orc, H, b.conv2, b.da2, b.db1, nm + " conv2 dgrad")
    check_bn_bwd(orc, b.bn1, b.a1, b.b1, b.db1, b.da1, None, nm + " bn1 bwd")
    check_wgrad(orc, H, b.conv1, b.x, b.da1, nm + " conv1 wgrad")
    dx = block_dx(net, i)
    d = b.conv1.desc
    idx = _rng(nm + " dx").integers(0, d.n * d.h * d.w * d.c, NS_FWD)
    g = f64(_gather(dx, idx))
    V1, A1, T1 = dgrad_ref(orc, H, b.conv1, b.da1, idx)
    if b.proj:
        check_bn_bwd(orc, b.bnp, b.ap, None, b.dres, b.dap, None, nm + " bnp bwd")
        check_wgrad(orc, H, b.convp, b.x, b.dap, nm + " proj wgrad")
        # dx = rn(conv1's data gradient + the projection's, accumulated into it)
        Vp, Ap, Tp = dgrad_ref(orc, H, b.convp, b.dap, idx)
        B = conv_bound(A1, T1) + conv_bound(Ap, Tp)
        _close(g, V1 + Vp, B + U * (np.abs(V1 + Vp) + B), nm + " dx (conv1 + proj data gradients)")
    else:
        # dx = rn(conv1's data gradient + dy where the block's last ReLU passed)
        a = f64(_gather(b.dy, idx))
        on = mask_at(b.bn3.mask, d.c, idx)
        ref = V1 + np.where(on, a, 0.0)
        B = conv_bound(A1, T1)
        _close(g, ref, B + U * (np.abs(ref) + B), nm + " dx (data gradient + shortcut)")


def test_stem_backward(orc, step):
    net, H = step, Host()
    n4, h0, hp = 4, net.h0, net.hp
    # max-pool backward over 4 whole images, from the GPU's b0 and dp0
    b0 = host(net.b0[: n4 * h0 * h0 * 64])
    dp0 = host(net.dp0[: n4 * hp * hp * 64])
    dxo, A = orc.maxpool_bwd(b0, dp0, n4, h0, h0, 64)
    _close(f64(host(net.db0[: n4 * h0 * h0 * 64])), dxo, 3 * U * A, "maxpool bwd")
    check_bn_bwd(orc, net.bn0, net.a0, net.b0, net.db0, net.da0, None, "bn0 bwd")
    # the longest FP16 reduction of the step: 256 x 112 x 112 = 3,211,264 pixels
    check_wgrad(orc, H, net.stem, net.x, net.da0, "stem wgrad")
