"""Pins of the oracle's composed ResNet-50 training step (oracle/resnet50.py)
against facts fixed outside it:

* the architecture of ResNet-50 v1.5 (paper Sec. 5.1): parameter counts,
  per-image multiply-adds, the stride on each bottleneck's 3x3 conv, the stage
  output sizes;
* the zero-gamma initialisation of each block's last BatchNorm (Sec. 5.1):
  identity blocks pass their input through exactly;
* the softmax cross-entropy closed form at zero logits (ln K, and dlogits =
  (1/K - onehot) / B), with every upstream gradient exactly zero;
* the composed forward and backward against reverse-mode automatic
  differentiation of an independent binary64 PyTorch model of the same network
  (paper Sec. 4.2's x0.25 after every BatchNorm of a residual block), piece by
  piece on the oracle's weights, inputs and output gradients.  The oracle's
  backward is a hand-written chain of layer calls; the PyTorch model's
  backward is autograd's, so a mis-wired gradient (the residual's share, the
  projection's branch, a BatchNorm's scale or ReLU) shows up as an O(1)
  disagreement, far above the FP16 storage error.  Planted wiring mistakes are
  checked to fail the comparison.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_1911_07384_gb300 import synthetic as syn


def f64(bits):
    return np.asarray(bits).view(np.float16).astype(np.float64)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


@pytest.fixture(scope="module")
def oresnet(orc):
    from oracle import resnet50 as m

    return m


def test_parameter_counts_v15(oresnet):
    """ResNet-50 has 25,557,032 parameters: 25,502,912 conv / FC weights, 1,000
    FC biases (all decayed) and 53,120 BatchNorm gamma / beta (no decay)."""
    net = oresnet.OracleResNet50(1, 224, 1000)
    wd, nowd = net.param_counts()
    assert (wd, nowd) == (25_503_912, 53_120)
    assert wd + nowd == 25_557_032
    assert sum(c[1].size for c in net.convs.values()) == 25_502_912


def test_v15_wiring_and_sizes(oresnet):
    """v1.5: the stride of a stage's first block sits on its 3x3 conv (and the
    projection), never on the first 1x1; spatial sizes 112 (stem), 56 (pool),
    then 56 / 28 / 14 / 7 at the four stages for a 224 x 224 input; about 4.09 G
    multiply-adds per image forward."""
    net = oresnet.OracleResNet50(1, 224, 1000)
    assert net.h0 == 112 and net.hp == 56
    outs = {}
    for nm, h, h2, cin, width, proj in net.blocks:
        st = net.convs[nm + "c2"][0][7]
        assert net.convs[nm + "c1"][0][7] == 1 and net.convs[nm + "c3"][0][7] == 1
        assert net.convs[nm + "c2"][0][5:7] == (3, 3)
        if proj:
            assert net.convs[nm + "cp"][0][7] == st
            assert st == (1 if nm.startswith("s0") else 2)
        else:
            assert st == 1
        outs[nm[:2]] = (h2, 4 * width)
    assert outs == {"s0": (56, 256), "s1": (28, 512), "s2": (14, 1024), "s3": (7, 2048)}
    assert [nm for nm, *_ in net.blocks].count("s2b5") == 1 and len(net.blocks) == 16
    macs = 0
    for d, w, _ in net.convs.values():
        N, H, W, C, K, R, S, stv, pad = d
        P = (H + 2 * pad - R) // stv + 1
        macs += P * P * K * C * R * S
    assert abs(macs / 1e9 - 4.09) < 0.01, macs


def test_identity_blocks_exact_at_init(oresnet):
    """With gamma = 0 in the last BatchNorm (beta = 0), an identity block's
    output is ReLU(0 + x) = x for its non-negative input x, bit for bit."""
    net = oresnet.OracleResNet50(2, 32, 10)
    imgs = syn.images_f16(syn.seed_for(4, "x"), 2, 32, 32, 3)
    labs = syn.labels(syn.seed_for(4, "labels"), 2, 10)
    _, cache = net.forward(imgs, labs)
    n_id = 0
    for nm, *_, proj in net.blocks:
        x, a1, b1, a2, b2, a3, ap, bp, y = cache["act"][nm]
        if not proj:
            assert np.array_equal(y, x), nm
            n_id += 1
        else:
            assert np.array_equal(y, f16(np.maximum(f64(bp), 0.0))), nm
    assert n_id == 12


def test_zero_classifier_closed_form(oresnet):
    """FC weights and bias zero: logits 0, loss = ln 1000, dlogits = (1/1000 -
    onehot) / B; df = 0, so every gradient before the classifier is zero."""
    B, K = 2, 1000
    net = oresnet.OracleResNet50(B, 32, K)
    net.convs["fc"][1][:] = 0
    imgs = syn.images_f16(syn.seed_for(4, "x"), B, 32, 32, 3)
    labs = syn.labels(syn.seed_for(4, "labels"), B, K)
    loss, cache = net.forward(imgs, labs)
    assert abs(loss - math.log(K)) < 1e-12
    onehot = np.zeros((B, K))
    onehot[np.arange(B), labs] = 1.0
    assert np.allclose(cache["dlogits"].reshape(B, K), (1.0 / K - onehot) / B, rtol=0, atol=1e-16)
    grads, bgrads, gbias = net.backward(cache)
    for name, g in grads.items():
        if name != "fc":
            assert not np.any(f64(g)), name
    for name, g in bgrads.items():
        assert not np.any(f64(g)), name
    assert np.allclose(f64(gbias), f64(f16(onehot.mean(0) * -1 + 1.0 / K)), atol=2.0 ** -24)


# ---------------------------------------------------------------- autograd comparison
# The comparison is made piece by piece -- the head (average pool, classifier,
# loss), each bottleneck block, the stem -- each piece fed the oracle's own
# binary16 input and output gradient (teacher forcing).  At the small sizes a
# CPU test affords, BatchNorm over a few rows amplifies the FP16 storage error
# through 16 blocks (about 10% relative by the last stage at 64 x 64, batch 4),
# which would hide a wiring mistake in a whole-network comparison; per piece
# the disagreement stays near the storage error, and a mis-wired piece is off
# by O(1).

def _t(bits, shape=None):
    a = torch.tensor(f64(bits))
    return a.reshape(shape) if shape is not None else a


def _nchw(bits, N, H, C):
    return _t(bits, (N, H, H, C)).permute(0, 3, 1, 2).contiguous()


def _nhwc(t):
    return t.detach().permute(0, 2, 3, 1).numpy().ravel()


def oresnet_eps():
    return float(np.uint16(0x00A8).view(np.float16))


class _Torch:
    """Binary64 PyTorch pieces of ResNet-50 v1.5 on the oracle's parameters:
    conv -> BatchNorm (batch statistics, biased variance) x s (0.25 in every
    block, 1 at the stem) [+ shortcut] [-> ReLU]."""

    def __init__(self, net):
        self.net = net
        self.P = {}
        for name, (d, w, _) in net.convs.items():
            K, R, S, C = d[4], d[5], d[6], d[3]
            self.P[name] = _t(w, (K, R, S, C)).permute(0, 3, 1, 2).contiguous().requires_grad_()
        for name, st in net.bns.items():
            self.P[name + "g"] = _t(st[1]).requires_grad_()
            self.P[name + "b"] = _t(st[2]).requires_grad_()
        self.P["bias"] = _t(net.bias).requires_grad_()

    def conv(self, name, t):
        d = self.net.convs[name][0]
        return F.conv2d(t, self.P[name], stride=d[7], padding=d[8])

    def bn(self, name, t, s, relu, shortcut=None):
        y = F.batch_norm(t, None, None, self.P[name + "g"], self.P[name + "b"], training=True,
                         eps=oresnet_eps()) * s
        if shortcut is not None:
            y = y + shortcut
        return F.relu(y) if relu else y

    def stem(self, x):
        return F.max_pool2d(self.bn("bn0", self.conv("stem", x), 1.0, True), 3, 2, 1)

    def block(self, nm, proj, h):
        t = self.bn(nm + "n1", self.conv(nm + "c1", h), 0.25, True)
        t = self.bn(nm + "n2", self.conv(nm + "c2", t), 0.25, True)
        sc = self.bn(nm + "np", self.conv(nm + "cp", h), 0.25, False) if proj else h
        return self.bn(nm + "n3", self.conv(nm + "c3", t), 0.25, True, shortcut=sc)

    def head(self, h, labels):
        f = h.mean(dim=(2, 3), keepdim=True)
        logits = self.conv("fc", f).flatten(1) + self.P["bias"]
        return F.cross_entropy(logits, torch.tensor(np.asarray(labels, np.int64))), logits


def _rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _randomise_bn(net, seed):
    """gamma ~ 1 + 0.2 N(0,1), beta ~ 0.1 N(0,1) in every BatchNorm, so that no
    block is the identity and every gradient is non-zero."""
    rng = np.random.default_rng(seed)
    for st in net.bns.values():
        C = st[0]
        st[1] = f16(1.0 + 0.2 * rng.standard_normal(C))
        st[2] = f16(0.1 * rng.standard_normal(C))


def _compare(net, imgs, labs):
    """Relative L2 disagreement, per piece and tensor, between the oracle's
    composed step and autograd on the same pieces."""
    loss, cache = net.forward(imgs, labs)
    grads, bgrads, gbias = net.backward(cache)
    T = _Torch(net)
    N, act, dys = net.N, cache["act"], cache["dy"]
    out = {}

    def pgrad(name):
        return _nhwc(T.P[name].grad) if T.P[name].dim() == 4 else T.P[name].grad.numpy()

    # head: the last block's output -> loss
    last = net.blocks[-1][0]
    y = _nchw(act[last][8], N, net.hl, net.cl).requires_grad_()
    tl, logits = T.head(y, labs)
    tl.backward()
    out["loss"] = abs(loss - float(tl.detach())) / float(tl.detach())
    out["logits"] = _rel(f64(cache["logits"]).ravel(), logits.detach().numpy().ravel())
    out["fc"] = _rel(f64(grads["fc"]), pgrad("fc"))
    out["bias"] = _rel(f64(gbias), pgrad("bias"))
    out["dy:" + last] = _rel(f64(dys[last]), _nhwc(y.grad))
    # blocks, each from its own input and output gradient
    names = [b[0] for b in net.blocks]
    for k, (nm, h, h2, cin, width, proj) in enumerate(net.blocks):
        x = _nchw(act[nm][0], N, h, cin).requires_grad_()
        yt = T.block(nm, proj, x)
        yt.backward(_nchw(dys[nm], N, h2, 4 * width))
        out["y:" + nm] = _rel(f64(act[nm][8]), _nhwc(yt))
        dx_oracle = dys[names[k - 1]] if k > 0 else cache["dp0"]
        out["dx:" + nm] = _rel(f64(dx_oracle), _nhwc(x.grad))
        for c in ("c1", "c2", "c3") + (("cp",) if proj else ()):
            out[nm + c] = _rel(f64(grads[nm + c]), pgrad(nm + c))
        for b in ("n1", "n2", "n3") + (("np",) if proj else ()):
            out[nm + b + "g"] = _rel(f64(bgrads[nm + b + "g"]), pgrad(nm + b + "g"))
            out[nm + b + "b"] = _rel(f64(bgrads[nm + b + "b"]), pgrad(nm + b + "b"))
    # stem: images -> max-pool output
    p0 = T.stem(_nchw(imgs, N, net.image, 3))
    p0.backward(_nchw(cache["dp0"], N, net.hp, 64))
    out["p0"] = _rel(f64(cache["p0"]), _nhwc(p0))
    out["stem"] = _rel(f64(grads["stem"]), pgrad("stem"))
    out["bn0g"] = _rel(f64(bgrads["bn0g"]), pgrad("bn0g"))
    out["bn0b"] = _rel(f64(bgrads["bn0b"]), pgrad("bn0b"))
    return out


@pytest.fixture(scope="module")
def step_inputs():
    B, img, K = 4, 64, 10
    imgs = syn.images_f16(syn.seed_for(4, "x"), B, img, img, 3)
    labs = syn.labels(syn.seed_for(4, "labels"), B, K)
    return B, img, K, imgs, labs


# Per-piece disagreement from the FP16 storage of every layer's output: median
# about 1.6%, worst about 5% (BatchNorm gradients over 16-1,024 rows are sums
# with heavy cancellation, so their relative error is well above 2^-11).  The
# planted mistakes below give 0.7-3.5 on dozens of tensors.
TOL = 0.1


def test_backward_matches_autograd(oresnet, step_inputs):
    B, img, K, imgs, labs = step_inputs
    net = oresnet.OracleResNet50(B, img, K)
    _randomise_bn(net, 7)
    out = _compare(net, imgs, labs)
    bad = {k: v for k, v in out.items() if not v < TOL}
    assert not bad, bad
    assert np.median(list(out.values())) < 0.03, np.median(list(out.values()))


@pytest.mark.parametrize("mistake", ["proj_scale_1", "residual_after_relu", "n3_without_mask"])
def test_planted_wiring_mistake_is_caught(oresnet, step_inputs, monkeypatch, mistake):
    """The comparison is sensitive: a plausible mistake planted in the oracle's
    composition breaks it -- the projection BatchNorm left unscaled, the
    shortcut added after the last ReLU instead of before it, the last
    BatchNorm's backward taken without its ReLU decisions."""
    B, img, K, imgs, labs = step_inputs
    net = oresnet.OracleResNet50(B, img, K)
    _randomise_bn(net, 7)
    if mistake == "proj_scale_1":
        for name, st in net.bns.items():
            if name.endswith("np"):
                st[5] = 1.0
    elif mistake == "residual_after_relu":
        orig = net._bf

        def bf(name, x, residual=None):
            y = orig(name, x)
            return y if residual is None else f16(f64(y) + f64(residual))

        monkeypatch.setattr(net, "_bf", bf)
    else:
        orig = net._bb

        def bb(name, x, y, dy):  # the last BatchNorm's backward taken without its ReLU mask
            return orig(name, x, None if name.endswith("n3") else y, dy)

        monkeypatch.setattr(net, "_bb", bb)
    out = _compare(net, imgs, labs)
    assert max(out.values()) > 5 * TOL, max(out.values())
