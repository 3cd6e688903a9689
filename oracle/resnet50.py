"""ORACLE -- test infrastructure only (tests, smoke check, bench CPU baseline).

One ResNet-50 v1.5 training step composed from the oracle's layer functions
(paper Sec. 5.1: ResNet-50, SGD with momentum 0.9, weight decay 1e-4 on
conv/FC parameters, none on BatchNorm parameters, zero gamma in the last
BatchNorm of every residual block; Sec. 5.2: every tensor stored in FP16, no
master copy; Sec. 4.2: x0.25 after every BatchNorm of a residual block, the
stem's BatchNorm unchanged).  Each layer is evaluated in binary64 and its
result rounded once to binary16 (the storage format); the update is the
oracle's bit-exact FP16 step.  Written independently of the CUDA package.
"""
from __future__ import annotations

import zlib

import numpy as np

from . import (avgpool_bwd, avgpool_fwd, bn_bwd, bn_fwd, conv_dgrad, conv_fwd, conv_out_hw,
               conv_wgrad, f16_to_f64, f64_to_f16, maxpool_bwd, maxpool_fwd, sgd_update,
               softmax_xent)

LR, MOMENTUM, WD = 0x2E66, 0x3B33, 0x068E
EPS = float(np.uint16(0x00A8).view(np.float16))


def _he(seed, K, R, S, C):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((K, R, S, C)) * np.sqrt(2.0 / (C * R * S))).astype(np.float16).view(
        np.uint16)


class OracleResNet50:
    def __init__(self, batch, image=224, classes=1000, seed_cfg=4):
        self.N, self.image, self.classes = batch, image, classes
        self.convs = {}   # name -> [desc tuple, w, v]
        self.bns = {}     # name -> [C, gamma, beta, vg, vb, s, relu, residual]
        N = batch
        self._conv("stem", (N, image, image, 3, 64, 7, 7, 2, 3), seed_cfg)
        h = conv_out_hw(image, image, 7, 7, 2, 3)[0]
        self.h0 = h
        self._bn("bn0", 64, 1.0, True, False, False)
        h = (h - 1) // 2 + 1
        self.hp = h
        cin = 64
        self.blocks = []
        for si, (width, nb, stride) in enumerate([(64, 3, 1), (128, 4, 2), (256, 6, 2), (512, 3, 2)]):
            for b in range(nb):
                st = stride if b == 0 else 1
                nm = f"s{si}b{b}"
                h2 = (h + 2 - 3) // st + 1
                self._conv(nm + "c1", (N, h, h, cin, width, 1, 1, 1, 0), seed_cfg)
                self._bn(nm + "n1", width, 0.25, True, False, False)
                self._conv(nm + "c2", (N, h, h, width, width, 3, 3, st, 1), seed_cfg)
                self._bn(nm + "n2", width, 0.25, True, False, False)
                self._conv(nm + "c3", (N, h2, h2, width, 4 * width, 1, 1, 1, 0), seed_cfg)
                self._bn(nm + "n3", 4 * width, 0.25, True, True, True)
                if b == 0:
                    self._conv(nm + "cp", (N, h, h, cin, 4 * width, 1, 1, st, 0), seed_cfg)
                    self._bn(nm + "np", 4 * width, 0.25, False, False, False)
                self.blocks.append((nm, h, h2, cin, width, b == 0))
                h, cin = h2, 4 * width
        self.hl, self.cl = h, cin
        self._conv("fc", (N, 1, 1, cin, classes, 1, 1, 1, 0), seed_cfg)
        self.bias = np.zeros(classes, np.uint16)
        self.vbias = np.zeros(classes, np.uint16)

    def _conv(self, name, desc, seed_cfg):
        _, _, _, C, K, R, S, _, _ = desc
        w = _he(zlib.crc32(f"{seed_cfg}:{name}".encode()), K, R, S, C)
        self.convs[name] = [desc, w, np.zeros_like(w)]

    def _bn(self, name, C, s, relu, residual, zero_gamma):
        one = np.float16(1.0).view(np.uint16)
        g = np.full(C, 0 if zero_gamma else one, np.uint16)
        self.bns[name] = [C, g, np.zeros(C, np.uint16), np.zeros(C, np.uint16), np.zeros(C, np.uint16), s,
                          relu, residual]

    # ------------------------------------------------------------------ layers
    def _cf(self, name, x):
        d, w, _ = self.convs[name]
        V, _, _ = conv_fwd(x, w, *d)
        return f64_to_f16(V)

    def _cb(self, name, x, dy, need_dx=True):
        d, w, _ = self.convs[name]
        gw = f64_to_f16(conv_wgrad(x, dy, *d)[0])
        dx = f64_to_f16(conv_dgrad(dy, w, *d)[0]) if need_dx else None
        return gw, dx

    def _bf(self, name, x, residual=None):
        C, g, b, _, _, s, relu, _ = self.bns[name]
        R = x.size // C
        y, _, _, _ = bn_fwd(x, g, b, residual, R, C, EPS, s, relu)
        return f64_to_f16(y.ravel())

    def _bb(self, name, x, y, dy):
        C, g, _, _, _, s, relu, _ = self.bns[name]
        R = x.size // C
        dx, dg, db, dres = bn_bwd(x, g, dy, y if relu else None, R, C, EPS, s, relu)
        return f64_to_f16(dx.ravel()), f64_to_f16(dg), f64_to_f16(db), f64_to_f16(dres.ravel())

    # ------------------------------------------------------------------ step
    def forward(self, images, labels):
        """Forward pass and loss.  Returns (loss, cache); cache holds every
        layer's binary16 output (per block: x, a1, b1, a2, b2, a3, ap, bp, y),
        the stem's (a0, b0, p0), the pooled features f, the logits and the
        loss gradients (dlogits and dbias, binary64 before storage)."""
        N = self.N
        act = {}
        a0 = self._cf("stem", images)
        b0 = self._bf("bn0", a0)
        p0 = f64_to_f16(maxpool_fwd(b0, N, self.h0, self.h0, 64))
        h = p0
        for nm, hh, h2, cin, width, proj in self.blocks:
            x = h
            a1 = self._cf(nm + "c1", x)
            b1 = self._bf(nm + "n1", a1)
            a2 = self._cf(nm + "c2", b1)
            b2 = self._bf(nm + "n2", a2)
            a3 = self._cf(nm + "c3", b2)
            if proj:
                ap = self._cf(nm + "cp", x)
                bp = self._bf(nm + "np", ap)
            else:
                ap, bp = None, x
            y = self._bf(nm + "n3", a3, residual=bp)
            act[nm] = (x, a1, b1, a2, b2, a3, ap, bp, y)
            h = y
        f = f64_to_f16(avgpool_fwd(h, N, self.hl * self.hl, self.cl))
        logits = self._cf("fc", f)
        loss, dl, db = softmax_xent(logits, self.bias, labels, N, self.classes)
        cache = dict(images=images, a0=a0, b0=b0, p0=p0, act=act, f=f, logits=logits, dlogits=dl, dbias=db)
        return loss, cache

    def backward(self, cache):
        """Backward pass through the cached forward.  Returns (grads, bgrads,
        gbias): binary16 gradients of every conv / FC weight (by conv name),
        of every BatchNorm gamma and beta (by BN name + "g" / "b") and of the FC
        bias.  Also records in the cache each block's output gradient
        (cache["dy"][name]) and the max-pool output's (cache["dp0"])."""
        N, act = self.N, cache["act"]
        dl, gbias = f64_to_f16(cache["dlogits"]), f64_to_f16(cache["dbias"])
        grads, bgrads = {}, {}
        grads["fc"], df = self._cb("fc", cache["f"], dl)
        dy = f64_to_f16(avgpool_bwd(df, N, self.hl * self.hl, self.cl))
        cache["dy"] = dys = {}  # each block's output gradient, as the block received it
        for nm, hh, h2, cin, width, proj in reversed(self.blocks):
            x, a1, b1, a2, b2, a3, ap, bp, y = act[nm]
            dys[nm] = dy
            da3, bgrads[nm + "n3g"], bgrads[nm + "n3b"], dres = self._bb(nm + "n3", a3, y, dy)
            grads[nm + "c3"], db2 = self._cb(nm + "c3", b2, da3)
            da2, bgrads[nm + "n2g"], bgrads[nm + "n2b"], _ = self._bb(nm + "n2", a2, b2, db2)
            grads[nm + "c2"], db1 = self._cb(nm + "c2", b1, da2)
            da1, bgrads[nm + "n1g"], bgrads[nm + "n1b"], _ = self._bb(nm + "n1", a1, b1, db1)
            grads[nm + "c1"], dx1 = self._cb(nm + "c1", x, da1)
            if proj:
                dap, bgrads[nm + "npg"], bgrads[nm + "npb"], _ = self._bb(nm + "np", ap, None, dres)
                grads[nm + "cp"], dxp = self._cb(nm + "cp", x, dap)
                dy = f64_to_f16(f16_to_f64(dx1) + f16_to_f64(dxp))
            else:
                dy = f64_to_f16(f16_to_f64(dx1) + f16_to_f64(dres))
        cache["dp0"] = dy  # the gradient with respect to the max-pool output
        b0 = cache["b0"]
        db0 = f64_to_f16(maxpool_bwd(b0, dy, N, self.h0, self.h0, 64)[0])
        da0, bgrads["bn0g"], bgrads["bn0b"], _ = self._bb("bn0", cache["a0"], b0, db0)
        grads["stem"], _ = self._cb("stem", cache["images"], da0, need_dx=False)
        return grads, bgrads, gbias

    def update(self, grads, bgrads, gbias):
        """The pure-FP16 SGD step on every parameter: weight decay on conv / FC
        weights and the FC bias, none on BatchNorm parameters (Sec. 5.1)."""
        for name, g in grads.items():
            c = self.convs[name]
            c[1], c[2] = sgd_update(c[1], c[2], g, LR, MOMENTUM, WD)
        self.bias, self.vbias = sgd_update(self.bias, self.vbias, gbias, LR, MOMENTUM, WD)
        for name, st in self.bns.items():
            st[1], st[3] = sgd_update(st[1], st[3], bgrads[name + "g"], LR, MOMENTUM, 0)
            st[2], st[4] = sgd_update(st[2], st[4], bgrads[name + "b"], LR, MOMENTUM, 0)

    def step(self, images, labels):
        """One training step (forward, backward, update); returns the loss."""
        loss, cache = self.forward(images, labels)
        self.update(*self.backward(cache))
        return loss

    def param_counts(self):
        """(decayed, not decayed) parameter counts: conv / FC weights and the FC
        bias; BatchNorm gamma and beta."""
        wd = sum(c[1].size for c in self.convs.values()) + self.bias.size
        nowd = sum(2 * st[0] for st in self.bns.values())
        return wd, nowd
