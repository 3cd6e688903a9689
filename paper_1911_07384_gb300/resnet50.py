"""ResNet-50 v1.5 pure-FP16 training step on top of libpf16 (host code only).

The network, the recipe and the FP16 rules are the paper's (Sec. 5.1, 5.2,
4.2): ResNet-50 trained with PyTorch's ImageNet recipe -- SGD with momentum
0.9, weight decay 1e-4 on conv/FC parameters and none on BatchNorm parameters,
gamma of the last BatchNorm of every residual block initialised to zero --
with every tensor and every operation in FP16, no master copy, and the output
of every BatchNorm inside a residual block multiplied by 0.25 (the stem's
BatchNorm is left as it is).

Every op of the step is one call into libpf16 on the current CUDA stream;
this module only lays out the buffers (torch supplies device memory) and
issues the calls, so the whole step can be captured once in a CUDA graph and
replayed.  Layout: activations NHWC, weights KRSC, parameters in two flat
16-byte-aligned FP16 arenas (decayed / not decayed), each with a gradient and a
momentum twin, so the update is two pf16_sgd_update calls.
"""
from __future__ import annotations

import numpy as np
import torch

from . import pf16
from . import synthetic as syn

LR = 0x2E66       # 0.1 in binary16 (0.0999755859375)
MOMENTUM = 0x3B33  # 0.9 (0.89990234375)
WD = 0x068E       # 1e-4 (1.00016594e-4)
EPS = 0x00A8      # 1e-5 (subnormal, 1.00135803e-5)
S_BLOCK = 0x3400  # 0.25: BatchNorms inside residual blocks
S_STEM = 0x3C00   # 1.0: the stem BatchNorm

STAGES = [(64, 3, 1), (128, 4, 2), (256, 6, 2), (512, 3, 2)]  # width, blocks, stride


def conv_shapes(batch=256, image=224, classes=1000):
    """(name, (N, H, W, C, K, R, S, stride, pad)) of every conv of the network, in
    forward order, without allocating anything."""
    out = [("stem", (batch, image, image, 3, 64, 7, 7, 2, 3))]
    h = (image + 6 - 7) // 2 + 1
    h = (h - 1) // 2 + 1
    cin = 64
    for si, (width, nb, stride) in enumerate(STAGES):
        for b in range(nb):
            st = stride if b == 0 else 1
            h2 = (h + 2 - 3) // st + 1
            nm = f"s{si + 1}b{b}"
            out.append((nm + ".conv1", (batch, h, h, cin, width, 1, 1, 1, 0)))
            out.append((nm + ".conv2", (batch, h, h, width, width, 3, 3, st, 1)))
            out.append((nm + ".conv3", (batch, h2, h2, width, 4 * width, 1, 1, 1, 0)))
            if b == 0:
                out.append((nm + ".proj", (batch, h, h, cin, 4 * width, 1, 1, st, 0)))
            h, cin = h2, 4 * width
    out.append(("fc", (batch, 1, 1, cin, classes, 1, 1, 1, 0)))
    return out


def _a8(n):
    return (n + 7) // 8 * 8


def _f16(x):
    return torch.from_numpy(np.ascontiguousarray(x).view(np.int16))


class Arena:
    """Flat FP16 parameter arena with gradient and momentum twins."""

    def __init__(self, name):
        self.name = name
        self.size = 0
        self.slots = []

    def add(self, numel):
        off = self.size
        self.size += _a8(numel)
        self.slots.append((off, numel))
        return off

    def allocate(self, device):
        n = max(self.size, 8)
        self.w = torch.zeros(n, dtype=torch.int16, device=device)
        self.g = torch.zeros(n, dtype=torch.int16, device=device)
        self.v = torch.zeros(n, dtype=torch.int16, device=device)

    def view(self, which, off, numel):
        return getattr(self, which)[off:off + numel]


class Conv:
    def __init__(self, net, n, h, w, c, k, r, s, stride, pad):
        self.net = net
        self.desc = pf16.conv_desc(n, h, w, c, k, r, s, stride, pad)
        self.P, self.Q = self.desc.out_hw()
        self.numel = k * r * s * c
        self.off = net.wd.add(self.numel)
        self.flops = 2 * n * self.P * self.Q * k * c * r * s
        net.convs.append(self)

    def bind(self):
        a = self.net.wd
        self.w, self.gw = a.view("w", self.off, self.numel), a.view("g", self.off, self.numel)
        # BatchNorm statistics of the output, written by the forward GEMM's epilogue
        size = pf16.conv_bnstats_size(self.desc)
        self.stats = torch.empty(size, dtype=torch.uint8, device=a.w.device) if size else None
        # backward statistics of the BatchNorm whose output gradient the data gradient is
        # (not for the 3x3 64 -> 64 layers: their data gradient alone runs at about
        # twice the rate it keeps with the statistics epilogue, which is bound by the
        # latency of its per-element work, and the BatchNorm's own statistics pass
        # costs less than the difference)
        # Stride-2 data gradients take them only where dx is large: at 56x56x128 (batch
        # 256) the fused epilogue (160 us) undercuts the plain data gradient plus the
        # BatchNorm's own statistics pass (115 + 74 us); at 28x28x256 the two are even
        # and at 14x14x512 the separate pass is cheaper.
        d = self.desc
        halo64 = d.r == 3 and d.s == 3 and d.stride == 1 and d.c == 64 and d.k == 64
        small_strided = d.stride != 1 and d.n * d.h * d.w * d.c < (1 << 26)
        size = pf16.conv_dgrad_bnstats_size(d) if d.c != 3 and not halo64 and not small_strided else 0
        self.dstats = torch.empty(size, dtype=torch.uint8, device=a.w.device) if size else None

    def fwd(self, x, y, with_stats=False, bn_in=None):
        """bn_in: the BN layer whose input x is; this conv applies it in its
        operand path (pf16_conv_fwd_bnin) and writes its ReLU mask."""
        if bn_in is not None:
            self.net.call("conv_fwd", self, pf16.conv_fwd_bnin, self.desc, x, bn_in.operand(with_mask=True), self.w,
                          y, self.stats if with_stats else None)
        elif with_stats:
            self.net.call("conv_fwd", self, pf16.conv_fwd_bnstats, self.desc, x, self.w, y, self.stats,
                          self.net.ws)
        else:
            self.net.call("conv_fwd", self, pf16.conv_fwd, self.desc, x, self.w, y, self.net.ws)

    def dgrad(self, dy, dx, accumulate=False, bn=None, add=None):
        """bn: (BN layer, its input x) when dx is that BatchNorm's output gradient and
        this layer takes its backward statistics (see bind); see BN.bwd(conv=).
        add (with bn, 1x1 only): (tensor, bit mask) added to the data gradient where
        the mask's bit is set -- an identity shortcut's share of dx."""
        if bn is not None and add is not None:
            layer, x = bn
            self.net.call("conv_dgrad", self, pf16.conv_dgrad_bnstats_add, self.desc, dy, self.w, dx, x,
                          layer.mask, layer.mean, layer.invstd, add[0], add[1], self.dstats)
        elif bn is not None:
            layer, x = bn
            self.net.call("conv_dgrad", self, pf16.conv_dgrad_bnstats, self.desc, dy, self.w, dx, x, layer.mask,
                          layer.mean, layer.invstd, self.dstats)
        else:
            self.net.call("conv_dgrad", self, pf16.conv_dgrad, self.desc, dy, self.w, dx, None,
                          pf16.PF16_ACCUMULATE if accumulate else 0)

    def fuses_bwd_stats(self):
        return self.dstats is not None

    def wgrad(self, x, dy, bn_in=None):
        """bn_in: as in fwd -- x is that BatchNorm's input."""
        net = self.net

        def call(ws):
            if bn_in is not None:
                net.call("conv_wgrad", self, pf16.conv_wgrad_bnin, self.desc, x, bn_in.operand(), dy, self.gw, ws)
            else:
                net.call("conv_wgrad", self, pf16.conv_wgrad, self.desc, x, dy, self.gw, ws)

        if net.side is None:
            call(net.ws)
            return
        # only the update reads the weight gradient: it runs on a branch of its own
        # (with its own workspace), off the chain of data gradients and BatchNorms
        net.side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(net.side):
            call(net.ws_w)


class BN:
    def __init__(self, net, n, h, w, c, post_scale, relu, residual=False, zero_gamma=False, swap=False):
        self.net = net
        flags = (pf16.PF16_BN_RELU if relu else 0) | (pf16.PF16_BN_RESIDUAL if residual else 0)
        flags |= pf16.PF16_BN_SWAP if swap else 0
        self.swap = swap
        self.desc = pf16.bn_desc(n, h, w, c, EPS, post_scale, flags)
        self.c = c
        self.zero_gamma = zero_gamma
        self.post_scale = post_scale
        self.relu = relu
        self.fused_apply = False  # applied in the next conv's operand path (the output is never stored)
        self.g_off = net.nowd.add(c)
        self.b_off = net.nowd.add(c)
        self.elems = n * h * w * c
        net.bns.append(self)

    def bind(self, device):
        a = self.net.nowd
        self.gamma, self.beta = a.view("w", self.g_off, self.c), a.view("w", self.b_off, self.c)
        self.dgamma, self.dbeta = a.view("g", self.g_off, self.c), a.view("g", self.b_off, self.c)
        self.mean = torch.empty(self.c, dtype=torch.int16, device=device)
        self.invstd = torch.empty(self.c, dtype=torch.int16, device=device)
        # ReLU decisions as one bit per element: the backward reads these
        # instead of the saved output
        relu = bool(self.desc.flags & pf16.PF16_BN_RELU)
        self.mask = torch.empty(self.elems // 8, dtype=torch.uint8, device=device) if relu else None

    def fwd(self, x, y, residual=None, conv=None):
        """conv: the layer whose fwd(with_stats=True) produced x (its statistics are used).
        y None: statistics only (mean, invstd), for a conv that applies this
        BatchNorm in its operand path and writes the ReLU mask."""
        self.net.call("bn_fwd", self, pf16.bn_fwd_bwd, self.desc, 0, self.net.ws, x=x, gamma=self.gamma,
                      beta=self.beta, residual=residual, y=y, mean=self.mean, invstd=self.invstd,
                      relu_mask=self.mask if y is not None else None,
                      conv_stats=conv.stats if conv is not None else None)

    def operand(self, with_mask=False):
        """This BatchNorm as a conv's operand transform (pf16_bn_operand)."""
        return pf16.bn_operand(self.mean, self.invstd, self.gamma, self.beta, self.post_scale, self.relu,
                               self.mask if with_mask else None)

    def bwd(self, x, y_saved, dy, dx, dresidual=None, conv=None, residual=None):
        """conv: the layer whose dgrad(bn=(self, x)) produced dy (its statistics are used);
        residual: the forward's residual input (read by the swap variant's backward)."""
        self.net.call("bn_bwd", self, pf16.bn_fwd_bwd, self.desc, 1, self.net.ws, x=x, gamma=self.gamma,
                      mean=self.mean, invstd=self.invstd, dy=dy, relu_mask=self.mask, dx=dx,
                      dgamma=self.dgamma, dbeta=self.dbeta, dresidual=dresidual,
                      conv_stats=conv.dstats if conv is not None else None,
                      residual=residual if self.desc.flags & pf16.PF16_BN_SWAP else None)
        self.fused_bwd = conv is not None


class Bottleneck:
    def __init__(self, net, n, h, cin, width, stride, proj, swap=False):
        self.cin, self.width, self.stride = cin, width, stride
        self.net = net
        cout = 4 * width
        self.conv1 = Conv(net, n, h, h, cin, width, 1, 1, 1, 0)
        self.bn1 = BN(net, n, h, h, width, S_BLOCK, relu=True)
        self.conv2 = Conv(net, n, h, h, width, width, 3, 3, stride, 1)
        h2 = self.conv2.P
        self.bn2 = BN(net, n, h2, h2, width, S_BLOCK, relu=True)
        self.conv3 = Conv(net, n, h2, h2, width, cout, 1, 1, 1, 0)
        # swap: Sec. 4.1's variant of the block's last BatchNorm, gamma * (s * xhat + shortcut) + beta
        self.bn3 = BN(net, n, h2, h2, cout, S_BLOCK, relu=True, residual=True, zero_gamma=True, swap=swap)
        self.proj = proj
        if proj:
            self.convp = Conv(net, n, h, h, cin, cout, 1, 1, stride, 0)
            self.bnp = BN(net, n, h2, h2, cout, S_BLOCK, relu=False)
        self.h, self.h2, self.n, self.cout = h, h2, n, cout
        # the layer whose data gradient carries bn3's backward statistics (the
        # next block's conv1, set by that block's backward), or None
        self.bn3_stats_conv = None
        # bn2 applied in conv3's operand path (forward and weight gradient): its
        # output b2 is never stored
        self.fuse_bn2 = net.bn_in_operand
        self.bn2.fused_apply = self.fuse_bn2

    def allocate(self, dev):
        n, h, h2, w, c = self.n, self.h, self.h2, self.width, self.cout
        e = lambda *s: torch.empty(int(np.prod(s)), dtype=torch.int16, device=dev)
        self.a1, self.b1 = e(n, h, h, w), e(n, h, h, w)
        self.a2 = e(n, h2, h2, w)
        self.b2 = None if self.fuse_bn2 else e(n, h2, h2, w)
        self.a3, self.y = e(n, h2, h2, c), e(n, h2, h2, c)
        self.dy = e(n, h2, h2, c)  # gradient w.r.t. y (written by the next block)
        self.da3 = e(n, h2, h2, c)
        self.db2, self.da2 = e(n, h2, h2, w), e(n, h2, h2, w)
        self.db1, self.da1 = e(n, h, h, w), e(n, h, h, w)
        if self.proj:
            self.ap, self.bp = e(n, h2, h2, c), e(n, h2, h2, c)
            self.dres, self.dap = e(n, h2, h2, c), e(n, h2, h2, c)

    def forward(self, x):
        self.x = x
        self.conv1.fwd(x, self.a1, with_stats=True)
        self.bn1.fwd(self.a1, self.b1, conv=self.conv1)
        self.conv2.fwd(self.b1, self.a2, with_stats=True)
        if self.fuse_bn2:  # bn2's statistics only; conv3 applies it to its operand
            self.bn2.fwd(self.a2, None, conv=self.conv2)
            self.conv3.fwd(self.a2, self.a3, with_stats=True, bn_in=self.bn2)
        else:
            self.bn2.fwd(self.a2, self.b2, conv=self.conv2)
            self.conv3.fwd(self.b2, self.a3, with_stats=True)
        if self.proj:
            self.convp.fwd(x, self.ap, with_stats=True)
            self.bnp.fwd(self.ap, self.bp, conv=self.convp)
            self.bn3.fwd(self.a3, self.y, residual=self.bp, conv=self.conv3)
        else:
            self.bn3.fwd(self.a3, self.y, residual=x, conv=self.conv3)
        return self.y

    def fuses_prev(self, prev):
        """Whether this block's first data gradient can produce the whole of
        dL/dx (shortcut share added in its epilogue) and, with it, the backward
        statistics of prev's last BatchNorm (prev: the block whose output is
        this block's input)."""
        return (not self.proj and self.conv1.fuses_bwd_stats() and prev.bn3.mask is not None
                and self.bn3.mask is not None and not prev.bn3.swap and not self.bn3.swap)

    def backward(self, dx, prev=None):
        """self.dy holds dL/dy; writes dL/dx into dx.  prev: the block whose
        output is this block's input, or None."""
        fuse = prev is not None and self.fuses_prev(prev)
        bn3_conv = self.bn3_stats_conv
        if self.proj:
            self.bn3.bwd(self.a3, self.y, self.dy, self.da3, dresidual=self.dres, residual=self.bp,
                         conv=bn3_conv)
        else:  # identity shortcut: its gradient (dy where the ReLU passed) is the start of dx
            self.bn3.bwd(self.a3, self.y, self.dy, self.da3, dresidual=None if fuse else dx, residual=self.x,
                         conv=bn3_conv)
        if self.fuse_bn2:
            self.conv3.wgrad(self.a2, self.da3, bn_in=self.bn2)
        else:
            self.conv3.wgrad(self.b2, self.da3)
        # the data gradients also reduce the next BatchNorm's backward statistics
        self.conv3.dgrad(self.da3, self.db2, bn=(self.bn2, self.a2))
        self.bn2.bwd(self.a2, self.b2, self.db2, self.da2, conv=self.conv3)
        self.conv2.wgrad(self.b1, self.da2)
        c2 = self.conv2 if self.conv2.fuses_bwd_stats() else None
        self.conv2.dgrad(self.da2, self.db1, bn=(self.bn1, self.a1) if c2 else None)
        self.bn1.bwd(self.a1, self.b1, self.db1, self.da1, conv=c2)
        self.conv1.wgrad(self.x, self.da1)
        if self.proj:
            self.conv1.dgrad(self.da1, dx)
            self.bnp.bwd(self.ap, None, self.dres, self.dap)
            self.convp.wgrad(self.x, self.dap)
            self.convp.dgrad(self.dap, dx, accumulate=True)
        elif fuse:
            # dx = shortcut share + data gradient in one epilogue, which also
            # reduces prev.bn3's backward statistics
            self.conv1.dgrad(self.da1, dx, bn=(prev.bn3, prev.a3), add=(self.dy, self.bn3.mask))
            prev.bn3_stats_conv = self.conv1
        else:
            self.conv1.dgrad(self.da1, dx, accumulate=True)
            if prev is not None:
                prev.bn3_stats_conv = None


def layer_label(layer):
    """Shape label of a Conv or BN layer ("n,h,w,c[,k,r,s,stride,pad]"), "-" for none."""
    d = getattr(layer, "desc", None)
    if d is None:
        return "-" if layer is None else str(layer)
    keep = ("n", "h", "w", "c", "k", "r", "s", "stride", "pad")
    return ",".join(str(getattr(d, f[0])) for f in d._fields_ if f[0] in keep)


def nvtx_hook(kind, layer, fn, *args, **kw):
    """Instrumentation hook (ResNet50(hook=nvtx_hook)): wraps each library call
    in an NVTX range "pf16:<kind>:<layer>", so that profilers can attribute
    kernels to calls (e.g. ncu --nvtx --nvtx-include "pf16:bn_bwd*/").  The
    ranges are host-side only; a step captured into a CUDA graph carries none."""
    torch.cuda.nvtx.range_push(f"pf16:{kind}:{layer_label(layer)}")
    try:
        return fn(*args, **kw)
    finally:
        torch.cuda.nvtx.range_pop()


class ResNet50:
    """Buffers and call sequence of one pure-FP16 ResNet-50 training step."""

    def __init__(self, batch=256, image=224, classes=1000, device="cuda", seed_cfg=4, hook=None, bn_swap=False,
                 wgrad_branch=False, exchange=None, bn_in_operand=False, stem_fused=True):
        """wgrad_branch: issue the weight gradients on a second stream that joins
        before the update (in a captured step graph: a parallel branch), so that
        they fill the gaps of the data-gradient chain; off, every call runs on the
        current stream in program order (what per-call timing needs).
        exchange: data-parallel training (Sec. 5.1): a callable applied, before
        the update, to each flat gradient arena (decayed, then not decayed) to
        average it over the ranks in place, e.g. functools.partial(
        dp.allreduce_mean_, group=g); None on one GPU.
        bn_in_operand: each block's second BatchNorm is applied in its last
        conv's operand path (bit-identical results, its output never stored);
        off by default: on GB300 the conv's transform costs more than the
        apply pass it replaces (the 1x1 convs re-transform each operand tile
        once per tile of the other GEMM dimension, and their epilogues already
        fill the SM's issue slots).
        stem_fused: the stem's BatchNorm, ReLU and max pooling forward run as
        one call (pf16_bn_relu_maxpool_fwd: bit-identical results, the
        BatchNorm's output never stored)."""
        self.N, self.image, self.classes, self.device = batch, image, classes, device
        self.stem_fused = stem_fused
        self.hook = hook  # optional callable(kind, layer, fn, *args) used for instrumentation
        self.exchange = exchange
        self.bn_in_operand = bn_in_operand
        self.side = torch.cuda.Stream(device=device) if wgrad_branch else None
        self.wd, self.nowd = Arena("decayed"), Arena("no-decay")
        self.convs, self.bns = [], []
        N = batch
        self.stem = Conv(self, N, image, image, 3, 64, 7, 7, 2, 3)
        h = self.stem.P
        self.bn0 = BN(self, N, h, h, 64, S_STEM, relu=True)
        self.h0 = h
        self.hp = (h - 1) // 2 + 1
        h, cin = self.hp, 64
        self.blocks = []
        for width, nb, stride in STAGES:
            for b in range(nb):
                blk = Bottleneck(self, N, h, cin, width, stride if b == 0 else 1, proj=(b == 0), swap=bn_swap)
                self.blocks.append(blk)
                h, cin = blk.h2, 4 * width
        self.hl, self.cl = h, cin
        self.fc = Conv(self, N, 1, 1, cin, classes, 1, 1, 1, 0)
        self.bias_off = self.wd.add(classes)
        self.seed_cfg = seed_cfg
        self._allocate()
        self._init_params()

    # ------------------------------------------------------------- buffers
    def _allocate(self):
        dev, N = self.device, self.N
        e = lambda *s: torch.empty(int(np.prod(s)), dtype=torch.int16, device=dev)
        self.wd.allocate(dev)
        self.nowd.allocate(dev)
        for c in self.convs:
            c.bind()
        for b in self.bns:
            b.bind(dev)
        self.bias = self.wd.view("w", self.bias_off, self.classes)
        self.dbias = self.wd.view("g", self.bias_off, self.classes)
        h0, hp = self.h0, self.hp
        self.x = e(N, self.image, self.image, 3)
        self.labels = torch.zeros(N, dtype=torch.int32, device=dev)
        self.a0, self.p0 = e(N, h0, h0, 64), e(N, hp, hp, 64)
        self.dp0, self.da0 = e(N, hp, hp, 64), e(N, h0, h0, 64)
        # the stem BatchNorm's output (not stored when fused with the pooling) and its gradient
        self.b0 = None if self.stem_fused else e(N, h0, h0, 64)
        self.db0 = e(N, h0, h0, 64)
        # position of each pooling window's maximum, kept from the forward for the backward
        self.pool_arg = torch.empty(N * hp * hp * 64, dtype=torch.uint8, device=dev)
        for b in self.blocks:
            b.allocate(dev)
        self.f = e(N, self.cl)
        self.logits = e(N, self.classes)
        self.dlogits = e(N, self.classes)
        self.df = e(N, self.cl)
        self.loss = e(1)
        ws = 0
        for c in self.convs:
            ws = max(ws, pf16.conv_workspace_size(c.desc, pf16.PF16_PASS_FWD),
                     pf16.conv_workspace_size(c.desc, pf16.PF16_PASS_WGRAD))
        for b in self.bns:
            ws = max(ws, pf16.bn_workspace_size(b.desc))
        ws = max(ws, pf16.softmax_xent_workspace_size(N, self.classes))
        self.ws = torch.empty(ws, dtype=torch.uint8, device=dev)
        # the weight gradients' own scratch when they run on the side branch
        wsw = max(pf16.conv_workspace_size(c.desc, pf16.PF16_PASS_WGRAD) for c in self.convs)
        self.ws_w = torch.empty(max(wsw, 256), dtype=torch.uint8, device=dev) if self.side is not None else None

    def _init_params(self):
        """He-normal conv / FC weights (std sqrt(2 / fan_in)), FC bias 0, BN gamma
        1 and beta 0, gamma 0 in the last BatchNorm of every block; momentum +0."""
        for i, c in enumerate(self.convs):
            d = c.desc
            wbits = syn.he_normal_f16(syn.seed_for(self.seed_cfg, "w", i), d.k, d.r, d.s, d.c)
            c.w.copy_(_f16(wbits.ravel()))
        self.bias.zero_()
        one = int(np.float16(1.0).view(np.uint16))
        for b in self.bns:
            b.gamma.fill_(0 if b.zero_gamma else one)
            b.beta.zero_()
        self.wd.v.zero_()
        self.nowd.v.zero_()

    def set_batch(self, images_bits, labels):
        self.x.copy_(_f16(images_bits.ravel()))
        self.labels.copy_(torch.from_numpy(np.ascontiguousarray(labels, np.int32)))

    # ------------------------------------------------------------- calls
    def call(self, kind, layer, fn, *args, **kw):
        if self.hook is not None:
            return self.hook(kind, layer, fn, *args, **kw)
        return fn(*args, **kw)

    def forward(self):
        self.stem.fwd(self.x, self.a0, with_stats=True)
        if self.stem_fused:
            b = self.bn0
            self.call("bn_pool_fwd", b, pf16.bn_relu_maxpool_fwd, b.desc, self.ws, self.p0, self.pool_arg,
                      x=self.a0, gamma=b.gamma, beta=b.beta, mean=b.mean, invstd=b.invstd, relu_mask=b.mask,
                      conv_stats=self.stem.stats)
        else:
            self.bn0.fwd(self.a0, self.b0, conv=self.stem)
            self.call("maxpool_fwd", None, pf16.maxpool_fwd_argmax, self.b0, self.p0, self.pool_arg, self.N,
                      self.h0, self.h0, 64)
        h = self.p0
        for b in self.blocks:
            h = b.forward(h)
        self.call("avgpool_fwd", None, pf16.avgpool_fwd, h, self.f, self.N, self.hl * self.hl, self.cl)
        self.fc.fwd(self.f, self.logits)
        self.call("softmax_xent", None, pf16.softmax_xent, self.logits, self.bias, self.labels, self.N,
                  self.classes, self.loss, self.dlogits, self.dbias, self.ws)

    def backward(self):
        self.fc.wgrad(self.f, self.dlogits)
        self.fc.dgrad(self.dlogits, self.df)
        last = self.blocks[-1]
        self.call("avgpool_bwd", None, pf16.avgpool_bwd, self.df, last.dy, self.N, self.hl * self.hl,
                  self.cl)
        for i in range(len(self.blocks) - 1, -1, -1):
            dx = self.blocks[i - 1].dy if i > 0 else self.dp0
            self.blocks[i].backward(dx, self.blocks[i - 1] if i > 0 else None)
        # the pooling's backward, then the stem BatchNorm's (ReLU decisions from
        # its bit mask: with the fused forward its output is not stored)
        self.call("maxpool_bwd", None, pf16.maxpool_bwd_argmax, self.pool_arg, self.dp0, self.db0, self.N,
                  self.h0, self.h0, 64)
        self.bn0.bwd(self.a0, self.b0, self.db0, self.da0)
        self.stem.wgrad(self.x, self.da0)

    def update(self):
        if self.side is not None:  # every weight gradient is in before the update reads it
            torch.cuda.current_stream().wait_stream(self.side)
        if self.exchange is not None:  # the ranks' gradients averaged, in a fixed FP16 order
            self.call("exchange", None, self.exchange, self.wd.g)
            self.call("exchange", None, self.exchange, self.nowd.g)
        self.call("sgd", None, pf16.sgd_update, self.wd.w, self.wd.v, self.wd.g, LR, MOMENTUM, WD)
        self.call("sgd", None, pf16.sgd_update, self.nowd.w, self.nowd.v, self.nowd.g, LR, MOMENTUM, 0)

    def step(self):
        self.forward()
        self.backward()
        self.update()

    # ------------------------------------------------------------- accounting
    def conv_flops(self):
        """Algorithmic convolution FLOPs of one step: 2*N*P*Q*K*C*R*S for each of
        forward, data gradient (not for the stem) and weight gradient."""
        total = 0
        for c in self.convs:
            total += c.flops * (2 if c is self.stem else 3)
        return total

    def param_count(self):
        return (sum(n for _, n in self.wd.slots), sum(n for _, n in self.nowd.slots))
