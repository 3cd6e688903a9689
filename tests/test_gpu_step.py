"""The full ResNet-50 pure-FP16 training step on the GPU: structural
invariants that hold exactly, and agreement with the oracle's composition of
the same step (same weights and inputs) on a small image size."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from paper_1911_07384_gb300.resnet50 import ResNet50
from gpu_util import f64, host

pytestmark = pytest.mark.gpu


def small_net(batch=2, image=64):
    net = ResNet50(batch=batch, image=image, seed_cfg=4)
    net.set_batch(syn.images_f16(syn.seed_for(4, "x"), batch, image, image, 3),
                  syn.labels(syn.seed_for(4, "labels"), batch))
    return net


def test_identity_blocks_pass_input_through_at_init():
    """Zero gamma in the last BatchNorm of each block (Sec. 5.1) makes every
    identity-shortcut block output equal its input exactly."""
    net = small_net()
    net.forward()
    assert pf16.sync_status() == 0
    for b in net.blocks:
        if not b.proj:
            assert torch.equal(b.y, b.x)


def test_parameter_count_and_flops():
    net = small_net()
    wd, nowd = net.param_count()
    assert wd == 25_502_912 + 1000 and nowd == 53_120
    assert net.conv_flops() > 0


def test_step_matches_oracle_composition(orc):
    """Initial loss within FP16 error of the oracle's step with the same
    weights; the loss is near ln(1000) at initialisation."""
    from oracle import resnet50 as oresnet

    net = small_net()
    onet = oresnet.OracleResNet50(2, 64, 1000)
    assert len(onet.convs) == len(net.convs)
    for (name, c), gc in zip(onet.convs.items(), net.convs):
        c[1] = host(gc.w).reshape(c[1].shape)
    imgs = syn.images_f16(syn.seed_for(4, "x"), 2, 64, 64, 3)
    labs = syn.labels(syn.seed_for(4, "labels"), 2)
    net.step()
    assert pf16.sync_status() == 0
    gpu_loss = float(f64(host(net.loss))[0])
    ref_loss = onet.step(imgs, labs)
    assert abs(gpu_loss - ref_loss) <= 0.02 * ref_loss + 0.02, (gpu_loss, ref_loss)
    assert abs(ref_loss - np.log(1000)) < 2.5
    # a second step sees the updated weights: both implementations moved the same way
    net.step()
    gpu2 = float(f64(host(net.loss))[0])
    ref2 = onet.step(imgs, labs)
    assert abs(gpu2 - ref2) <= 0.05 * ref2 + 0.05, (gpu2, ref2)


def test_graph_replay_is_deterministic():
    net = small_net()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        net.step()
    torch.cuda.synchronize()
    w0 = net.wd.w.clone()
    g = torch.cuda.CUDAGraph()
    # capture without running, then compare a replay against an eager step from the same state
    saved = [t.clone() for t in (net.wd.w, net.wd.v, net.nowd.w, net.nowd.v)]
    with torch.cuda.graph(g, stream=s):
        net.step()
    for t, v in zip((net.wd.w, net.wd.v, net.nowd.w, net.nowd.v), saved):
        t.copy_(v)
    g.replay()
    torch.cuda.synchronize()
    after_graph = net.wd.w.clone()
    for t, v in zip((net.wd.w, net.wd.v, net.nowd.w, net.nowd.v), saved):
        t.copy_(v)
    with torch.cuda.stream(s):
        net.step()
    torch.cuda.synchronize()
    assert torch.equal(after_graph, net.wd.w)
    assert not torch.equal(w0, net.wd.w)


def test_swap_variant_step():
    """The BN-swap variant (Sec. 4.1) in every block's last BatchNorm: with the
    zero-gamma initialisation each block computes ReLU(0 * (s xhat + r) + 0) = 0,
    so every block output is exactly zero, the logits are the (zero) bias and
    the first loss is the uniform value; the step then runs and replays."""
    net = ResNet50(batch=2, image=64, seed_cfg=4, bn_swap=True)
    net.set_batch(syn.images_f16(syn.seed_for(4, "x"), 2, 64, 64, 3), syn.labels(syn.seed_for(4, "labels"), 2))
    net.forward()
    assert pf16.sync_status() == 0
    for b in net.blocks:
        assert not torch.any(b.y)
    net.step()
    assert pf16.sync_status() == 0
    loss = float(f64(host(net.loss))[0])
    assert abs(loss - np.log(1000)) < 2 ** -8 * np.log(1000)
    net.step()
    assert pf16.sync_status() == 0
    assert np.isfinite(float(f64(host(net.loss))[0]))


def test_weight_gradient_branch_is_bit_identical():
    """Weight gradients on a side branch that joins before the update (the
    captured step graph of bench.py) give the same bits as program order: two
    steps, every weight, momentum and loss compared exactly."""
    results = []
    for branch in (False, True):
        net = ResNet50(batch=2, image=64, seed_cfg=4, wgrad_branch=branch)
        net.set_batch(syn.images_f16(syn.seed_for(4, "x"), 2, 64, 64, 3), syn.labels(syn.seed_for(4, "labels"), 2))
        stream = torch.cuda.Stream()
        with torch.cuda.stream(stream):
            net.step()
            net.step()
        torch.cuda.synchronize()
        assert pf16.sync_status(stream) == 0
        results.append([t.clone() for t in (net.wd.w, net.wd.v, net.nowd.w, net.nowd.v, net.loss)])
    for a, b in zip(*results):
        assert torch.equal(a, b)


def test_bn_in_operand_path_step_is_bit_identical():
    """Each block's second BatchNorm applied in its last conv's operand path
    against the same BatchNorm stored and read back (the default): two steps
    at batch 4 on 64 x 64 and one at batch 8 on 96 x 96 (a ragged last tile in
    stage 4), every weight, momentum and loss compared exactly."""
    for batch, image, steps in ((4, 64, 2), (8, 96, 1)):
        results = []
        for fused in (False, True):
            net = ResNet50(batch=batch, image=image, seed_cfg=4, bn_in_operand=fused)
            net.set_batch(syn.images_f16(syn.seed_for(4, "x"), batch, image, image, 3),
                          syn.labels(syn.seed_for(4, "labels"), batch))
            for _ in range(steps):
                net.step()
            torch.cuda.synchronize()
            assert pf16.sync_status() == 0
            assert all(b.fuse_bn2 == fused and (b.b2 is None) == fused for b in net.blocks)
            results.append([t.clone() for t in (net.wd.w, net.wd.v, net.nowd.w, net.nowd.v, net.loss)])
        for a, b in zip(*results):
            assert torch.equal(a, b)
