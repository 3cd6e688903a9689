"""GPU parity of pf16_allreduce_combine, the combining step of the fixed-order
FP16 gradient average of data-parallel training (Sec. 5.1, 5.2): bit-exact
against the oracle for world sizes 1 to 1024 (powers of two and not), with
planes at a stride wider than their length, signed zeros, subnormals,
infinities and NaNs (NaN compared as NaN), in place and out of place.  The
ranks' gradients are emulated as planes in one device buffer: nothing waits
on another process."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import dp, pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev, f64, host

pytestmark = pytest.mark.gpu


def planes_for(world, n, stride, seed):
    g = syn.normal_f16(syn.seed_for(8, "dy", seed), (world, stride), 0.01)
    flat = g.reshape(-1)
    rng = np.random.default_rng(seed)
    for code in (0x0000, 0x8000, 0x0001, 0x8001, 0x03FF, 0x7C00, 0xFC00, 0x7E00, 0x7BFF):
        flat[rng.integers(0, flat.size, 7)] = code
    return g


def check_equal(got, ref):
    nan_g, nan_r = np.isnan(f64(got)), np.isnan(f64(ref))
    assert np.array_equal(nan_g, nan_r)
    assert np.array_equal(got[~nan_g], ref[~nan_r])


@pytest.mark.parametrize("world", [1, 2, 3, 4, 5, 8, 16, 17, 32, 64, 128, 1024])
def test_combine_bit_exact(orc, world):
    n = 8 * 613 if world <= 128 else 8 * 31
    stride = n + 24
    g = planes_for(world, n, stride, world)
    scale = dp.inv_world_bits(world)
    out = torch.empty(n, dtype=torch.int16, device="cuda")
    tg = dev(g.reshape(-1))
    pf16.allreduce_combine(tg, world, n, stride, scale, out)
    assert pf16.sync_status() == 0
    ref = orc.allreduce_combine(np.ascontiguousarray(g[:, :n]), scale)
    check_equal(host(out), ref)
    # in place on plane 0: the same bits, the other planes untouched
    pf16.allreduce_combine(tg, world, n, stride, scale, tg)
    assert pf16.sync_status() == 0
    h = host(tg).reshape(world, stride)
    check_equal(h[0, :n], ref)
    assert np.array_equal(h[1:], g[1:])


def test_combine_full_gradient_eight_ranks(orc):
    """The ResNet-50 gradient (25,557,032 values) split over 8 ranks: one
    rank's chunk of 3,194,632 values from 8 planes."""
    world = 8
    chunk = dp.chunk_size(25_557_032, world)
    g = syn.normal_f16(syn.seed_for(8, "x", 99), (world, chunk), 0.01)
    out = torch.empty(chunk, dtype=torch.int16, device="cuda")
    pf16.allreduce_combine(dev(g.reshape(-1)), world, chunk, chunk, dp.inv_world_bits(world), out)
    assert pf16.sync_status() == 0
    assert np.array_equal(host(out), orc.allreduce_combine(g, dp.inv_world_bits(world)))


def test_combine_rejects_bad_arguments():
    t = torch.zeros(1024, dtype=torch.int16, device="cuda")
    for args in [(t, 0, 64, 64), (t, 1025, 64, 64), (t, 2, 60, 64), (t, 2, 64, 60), (t, 2, 64, 68)]:
        with pytest.raises(pf16.PF16Error):
            pf16.allreduce_combine(args[0], args[1], args[2], args[3], 0x3800, t[512:])
    with pytest.raises(pf16.PF16Error):  # out overlapping plane 1
        pf16.allreduce_combine(t, 2, 64, 64, 0x3800, t[64:])
    with pytest.raises(pf16.PF16Error):  # misaligned
        pf16.allreduce_combine(t[1:], 2, 64, 64, 0x3800, t[512:])
    pf16.allreduce_combine(t, 2, 0, 64, 0x3800, t[512:])  # n = 0: nothing to do
    assert pf16.sync_status() == 0


def test_step_with_exchange_hook():
    """The training step's exchange hook runs before the update on both
    gradient arenas.  Two emulated ranks holding the same gradient average to
    exactly that gradient (rn(rn(g + g) * 0.5) = g without overflow), so the
    step is bit-identical to the step without an exchange."""
    from paper_1911_07384_gb300.resnet50 import ResNet50

    calls = []

    def two_identical_ranks(g):
        n = g.numel()
        stride = (n + 7) // 8 * 8
        planes = torch.zeros(2 * stride, dtype=torch.int16, device=g.device)
        planes[:n].copy_(g)
        planes[stride:stride + n].copy_(g)
        pf16.allreduce_combine(planes, 2, stride, stride, dp.inv_world_bits(2), planes)
        g.copy_(planes[:n])
        calls.append(n)

    nets = []
    for ex in (None, two_identical_ranks):
        net = ResNet50(batch=2, image=64, seed_cfg=4, exchange=ex)
        net.set_batch(syn.images_f16(syn.seed_for(4, "x"), 2, 64, 64, 3), syn.labels(syn.seed_for(4, "labels"), 2))
        net.step()
        net.step()
        assert pf16.sync_status() == 0
        nets.append(net)
    assert calls == [nets[1].wd.g.numel(), nets[1].nowd.g.numel()] * 2
    for a in ("wd", "nowd"):
        for t in ("w", "v", "g"):
            assert torch.equal(getattr(getattr(nets[0], a), t), getattr(getattr(nets[1], a), t))
