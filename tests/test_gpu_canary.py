"""Out-of-bounds writes, caught without a sanitizer: every output and every
workspace of a call sits inside a larger buffer whose guard zones before and
after hold a canary pattern, and the guards must be intact after the call.
Shapes have ragged tails (partial M and N tiles, odd sizes, stride phases)."""
import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev

pytestmark = pytest.mark.gpu

GUARD = 64          # int16 elements on each side (128 bytes, keeps 16-byte alignment)
CANARY = 0x5A5A


def guarded(n):
    buf = torch.full((GUARD + n + GUARD,), CANARY, dtype=torch.int16, device="cuda")
    return buf, buf[GUARD:GUARD + n]


def guarded_ws(nbytes):
    if not nbytes:
        return None, None
    buf = torch.full((256 + int(nbytes) + 256,), 0xA5, dtype=torch.uint8, device="cuda")
    return buf, buf[256:256 + int(nbytes)]


def intact(buf, n):
    h = buf.cpu()
    return bool((h[:GUARD] == CANARY).all()) and bool((h[GUARD + n:] == CANARY).all())


def intact_ws(buf, nbytes):
    if buf is None:
        return True
    h = buf.cpu()
    return bool((h[:256] == 0xA5).all()) and bool((h[256 + int(nbytes):] == 0xA5).all())


SHAPES = [
    (1, 7, 7, 64, 64, 3, 3, 1, 1),       # halo engine, one partial tile
    (2, 9, 9, 64, 128, 3, 3, 2, 1),      # strided 3x3, unequal stride phases
    (3, 10, 12, 128, 64, 3, 3, 2, 1),    # strided 3x3, even size: the four phases in one launch
    (2, 13, 13, 128, 256, 1, 1, 2, 0),   # strided 1x1
    (3, 10, 10, 192, 320, 3, 3, 1, 1),   # partial N tile
    (2, 31, 29, 3, 64, 7, 7, 2, 3),      # stem, odd H and W
    (16, 1, 1, 2048, 1000, 1, 1, 1, 0),  # classifier
]


def ids(s):
    return "N{}_{}x{}_C{}_K{}_{}x{}_s{}p{}".format(*s)


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_conv_passes_write_only_their_outputs(shape):
    N, H, W, C, K, R, S, st, pd = shape
    d = pf16.conv_desc(*shape)
    P, Q = d.out_hw()
    x = dev(syn.normal_f16(syn.seed_for(1, "x"), (N, H, W, C)))
    w = dev(syn.he_normal_f16(syn.seed_for(1, "w"), K, R, S, C))
    dy = dev(syn.normal_f16(syn.seed_for(1, "dy"), (N, P, Q, K), 0.01))
    ny, ndx, ndw = N * P * Q * K, N * H * W * C, K * R * S * C

    ybuf, y = guarded(ny)
    wsb = pf16.conv_workspace_size(d, pf16.PF16_PASS_FWD)
    wbuf, ws = guarded_ws(wsb)
    pf16.conv_fwd(d, x, w, y, ws)
    assert pf16.sync_status() == 0
    assert intact(ybuf, ny) and intact_ws(wbuf, wsb), "fwd"

    if C != 3:
        dxbuf, dx = guarded(ndx)
        wsb = pf16.conv_workspace_size(d, pf16.PF16_PASS_DGRAD)
        wbuf, ws = guarded_ws(wsb)
        pf16.conv_dgrad(d, dy, w, dx, ws)
        assert pf16.sync_status() == 0
        assert intact(dxbuf, ndx) and intact_ws(wbuf, wsb), "dgrad"

    dwbuf, dw = guarded(ndw)
    wsb = pf16.conv_workspace_size(d, pf16.PF16_PASS_WGRAD)
    wbuf, ws = guarded_ws(wsb)
    pf16.conv_wgrad(d, x, dy, dw, ws)
    assert pf16.sync_status() == 0
    assert intact(dwbuf, ndw) and intact_ws(wbuf, wsb), "wgrad"


@pytest.mark.parametrize("n", [1, 7, 9, 4099])
def test_sgd_writes_only_its_parameters(n):
    wbuf, w = guarded(n)
    vbuf, v = guarded(n)
    w.copy_(dev(syn.normal_f16(3, (n,), 0.05)))
    v.copy_(dev(syn.normal_f16(4, (n,), 0.01)))
    g = dev(syn.normal_f16(5, (n,), 0.05))
    pf16.sgd_update(w, v, g, 0x2E66, 0x3B33, 0x068E)
    assert pf16.sync_status() == 0
    assert intact(wbuf, n) and intact(vbuf, n)


@pytest.mark.parametrize("shape", [(1, 9, 10, 16), (3, 7, 7, 8)])
def test_maxpool_writes_only_its_outputs(shape):
    N, H, W, C = shape
    P, Q = (H + 2 - 3) // 2 + 1, (W + 2 - 3) // 2 + 1
    x = dev(syn.normal_f16(6, (N, H, W, C)))
    ybuf, y = guarded(N * P * Q * C)
    pf16.maxpool_fwd(x, y, N, H, W, C)
    assert pf16.sync_status() == 0
    assert intact(ybuf, N * P * Q * C)
    dxbuf, dx = guarded(N * H * W * C)
    pf16.maxpool_bwd(x, dev(syn.normal_f16(7, (N, P, Q, C))), dx, N, H, W, C)
    assert pf16.sync_status() == 0
    assert intact(dxbuf, N * H * W * C)
