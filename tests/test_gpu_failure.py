"""Failure detection on the GPU without a fault: a bounded device-side wait
whose producer never signals runs out, records PF16_ERR_TIMEOUT in the status
word, and returns; the host reads the status, and the context and the stream
stay usable for the next call.  Nothing here traps, faults or hangs the GPU:
the only wait is bounded by the GPU's global timer."""
import time

import numpy as np
import pytest
import torch

from paper_1911_07384_gb300 import pf16
from paper_1911_07384_gb300 import synthetic as syn
from gpu_util import dev, host

pytestmark = pytest.mark.gpu


def test_wait_on_a_flag_nothing_sets_times_out_and_the_context_survives(orc):
    flag = torch.zeros(4, dtype=torch.int32, device="cuda")
    assert pf16.sync_status() == 0
    t0 = time.perf_counter()
    pf16.wait_flag(flag, 1, 20_000_000)  # 20 ms: the flag stays 0
    assert pf16.sync_status() == pf16.PF16_ERR_TIMEOUT
    assert time.perf_counter() - t0 < 5.0
    assert pf16.sync_status() == 0  # reading the status cleared it

    # the stream and the context still work: a bit-exact update right after
    n = 4099
    w = syn.normal_f16(11, (n,), 0.05)
    v = syn.normal_f16(12, (n,), 0.01)
    g = syn.normal_f16(13, (n,), 0.05)
    tw, tv = dev(w), dev(v)
    pf16.sgd_update(tw, tv, dev(g), 0x2E66, 0x3B33, 0x068E)
    assert pf16.sync_status() == 0
    ew, ev = orc.sgd_update(w, v, g, 0x2E66, 0x3B33, 0x068E)
    assert np.array_equal(host(tw), ew) and np.array_equal(host(tv), ev)


def test_wait_on_a_flag_already_set_returns_at_once():
    flag = torch.full((4,), 7, dtype=torch.int32, device="cuda")
    pf16.wait_flag(flag, 7, 2_000_000_000)
    assert pf16.sync_status() == 0


def test_flag_set_by_an_earlier_copy_on_the_stream_is_seen():
    """A host-to-device copy queued before the wait sets the flag: the wait
    completes and reports nothing."""
    flag = torch.zeros(4, dtype=torch.int32, device="cuda")
    src = torch.full((4,), 3, dtype=torch.int32).pin_memory()
    flag.copy_(src, non_blocking=True)
    pf16.wait_flag(flag, 3, 2_000_000_000)
    assert pf16.sync_status() == 0
