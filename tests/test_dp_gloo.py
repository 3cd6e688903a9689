"""The data-parallel gradient exchange (paper_1911_07384_gb300/dp.py; Sec.
5.1's data-parallel training, averaged in FP16 as Sec. 5.2 requires) run as
2 and 4 gloo ranks on the CPU: all_to_all of the rank-owned chunks, the
fixed-order combine, all_gather.  The combining step here is the oracle's
(on a GPU it is pf16_allreduce_combine, checked bit for bit against the same
oracle in tests/test_gpu_dp.py).  Every rank must end with the same bits,
equal to the oracle's average of all ranks' gradients, for a gradient length
that is not a multiple of world * 8 (padded chunks)."""
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

from paper_1911_07384_gb300 import synthetic as syn

N_GRAD = 12_345


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _grad(rank, n):
    g = syn.normal_f16(syn.seed_for(8, "dy", rank), (n,), 0.01)
    g[rank::97] = 0x8000 if rank % 2 else 0x0001  # signed zeros and the smallest subnormal
    return g


def _oracle_combine(planes, world, chunk, scale):
    import oracle

    p = planes.numpy().view(np.uint16).reshape(world, chunk)
    return torch.from_numpy(oracle.allreduce_combine(p, scale).view(np.int16))


def _rank(rank, world, port, n, out):
    import torch.distributed as dist

    from paper_1911_07384_gb300 import dp

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        g = torch.from_numpy(_grad(rank, n).view(np.int16).copy())
        dp.allreduce_mean_(g, combine=_oracle_combine)
        out[rank] = g.numpy().view(np.uint16).tobytes()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 4])
def test_exchange_is_fixed_order_and_identical_on_every_rank(orc, world):
    port = _free_port()
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.start_processes(_rank, args=(world, port, N_GRAD, out), nprocs=world, start_method="spawn", join=True)
        res = {r: np.frombuffer(out[r], np.uint16) for r in range(world)}
    for r in range(1, world):
        assert np.array_equal(res[r], res[0])
    from paper_1911_07384_gb300 import dp

    planes = np.stack([_grad(r, N_GRAD) for r in range(world)])
    ref = orc.allreduce_combine(planes, dp.inv_world_bits(world))
    assert np.array_equal(res[0], ref)


def test_chunking():
    from paper_1911_07384_gb300 import dp

    assert dp.chunk_size(12_345, 4) == 3_088 and dp.chunk_size(8, 4) == 8
    assert dp.chunk_size(25_557_032, 8) % 8 == 0 and 8 * dp.chunk_size(25_557_032, 8) >= 25_557_032
    assert dp.inv_world_bits(1) == 0x3C00 and dp.inv_world_bits(4) == 0x3400 and dp.inv_world_bits(128) == 0x2000
