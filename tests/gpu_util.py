"""Helpers for the GPU parity tests: move binary16 bit arrays between numpy
and CUDA memory, and the error bounds the tests apply."""
import numpy as np

U = 2.0 ** -11  # unit roundoff of binary16


def dev(bits):
    import torch

    a = np.ascontiguousarray(bits)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


def host(t):
    return t.detach().cpu().numpy().view(np.uint16)


def f64(bits):
    return np.asarray(bits).view(np.float16).astype(np.float64)


def empty16(*shape):
    import torch

    return torch.empty(*shape, dtype=torch.int16, device="cuda")


def zeros16(*shape):
    import torch

    return torch.zeros(*shape, dtype=torch.int16, device="cuda")


def workspace(nbytes):
    import torch

    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device="cuda") if nbytes else None


def conv_bound(A, R):
    """The contract: |err| <= 4 * sqrt(R) * 2^-11 * sum|terms|, R = reduction length."""
    return 4.0 * np.sqrt(np.asarray(R, np.float64)) * U * A


def assert_conv_close(gpu_bits, V, A, R, what, prev=None):
    g = f64(gpu_bits).ravel()
    tol = conv_bound(A, R)
    ref = V if prev is None else f64(prev).ravel() + V
    if prev is not None:  # one more FP16 rounding of the accumulate
        tol = tol + U * np.abs(ref)
    assert np.all(np.isfinite(g)), f"{what}: non-finite output"
    err = np.abs(g - ref)
    bad = err > tol
    if bad.any():
        i = int(np.argmax(err - tol))
        raise AssertionError(f"{what}: {int(bad.sum())} of {g.size} outside the bound; worst index {i}: "
                             f"gpu {g[i]!r} oracle {ref[i]!r} A {A[i]!r} tol {tol[i]!r}")
    rel = float(np.sqrt(np.sum(err ** 2) / max(np.sum(ref ** 2), 1e-300)))
    return rel
