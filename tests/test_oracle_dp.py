"""Pins of the oracle's fixed-order FP16 gradient average (oracle.
allreduce_combine; the data-parallel exchange of Sec. 5.1 done in FP16 as
Sec. 5.2 requires): the reading is a pairwise tree of binary16 additions over
the ranks in rank order (+0 leaves up to a power of two), then one multiply by
rn(1/world).  Each pin is a fact fixed outside that code: the identity at one
rank, exact means where no rounding can occur, the pairwise-summation error
bound, numpy's own binary16 arithmetic, and the cases that tell the reading
apart from its alternatives (left-to-right order, scaling before summing)."""
import numpy as np
import pytest

from paper_1911_07384_gb300 import synthetic as syn

ONE = 0x3C00
U = 2.0 ** -11


def f64(b):
    return np.asarray(b).view(np.float16).astype(np.float64)


def h(x):
    return np.asarray(x, np.float64).astype(np.float16).view(np.uint16)


def inv(world):
    return int(h([1.0 / world])[0])


def test_one_rank_is_the_identity(orc):
    """world = 1, scale 1: every binary16 pattern, NaN payloads included, comes back unchanged."""
    allp = np.arange(65536, dtype=np.uint16)
    assert np.array_equal(orc.allreduce_combine(allp[None, :], ONE), allp)


@pytest.mark.parametrize("world", [2, 4, 8, 16])
def test_exact_when_nothing_rounds(orc, world):
    """Small multiples of 2^-10: every partial sum and the mean are binary16
    numbers, so the result is the exact mean."""
    rng = np.random.default_rng(world)
    ints = rng.integers(-64, 65, (world, 4096))
    planes = h(ints * 2.0 ** -10)
    got = f64(orc.allreduce_combine(planes, inv(world)))
    assert np.array_equal(got, ints.sum(0) * 2.0 ** -10 / world)


@pytest.mark.parametrize("world", [2, 3, 4, 5, 8, 16, 33, 128])
def test_pairwise_error_bound(orc, world):
    """|result - exact mean| <= (L + 1) u (sum |g_r|) |scale| + 2^-24 with
    L = ceil(log2 world) levels of additions (Higham's bound for pairwise
    summation) and one rounding of the scaling (plus the scale's own)."""
    g = syn.normal_f16(syn.seed_for(8, "dy", world), (world, 8192), 0.01)
    got = f64(orc.allreduce_combine(g, inv(world)))
    exact = f64(g).sum(0) / world
    L = int(np.ceil(np.log2(world)))
    tol = (L + 2) * U * np.abs(f64(g)).sum(0) / world + 2.0 ** -24
    assert np.all(np.abs(got - exact) <= tol)


@pytest.mark.parametrize("world", [2, 3, 4, 8])
def test_matches_numpy_binary16_arithmetic(orc, world):
    """The same tree evaluated with numpy's float16 operations (correctly
    rounded: binary32 has more than 2*11 + 2 bits) gives the same bits."""
    g = syn.normal_f16(syn.seed_for(8, "x", world), (world, 4096), 0.1).view(np.float16)
    leaves = [g[r] for r in range(world)]
    while len(leaves) & (len(leaves) - 1):
        leaves.append(np.zeros_like(g[0]))
    while len(leaves) > 1:
        leaves = [leaves[2 * k] + leaves[2 * k + 1] for k in range(len(leaves) // 2)]
    ref = leaves[0] if world == 1 else leaves[0] * np.float16(1.0 / world)
    got = orc.allreduce_combine(g.view(np.uint16), inv(world))
    assert np.array_equal(got, ref.view(np.uint16))


def test_pairwise_not_left_to_right():
    """(1, 2^-11, 2^-11, 2^-11): left to right, each 2^-11 is a tie that rounds
    back to 1; pairwise, the last two add to 2^-10 first, so the sum is 1 +
    2^-10."""
    import oracle

    p = h([[1.0], [2.0 ** -11], [2.0 ** -11], [2.0 ** -11]])
    assert f64(oracle.allreduce_combine(p, ONE))[0] == 1.0 + 2.0 ** -10


def test_sum_before_scale():
    """The sum comes first: two 2^-24 (the smallest subnormal) average to
    2^-24, where halving each first would round both to 0; and two 40,000s
    overflow to infinity, where halving first would give 40,000."""
    import oracle

    assert f64(oracle.allreduce_combine(h([[2.0 ** -24], [2.0 ** -24]]), inv(2)))[0] == 2.0 ** -24
    assert f64(oracle.allreduce_combine(h([[40000.0], [40000.0]]), inv(2)))[0] == np.inf


def test_rank_order_matters_and_pairs_commute():
    """Swapping the ranks of a pair (0 <-> 1) never changes a result (each node
    is a commutative addition); swapping ranks 1 and 2 can."""
    import oracle

    g = syn.normal_f16(syn.seed_for(8, "w", 4), (4, 20000), 1.0)
    a = oracle.allreduce_combine(g, inv(4))
    assert np.array_equal(a, oracle.allreduce_combine(g[[1, 0, 2, 3]], inv(4)))
    assert np.array_equal(a, oracle.allreduce_combine(g[[0, 1, 3, 2]], inv(4)))
    assert not np.array_equal(a, oracle.allreduce_combine(g[[0, 2, 1, 3]], inv(4)))
