"""GPU parity of the histogram FL search (searches whose remainder slots all lie at j <= 7: k <= 8, or
k <= 9 for signed codes) against the CPU oracle, bit-exact (Sec. IV-C, Eq. DSB_QE and Eq. MAE).

The histogram kernel takes different routes for different elements, and each is exercised here:
window keys (bins of count and sum of low bits), the per-block exponent band of the L^2 term and
the striped bins outside it, keys outside the window and subnormals (global moments), zeros and
the recount of bins that hold 65536 or more elements of one block."""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

RTOL = 1e-5


@pytest.fixture(scope="module")
def F():
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import fxpq
    return fxpq


def _check(F, x, S, klo, khi, fllo, flhi, score="l2"):
    err, best, st = F.fl_search(torch.from_numpy(x).cuda(), S, klo, khi, fllo, flhi, score=score)
    torch.cuda.synchronize()
    oerr, obest, oS, ost = oracle.fl_search(x, S, klo, khi, fllo, flhi, score=score)
    g = err.cpu().numpy()
    np.testing.assert_allclose(g, oerr, rtol=RTOL, atol=0)
    assert np.array_equal(g, oerr), np.argwhere(g != oerr)[:5]  # exact sums rounded once on both sides
    assert np.array_equal(best.cpu().numpy(), obest)
    s = F.stats_from_device(st)
    assert s.is_signed == oS and s.n == x.size and s.nonfinite == 0
    if x.size:
        assert s.min == ost["min"] and s.max == ost["max"]
        assert s.sum == ost["sum"] and s.sumsq == ost["sumsq"]


def _spread(seed, n, lo=-20, hi=10):
    """N(0,1) values scaled by 2^U{lo..hi}: exponents spread wider than one block's 16-exponent band,
    plus zeros, subnormals, halfway cases and values outside the search window."""
    rng = np.random.default_rng(seed)
    x = synth.normal(n, seed) * (np.float32(2.0) ** rng.integers(lo, hi, size=n).astype(np.float32))
    extra = np.array([0.0, -0.0, 0.5, -0.5, 1.5, 2.5, 127.5, -128.5, 255.5, 1e-40, -3e-39, 2.0 ** -30, 6.0e7,
                      -6.0e7, 0.75, 3.75, 1 - 2 ** -24, 2 ** 20 + 0.5, 1.9999999, -1.9999999, 2 ** -126,
                      2.0 ** 30, -(2.0 ** 30), 65535.5, 0.1875, 0.0625, 2.0 ** -60, 3.0e38], np.float32)
    x = np.concatenate([extra, x]).astype(np.float32)
    x[::53] = 0.0
    return x


@pytest.mark.parametrize("S", [-1, 0, 1])
@pytest.mark.parametrize("klo,khi", [(8, 8), (4, 4), (2, 8), (1, 8), (5, 7), (1, 1)])
@pytest.mark.parametrize("fllo,flhi", [(-8, 23), (0, 15), (-32, -1), (9, 40), (3, 3)])
def test_hist_grid_adversarial(F, S, klo, khi, fllo, flhi):
    x = _spread(7 * (khi + 3) + fllo + 40, 70001)
    _check(F, x, S, klo, khi, fllo, flhi)
    _check(F, np.abs(x), S, klo, khi, fllo, flhi)


@pytest.mark.parametrize("S", [-1, 1])
@pytest.mark.parametrize("klo,khi", [(9, 9), (3, 9)])
def test_hist_signed_nine_bits(F, S, klo, khi):
    """Signed codes at k = 9 still fit the histogram (slot j <= 7) when negatives force S = 1."""
    x = _spread(31 + khi, 40000)
    _check(F, x, S, klo, khi, -8, 23)


@pytest.mark.parametrize("klo,khi", [(8, 8), (1, 8), (3, 6)])
@pytest.mark.parametrize("S", [-1, 0, 1])
def test_hist_l1(F, S, klo, khi):
    x = _spread(55 + khi, 50001)
    _check(F, x, S, klo, khi, -8, 23, "l1")
    _check(F, np.abs(x), S, klo, khi, 0, 15, "l1")


@pytest.mark.parametrize("dist", ["normal", "laplace", "relu_normal"])
@pytest.mark.parametrize("n", [0, 1, 5, 1023, 16384, 32769, 300001])
def test_hist_sizes(F, dist, n):
    """Sizes around the block iteration (16384) and the chunking, including empty and one element."""
    x = synth.sweep_tensor(dist, n, 101 + n)
    _check(F, x, -1, 8, 8, -8, 23)
    _check(F, x, -1, 4, 4, -8, 23, "l1")


@pytest.mark.parametrize("value", [0.37, -1.25, 3.0, 2.0 ** -20])
def test_hist_constant_tensor_recount(F, value):
    """2^21 equal values: one bin of each block holds every element of its chunk (2^20), past the
    32-bit sum of low bits, so the block recounts that bin's sum in 64 bits."""
    x = np.full(1 << 21, value, np.float32)
    _check(F, x, -1, 8, 8, -8, 23)
    _check(F, x, 1, 2, 8, -8, 23, "l1")


def test_hist_two_values_recount(F):
    """Two values sharing a bin (equal high bits, different low bits) in every block, past the limit."""
    a = np.float32(0.7)
    b = np.frombuffer((np.frombuffer(a.tobytes(), np.uint32) ^ np.uint32(0x1234)).tobytes(), np.float32)[0]
    x = np.where(np.arange(3 << 20) % 3 == 0, a, b).astype(np.float32)
    _check(F, x, -1, 8, 8, -8, 23)


def test_hist_outside_window_only(F):
    """Every value saturates for every candidate or rounds to zero for every one: moments alone."""
    x = np.concatenate([synth.normal(5000, 3) * np.float32(2.0 ** 40), synth.normal(5000, 4) * np.float32(2.0 ** -50)])
    _check(F, x.astype(np.float32), -1, 8, 8, -8, 23)
    _check(F, x.astype(np.float32), -1, 8, 8, -8, 23, "l1")


def test_hist_unaligned(F):
    """A tensor that starts 4 bytes past a 16-byte boundary runs the scalar-load instance."""
    x = _spread(77, 100003)
    xd = torch.from_numpy(x).cuda()
    err, best, st = F.fl_search(xd[1:], -1, 8, 8, -8, 23)
    oerr, obest, _, _ = oracle.fl_search(x[1:], -1, 8, 8, -8, 23)
    assert np.array_equal(err.cpu().numpy(), oerr) and np.array_equal(best.cpu().numpy(), obest)


@pytest.mark.parametrize("dist,seed", [("normal", 2), ("laplace", 3), ("relu_normal", 4)])
@pytest.mark.parametrize("n", [1 << 24, 1 << 26])
def test_hist_full_row_large(F, dist, seed, n):
    """Full-size single-wordlength rows (k = 8, FL in [-8, 23], the calibration's search) of the
    FL-search sweep tensors at 16M and 64M values: all 32 scores, the argmin and the stats against
    the oracle, bit for bit."""
    x = synth.sweep_tensor(dist, n, seed)
    _check(F, x, -1, 8, 8, -8, 23)
