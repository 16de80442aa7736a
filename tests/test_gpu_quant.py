"""GPU parity of the quantizer and the FL search against the CPU oracle (bit-exact).

Integer outputs (codes, chosen FL) must be identical; the L2 scores are the exact sums rounded
once on both sides, so they are compared for equality (the stated 1e-5 relative tolerance is
checked as well, as the contract)."""
import ctypes

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


def _adv(seed, n):
    base = synth.normal(n, seed)
    rng = np.random.default_rng(seed)
    base = base * (np.float32(2.0) ** rng.integers(-12, 8, size=n).astype(np.float32))
    extra = np.array([0.0, -0.0, 0.5, -0.5, 1.5, 2.5, 127.5, -128.5, 255.5, 1e-40, -3e-39, 2.0 ** -30, 6.0e7,
                      -6.0e7, 0.75, 3.75, 1 - 2 ** -24, 2 ** 20 + 0.5, 1.9999999, -1.9999999, 2 ** -126,
                      2.0 ** 30, -(2.0 ** 30), 65535.5, 0.1875, 0.0625], np.float32)
    return np.concatenate([extra, base]).astype(np.float32)


DT = {"I8": (0, np.int8), "U8": (1, np.uint8), "I16": (2, np.int16), "U16": (3, np.uint16), "I32": (4, np.int32)}


@pytest.mark.parametrize("n", [0, 1, 3, 4, 1000, 4097, 1 << 20])
@pytest.mark.parametrize("k,S,fl,dt", [(8, 1, 5, "I8"), (8, 0, 3, "U8"), (4, 1, -2, "I8"), (16, 1, 12, "I16"),
                                       (12, 0, 20, "U16"), (16, 1, 40, "I32"), (2, 1, -32, "I8")])
def test_quantize_parity(F, n, k, S, fl, dt):
    x = _adv(n + k, max(n, 1))[:n]
    code, npdt = DT[dt]
    xd = torch.from_numpy(x).cuda()
    out = torch.empty(max(n, 1), dtype=getattr(torch, np.dtype(npdt).name), device="cuda")
    F.fxpq_quantize(xd, F.fmt(k, S, fl), code, out)
    torch.cuda.synchronize()
    want = oracle.quantize(x, k, S, fl)
    assert np.array_equal(out.cpu().numpy()[:n].astype(np.int64), want)


@pytest.mark.parametrize("n", [0, 5, 4097, 1 << 20])
@pytest.mark.parametrize("k,S,fl", [(8, 1, 5), (6, 0, 2), (12, 1, 9), (16, 0, 14)])
@pytest.mark.parametrize("offset", [0, 1])
def test_quantize_f16_flat(F, n, k, S, fl, offset):
    """fxpq_quantize to an fp16 code tensor (plane-major when k > 8), 16-byte aligned (vector path) and
    4-byte aligned (scalar path)."""
    x = _adv(n + k + 100, max(n + offset, 1))
    xd = torch.from_numpy(x).cuda()[offset:offset + n]
    f = F.fmt(k, S, fl)
    out = torch.empty(max(n, 1) * F.planes(f), dtype=torch.float16, device="cuda")
    F.fxpq_quantize(xd, f, F.DT_F16, out)
    torch.cuda.synchronize()
    want = oracle.quantize(x[offset:offset + n], k, S, fl)
    got = F.codes_to_int(out[: n * F.planes(f)].cpu(), f, (n,)).numpy()
    assert np.array_equal(got, want)


def test_quantize_unaligned_and_nonfinite(F):
    x = _adv(5, 999)
    xd = torch.from_numpy(x).cuda()
    out = torch.empty(x.size - 1, dtype=torch.int8, device="cuda")
    F.fxpq_quantize(xd[1:], F.fmt(8, 1, 6), F.DT_I8, out)  # 4-byte aligned only: scalar path
    assert np.array_equal(out.cpu().numpy().astype(np.int64), oracle.quantize(x[1:], 8, 1, 6))
    assert F.fxpq_get_device_status() == 0
    bad = torch.tensor([1.0, float("nan"), float("inf"), 2.0], device="cuda")
    o2 = torch.empty(4, dtype=torch.int8, device="cuda")
    F.fxpq_quantize(bad, F.fmt(8, 1, 0), F.DT_I8, o2)
    assert F.fxpq_get_device_status() == 3  # FXPQ_ERR_NONFINITE latched
    assert F.fxpq_get_device_status() == 0  # and cleared
    assert o2.cpu().tolist() == [1, 0, 0, 2]


@pytest.mark.parametrize("k", [4, 8, 12, 16])
@pytest.mark.parametrize("C,Cp", [(3, 8), (27, 32), (64, 64)])
def test_quantize_rows_and_images(F, k, C, Cp):
    rows = 37
    x = synth.normal(rows * C, 7 + k)
    out = torch.empty(rows * Cp * (2 if k > 8 else 1), dtype=torch.float16, device="cuda")
    F.fxpq_quantize_rows(torch.from_numpy(x).cuda(), rows, C, F.fmt(k, 1, k - 3), Cp, out)
    got = F.codes_to_int(out.cpu(), F.fmt(k, 1, k - 3), (rows, Cp)).numpy()
    want = oracle.quantize(x, k, 1, k - 3).reshape(rows, C)
    assert np.array_equal(got[:, :C], want) and np.all(got[:, C:] == 0)
    imgs = synth.images(2, 9, hw=13)
    out = torch.empty(2 * 13 * 13 * 8 * (2 if k > 8 else 1), dtype=torch.float16, device="cuda")
    F.fxpq_quantize_images(torch.from_numpy(imgs).cuda(), F.fmt(k, 1, k - 4), 8, out)
    got = F.codes_to_int(out.cpu(), F.fmt(k, 1, k - 4), (2, 13, 13, 8)).numpy()
    want = oracle.quantize(np.transpose(imgs, (0, 2, 3, 1)), k, 1, k - 4).reshape(2, 13, 13, 3)
    assert np.array_equal(got[..., :3], want) and np.all(got[..., 3:] == 0)


def _check_search(F, x, S, klo, khi, fllo, flhi, score="l2"):
    err, best, st = F.fl_search(torch.from_numpy(x).cuda(), S, klo, khi, fllo, flhi, score=score)
    torch.cuda.synchronize()
    oerr, obest, oS, ost = oracle.fl_search(x, S, klo, khi, fllo, flhi, score=score)
    g = err.cpu().numpy()
    assert np.array_equal(best.cpu().numpy(), obest)
    np.testing.assert_allclose(g, oerr, rtol=RTOL, atol=0)
    assert np.array_equal(g, oerr)  # exact sums rounded once on both sides
    s = F.stats_from_device(st)
    assert s.is_signed == oS and s.n == x.size and s.nonfinite == 0
    if x.size:
        assert s.min == ost["min"] and s.max == ost["max"]
        assert s.sum == ost["sum"] and s.sumsq == ost["sumsq"]


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_fl_search_adversarial_full_grid(F, seed):
    x = _adv(seed, 3000)
    _check_search(F, x, -1, 2, 16, -8, 23)
    _check_search(F, np.abs(x), -1, 2, 16, -8, 23)
    _check_search(F, x, 0, 2, 16, -8, 23)


@pytest.mark.parametrize("dist", ["normal", "laplace", "relu_normal"])
@pytest.mark.parametrize("n", [0, 1, 5, 1023, 70001])
def test_fl_search_small_sizes_and_ranges(F, dist, n):
    x = synth.sweep_tensor(dist, n, 11 + n)
    _check_search(F, x, -1, 2, 16, -8, 23)
    _check_search(F, x, 1, 8, 8, 0, 15)
    _check_search(F, x, -1, 3, 9, -32, -1)
    _check_search(F, x, -1, 13, 16, 9, 40)


@pytest.mark.parametrize("score", ["l2", "l1"])
@pytest.mark.parametrize("seed", [4, 5])
def test_fl_search_scores_with_one_bit_rows(F, score, seed):
    """Both scores over k = 1..16 (k = 1: the binary quantizer for S = 1, the levels {0, 1} for S = 0),
    exact zeros included, bit-identical to the oracle."""
    x = _adv(seed, 3000)
    x[::97] = 0.0
    x[5] = -0.0
    _check_search(F, x, -1, 1, 16, -8, 23, score)
    _check_search(F, np.abs(x), -1, 1, 16, -8, 23, score)
    _check_search(F, x, 0, 1, 16, -8, 23, score)
    _check_search(F, x, 1, 1, 1, -8, 23, score)


@pytest.mark.parametrize("dist", ["normal", "laplace", "relu_normal"])
@pytest.mark.parametrize("n", [0, 1, 1023, 70001])
def test_fl_search_l1_sizes_and_ranges(F, dist, n):
    x = synth.sweep_tensor(dist, n, 17 + n)
    _check_search(F, x, -1, 1, 16, -8, 23, "l1")
    _check_search(F, x, 1, 8, 8, 0, 15, "l1")
    _check_search(F, x, -1, 13, 16, 9, 40, "l1")


def test_quantize_binary(F):
    """The binary quantizer: -1 for x < 0, 0 otherwise (-0.0 included), to int8 and to an fp16 code tensor."""
    x = _adv(9, 5000)
    x[:3] = [-0.0, 0.0, -1e-45]
    xd = torch.from_numpy(x).cuda()
    want = oracle.quantize(x, 1, 1, 3)
    o8 = torch.empty(x.size, dtype=torch.int8, device="cuda")
    F.fxpq_quantize(xd, F.fmt(1, 1, 3), F.DT_I8, o8)
    assert np.array_equal(o8.cpu().numpy().astype(np.int64), want)
    o16 = torch.empty(x.size, dtype=torch.float16, device="cuda")
    F.fxpq_quantize(xd, F.fmt(1, 1, 3), F.DT_F16, o16)
    assert np.array_equal(o16.cpu().numpy().astype(np.int64), want)
    words = torch.empty(F.packed_words(x.size, F.fmt(1, 1, 3)), dtype=torch.int32, device="cuda")
    F.fxpq_pack_codes(o16, x.size, F.fmt(1, 1, 3), words)
    assert np.array_equal(words.cpu().numpy().view(np.uint32), oracle.pack_codes(want, 1))


def test_fl_search_ties_pick_smallest_fl(F):
    x = np.array([0.75], np.float32)
    err, best, _ = F.fl_search(torch.from_numpy(x).cuda(), 0, 2, 2, 0, 1)
    assert err.cpu().tolist() == [[0.0625, 0.0625]] and best.item() == 0
    grid = (np.arange(-128, 128) / 32.0).astype(np.float32)  # exact on FL >= 5 at 8 bits
    err, best, _ = F.fl_search(torch.from_numpy(grid).cuda(), 1, 8, 8, 0, 10)
    assert best.item() == 5 and err.cpu().numpy()[0, 5] == 0.0


def test_fl_search_nonfinite_latches_status(F):
    x = torch.tensor([1.0, float("inf"), -2.0], device="cuda")
    err, best, st = F.fl_search(x, -1, 8, 8, 0, 3)
    assert F.fxpq_get_device_status() == 3
    assert F.stats_from_device(st).nonfinite == 1


@pytest.mark.parametrize("dist,seed", [("normal", 2), ("laplace", 3), ("relu_normal", 4)])
def test_fl_search_config_1m_full_sweep(F, dist, seed):
    x = synth.sweep_tensor(dist, 1 << 20, seed)
    _check_search(F, x, -1, 2, 16, -8, 23)


@pytest.mark.parametrize("n", [1 << 24, 1 << 26])
def test_fl_search_config_large_sampled(F, n):
    """Full-size sweep: sampled cells recomputed by the oracle one by one; argmin checked against
    the GPU's own scores; stats exact."""
    x = synth.sweep_tensor("normal", n, 2)
    err, best, st = F.fl_search(torch.from_numpy(x).cuda(), -1, 2, 16, -8, 23)
    g = err.cpu().numpy()
    b = best.cpu().numpy()
    s = F.stats_from_device(st)
    assert s.is_signed == 1
    for ki, k in enumerate(range(2, 17)):
        assert b[ki] == -8 + int(np.argmin(g[ki]))
    rng = np.random.default_rng(n)
    cells = [(8, int(b[6])), (2, int(b[0])), (16, int(b[14])), (5, 11)] + [(int(rng.integers(2, 17)), int(rng.integers(-8, 24)))]
    for k, fl in cells:
        assert g[k - 2, fl + 8] == oracle.l2_error(x, k, 1, fl)
    assert s.sumsq == oracle.exact_sum(x.astype(np.float64) ** 2)
    assert s.min == float(x.min()) and s.max == float(x.max())


def test_fl_search_l1_large_sampled(F):
    """16M Laplace values, k = 1..16 with the L1 score: sampled cells (the k = 1 binary row included)
    recomputed by the oracle one by one, argmin against the GPU's own scores."""
    n = 1 << 24
    x = synth.sweep_tensor("laplace", n, 3)
    err, best, st = F.fl_search(torch.from_numpy(x).cuda(), -1, 1, 16, -8, 23, score="l1")
    g = err.cpu().numpy()
    b = best.cpu().numpy()
    for ki in range(16):
        assert b[ki] == -8 + int(np.argmin(g[ki]))
    for k, fl in [(1, int(b[0])), (1, -8), (8, int(b[7])), (3, 2), (16, 23)]:
        assert g[k - 1, fl + 8] == oracle.l1_error(x, k, 1, fl)


def test_fl_search_batch_matches_oracle(F):
    """A batch mixing sizes (0 to 300k), wordlength ranges (one k, several k, the full sweep), fixed
    and automatic signedness and an unaligned tensor: every item equals the oracle's search, and
    more than 32 items run as several groups."""
    import paper_2203_12091_gb300._lib as L
    specs = []
    for i in range(37):
        dist = ("normal", "laplace", "relu_normal")[i % 3]
        n = (0, 1, 17, 1023, 4097, 70001, 300000)[i % 7]
        klo, khi = ((8, 8), (4, 4), (16, 16), (2, 16), (3, 9), (12, 13))[i % 6]
        S = (-1, 0, 1)[i % 3] if i % 5 else -1
        fllo, flhi = ((-8, 23), (0, 15), (-32, -1))[i % 3]
        specs.append((synth.sweep_tensor(dist, n, 100 + i), S, klo, khi, fllo, flhi, i % 4 == 3))
    items, keep = [], []
    for x, S, klo, khi, fllo, flhi, unaligned in specs:
        xd = torch.from_numpy(np.concatenate([np.zeros(1, np.float32), x])).cuda()
        xd = xd[1:] if unaligned else xd[1:].clone()
        nk, nfl = khi - klo + 1, flhi - fllo + 1
        err = torch.empty(nk * nfl, dtype=torch.float64, device="cuda")
        best = torch.empty(nk, dtype=torch.int32, device="cuda")
        st = torch.empty(ctypes.sizeof(L.Stats), dtype=torch.uint8, device="cuda")
        keep.append((xd, err, best, st))
        items.append(L.FlSearchItem(xd.data_ptr(), x.size, S, klo, khi, fllo, flhi, err.data_ptr(), best.data_ptr(),
                                    st.data_ptr()))
    ws = torch.empty(F.fxpq_fl_search_batch_workspace(len(items)), dtype=torch.uint8, device="cuda")
    F.fxpq_fl_search_batch(items, ws)
    torch.cuda.synchronize()
    assert F.fxpq_get_device_status() == 0
    for (x, S, klo, khi, fllo, flhi, _), (xd, err, best, st) in zip(specs, keep):
        oerr, obest, oS, ost = oracle.fl_search(x, S, klo, khi, fllo, flhi)
        assert np.array_equal(best.cpu().numpy(), obest)
        assert np.array_equal(err.cpu().numpy(), oerr.reshape(-1))
        s = F.stats_from_device(st)
        assert s.is_signed == oS and s.n == x.size
        if x.size:
            assert s.min == ost["min"] and s.max == ost["max"] and s.sum == ost["sum"] and s.sumsq == ost["sumsq"]


def test_quantize_batch_device_formats(F):
    """fxpq_quantize_batch reads S and FL from device memory: rows items (one and two planes, padded
    and unpadded channels, with and without the L1 bound) and flat int32 items equal the oracle's
    quantizer; the L1 bound equals the largest per-output-channel sum of |code|."""
    import paper_2203_12091_gb300._lib as L
    rng = np.random.default_rng(5)
    cases = [  # kind, k, S, fl, K, RS, C, Cp, want_l1
        ("rows", 8, 1, 9, 64, 9, 64, 64, True),
        ("rows", 5, 1, 6, 32, 9, 3, 8, True),
        ("rows", 16, 1, 14, 16, 9, 8, 8, False),
        ("rows", 12, 0, 7, 8, 1, 40, 40, False),
        ("flat", 16, 1, 20, 1000, 0, 0, 0, False),
        ("flat", 7, 0, 3, 1, 0, 0, 0, False),
    ]
    fmt_buf = torch.zeros(len(cases) * 64, dtype=torch.uint8, device="cuda")
    host_fmt = bytearray(len(cases) * 64)
    items, keep = [], []
    l1 = torch.zeros(len(cases), dtype=torch.int64, device="cuda")
    for i, (kind, k, S, fl, K, RS, C, Cp, want_l1) in enumerate(cases):
        host_fmt[64 * i:64 * i + 4] = int(fl).to_bytes(4, "little", signed=True)
        st = L.Stats(0.0, 0.0, S, 0, 0.0, 0.0, 0)
        host_fmt[64 * i + 8:64 * i + 8 + ctypes.sizeof(L.Stats)] = bytes(st)
        if kind == "rows":
            x = (rng.standard_normal((K * RS, C)) * 2.0 ** (-fl + k - 3)).astype(np.float32)
            out = torch.empty(K * RS * Cp * (2 if k > 8 else 1), dtype=torch.float16, device="cuda")
        else:
            x = (rng.standard_normal(K) * 2.0 ** (-fl + k - 2)).astype(np.float32)
            out = torch.empty(K, dtype=torch.int32, device="cuda")
        xd = torch.from_numpy(x).cuda()
        keep.append((xd, out, x))
        base = fmt_buf.data_ptr() + 64 * i
        items.append(L.QuantizeItem(xd.data_ptr(), out.data_ptr(), L.QB_ROWS_F16 if kind == "rows" else L.QB_FLAT_I32,
                                    k, K * RS if kind == "rows" else K, C, Cp, max(RS, 1), 0, base, base + 8,
                                    l1.data_ptr() + 8 * i if want_l1 else None))
    fmt_buf.copy_(torch.frombuffer(host_fmt, dtype=torch.uint8))
    F.fxpq_quantize_batch(items)
    torch.cuda.synchronize()
    assert F.fxpq_get_device_status() == 0
    l1h = l1.cpu().numpy()
    for i, ((kind, k, S, fl, K, RS, C, Cp, want_l1), (xd, out, x)) in enumerate(zip(cases, keep)):
        want = np.asarray(oracle.quantize(x, k, S, fl)).reshape(x.shape)
        if kind == "rows":
            got = F.codes_to_int(out.cpu(), F.fmt(k, S, fl), (K * RS, Cp)).numpy()
            assert np.array_equal(got[:, :C], want) and np.all(got[:, C:] == 0)
            if want_l1:
                assert l1h[i] == np.abs(want).reshape(K, -1).sum(axis=1).max()
        else:
            assert np.array_equal(out.cpu().numpy(), want)


def _f16_codes(c, k):
    """fp16 code tensor of a flat code array (plane-major hi / lo limbs when k > 8)."""
    c = np.asarray(c, dtype=np.int64)
    if k <= 8:
        return torch.from_numpy(c.astype(np.float16)).cuda()
    hi = c >> 8
    return torch.from_numpy(np.concatenate([hi, c - (hi << 8)]).astype(np.float16)).cuda()


@pytest.mark.parametrize("k,S", [(2, 1), (3, 0), (4, 1), (5, 1), (8, 0), (8, 1), (11, 1), (16, 0), (16, 1)])
@pytest.mark.parametrize("n", [0, 1, 31, 33, 1000])
def test_pack_unpack_parity(F, k, S, n):
    """fxpq_pack_codes word for word against the oracle's packed layout; fxpq_unpack_codes restores the
    codes (sign-extended when S = 1)."""
    rng = np.random.default_rng(k * 100 + n + S)
    c = rng.integers(oracle.qmin(k, S), oracle.qmax(k, S) + 1, size=n)
    c[: min(2, n)] = [oracle.qmin(k, S), oracle.qmax(k, S)][: min(2, n)]
    f = F.fmt(k, S, 0)
    nw = F.packed_words(n, f)
    words = torch.full((max(nw, 1),), 0x5A5A5A5A, dtype=torch.int32, device="cuda")
    F.fxpq_pack_codes(_f16_codes(c, k) if n else torch.empty(1, dtype=torch.float16, device="cuda"), n, f, words)
    torch.cuda.synchronize()
    got = words.cpu().numpy().view(np.uint32)[:nw]
    assert np.array_equal(got, oracle.pack_codes(c, k))
    out = torch.empty(max(n, 1) * F.planes(f), dtype=torch.float16, device="cuda")
    F.fxpq_unpack_codes(words, n, f, out)
    assert np.array_equal(F.codes_to_int(out[: n * F.planes(f)].cpu(), f, (n,)).numpy(), c)


@pytest.mark.parametrize("k,S", [(4, 1), (12, 1)])
def test_pack_unpack_large_sampled(F, k, S):
    """64M + 5 codes: the round trip is exact everywhere and sampled groups match the oracle's words."""
    n = (1 << 26) + 5
    rng = np.random.default_rng(k)
    c = rng.integers(oracle.qmin(k, S), oracle.qmax(k, S) + 1, size=n)
    f = F.fmt(k, S, 0)
    words = torch.empty(F.packed_words(n, f), dtype=torch.int32, device="cuda")
    F.fxpq_pack_codes(_f16_codes(c, k), n, f, words)
    out = torch.empty(n * F.planes(f), dtype=torch.float16, device="cuda")
    F.fxpq_unpack_codes(words, n, f, out)
    assert np.array_equal(F.codes_to_int(out.cpu(), f, (n,)).numpy(), c)
    w = words.cpu().numpy().view(np.uint32)
    ng = (n + 31) // 32
    for g in list(rng.integers(0, ng, size=40)) + [ng - 1]:
        seg = c[32 * g: 32 * g + 32]
        assert np.array_equal(w[g * k:(g + 1) * k], oracle.pack_codes(seg, k)), g
