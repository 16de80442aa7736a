"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: each check uses the paper's printed examples
(tests/golden/*.txt), closed forms, invariants, or an exact brute force in Python Fractions.
"""
import itertools
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from oracle import net as onet

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    out = []
    with open(os.path.join(GOLD, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                out.append(line.split())
    return out


def F(x):
    return Fraction(float(x))


def frac_q(x, k, S, fl):
    """Quantizer as nearest member of domQ (ties to the even code), exact."""
    y = F(x) * Fraction(2) ** fl
    m = oracle.frac_round_half_even(y)
    return min(max(m, -S * 2 ** (k - S)), 2 ** (k - S) - 1)


def frac_l2(xs, k, S, fl):
    tot = Fraction(0)
    for x in xs:
        d = F(x) - Fraction(frac_q(x, k, S, fl)) * Fraction(2) ** (-fl)
        tot += d * d
    return tot


# ---------------------------------------------------------------- paper examples
def test_paper_format_examples():
    for a, b, S, x, v in _rows("paper_format_examples.txt"):
        a, b, S = int(a), int(b), int(S)
        k = a + b
        code = oracle.quantize(np.array([float(x)], np.float32), k, S, b)[0]
        assert Fraction(int(code)) * Fraction(2) ** (-b) == F(np.float32(float(v))), (a, b, x)


def test_paper_format_value_sets():
    # U(3,-1): values {0,2,4,6}; S(-1,3): {-0.25,-0.125,0,0.125}
    grid = np.linspace(-20, 20, 4001).astype(np.float32)
    u = set((oracle.quantize(grid, 2, 0, -1) * 2.0).tolist())
    s = set((oracle.quantize(grid / 40, 2, 1, 3) / 8.0).tolist())
    assert u == {0.0, 2.0, 4.0, 6.0}
    assert s == {-0.25, -0.125, 0.0, 0.125}


def test_paper_format_levels():
    for a, b, S, k, lo, hi in _rows("paper_formats.txt"):
        a, b, S, k, lo, hi = map(int, (a, b, S, k, lo, hi))
        assert a + b == k
        assert oracle.qmin(k, S) == lo and oracle.qmax(k, S) == hi
        x = np.array([1e6, -1e6], np.float32)
        c = oracle.quantize(x, k, S, b)
        assert c[0] == hi and c[1] == lo
    # 6-bit signed range [-32*2^-beta, 31*2^-beta]
    for beta in (5, 7, 8, 9):
        c = oracle.quantize(np.array([1e3, -1e3], np.float32), 6, 1, beta)
        assert c[0] * 2.0 ** -beta == 31 * 2.0 ** -beta and c[1] * 2.0 ** -beta == -32 * 2.0 ** -beta


def test_round_half_even_ties():
    x = np.array([0.5, 1.5, 2.5, -1.5, -0.5, 3.5, -2.5], np.float32)
    assert oracle.quantize(x, 8, 1, 0).tolist() == [0, 2, 2, -2, 0, 4, -2]


# ---------------------------------------------------------------- quantizer
def _adversarial(seed, n=64):
    rng = np.random.default_rng(seed)
    base = synth.normal(n, seed)
    extra = np.array([0.0, -0.0, 0.5, -0.5, 1.5, 2.5, 127.5, -128.5, 255.5, 1e-40, -3e-39,
                      2.0 ** -30, 6.0e7, -6.0e7, 0.75, 3.75, 1 - 2 ** -24, 2 ** 20 + 0.5], np.float32)
    scale = np.float32(2.0) ** rng.integers(-6, 6, size=n).astype(np.float32)
    return np.concatenate([base * scale, extra]).astype(np.float32)


def test_quantize_matches_nearest_in_domQ():
    xs = _adversarial(11)
    for k, S, fl in itertools.product([2, 3, 5, 8, 9, 16], [0, 1], [-8, -1, 0, 3, 7, 23]):
        got = oracle.quantize(xs, k, S, fl)
        want = [frac_q(x, k, S, fl) for x in xs]
        assert got.tolist() == want, (k, S, fl)


def test_quantize_invariants():
    xs = np.sort(_adversarial(12, 2000))
    for k, S, fl in [(8, 1, 5), (4, 0, 2), (16, 1, 12), (3, 1, -2)]:
        c = oracle.quantize(xs, k, S, fl)
        v = c.astype(np.float64) * 2.0 ** -fl
        lo, hi = oracle.qmin(k, S), oracle.qmax(k, S)
        inside = (xs.astype(np.float64) >= lo * 2.0 ** -fl) & (xs.astype(np.float64) <= hi * 2.0 ** -fl)
        # |x - x~| <= 2^-(FL+1) inside the range
        assert np.all(np.abs(xs[inside].astype(np.float64) - v[inside]) <= 2.0 ** -(fl + 1))
        # exact saturation
        assert np.all(c[xs.astype(np.float64) > hi * 2.0 ** -fl] == hi)
        assert np.all(c[xs.astype(np.float64) < lo * 2.0 ** -fl] == lo)
        # monotone
        assert np.all(np.diff(c) >= 0)
        # idempotent on representable values
        assert np.array_equal(oracle.quantize(v.astype(np.float32), k, S, fl), c)
        # sign symmetry away from Qmin
        if S == 1:
            cn = oracle.quantize(-xs, k, S, fl)
            ok = (c > lo) & (cn > lo)
            assert np.array_equal(cn[ok], -c[ok])


# ---------------------------------------------------------------- L2 error (Eq. DSB_QE)
def test_exact_sum_accumulator_vs_fractions():
    rng = np.random.default_rng(3)
    for trial in range(20):
        n = int(rng.integers(1, 200))
        v = rng.standard_normal(n) * 2.0 ** rng.integers(-300, 300, size=n)
        if trial % 3 == 0:  # heavy cancellation
            v = np.concatenate([v, -v[: n // 2], [1e-300, -1e300, 1e300]])
        want = float(sum((Fraction(float(t)) for t in v), Fraction(0)))
        assert oracle.exact_sum(v) == want


def test_l2_single_element_closed_form():
    for x in [0.3, -0.7, 5.25, 1e-3, -100.0, 0.0]:
        for k, S, fl in [(8, 1, 4), (2, 0, 1), (16, 1, 20), (5, 0, -3)]:
            want = float(frac_l2([np.float32(x)], k, S, fl))
            assert oracle.l2_error(np.array([x], np.float32), k, S, fl) == want


def test_l2_zero_on_grid():
    codes = np.arange(-128, 128)
    for fl in [-3, 0, 5, 20]:
        x = (codes * 2.0 ** -fl).astype(np.float32)
        assert oracle.l2_error(x, 8, 1, fl) == 0.0
        assert oracle.l2_error(x, 9, 1, fl) == 0.0
        assert oracle.l2_error(x, 7, 1, fl) > 0.0  # does not fit 7 bits


def test_l2_bruteforce_all_candidates():
    for seed in (21, 22):
        xs = _adversarial(seed, 10)[:16]
        err, best, S, st = oracle.fl_search(xs, -1, 2, 16, -8, 23)
        assert S == 1
        for ki, k in enumerate(range(2, 17)):
            exact = [frac_l2(xs, k, S, fl) for fl in range(-8, 24)]
            assert err[ki].tolist() == [float(e) for e in exact]
            m = min(exact)
            assert best[ki] == -8 + exact.index(m)  # first minimum: ties go to the smallest FL


def test_fl_search_tie_goes_to_smallest_fl():
    # single x = 0.75, k = 2 unsigned: FL=0 -> code 1 (err 1/16); FL=1 -> code 2 (value 1, err 1/16)
    x = np.array([0.75], np.float32)
    err, best, S, _ = oracle.fl_search(x, 0, 2, 2, 0, 1)
    assert err[0, 0] == err[0, 1] == 0.0625 and best[0] == 0
    err, best, S, _ = oracle.fl_search(x, 0, 2, 2, -2, 3)
    assert best[0] == 2 and err[0, 4] == 0.0


def test_unsigned_equals_signed_one_more_bit_on_nonnegative():
    xs = np.abs(_adversarial(31, 300))
    for k in (2, 5, 8, 15):
        for fl in (-4, 0, 6, 19):
            assert np.array_equal(oracle.quantize(xs, k, 0, fl), oracle.quantize(xs, k + 1, 1, fl))
            assert oracle.l2_error(xs, k, 0, fl) == oracle.l2_error(xs, k + 1, 1, fl)


def test_unsigned_negative_inputs_saturate_to_zero():
    xs = -np.abs(_adversarial(32, 100))
    assert np.all(oracle.quantize(xs, 6, 0, 3) == 0)
    assert oracle.l2_error(xs, 6, 0, 3) == float(sum(F(x) ** 2 for x in xs))


def test_stats_and_sign_strategy():
    xs = _adversarial(41, 500)
    _, _, S, st = oracle.fl_search(xs, -1, 8, 8, 0, 1)
    assert S == 1 and st["min"] == float(xs.min()) and st["max"] == float(xs.max())
    assert st["sum"] == float(sum(F(x) for x in xs))
    assert st["sumsq"] == float(sum(F(x) ** 2 for x in xs))
    _, _, S, _ = oracle.fl_search(np.abs(xs), -1, 8, 8, 0, 1)
    assert S == 0


def test_fl_init_hand_cases():
    # unsigned: psi = max/(2^k-1) = 1/255 -> beta_hat = log2(255) = 7.994
    assert oracle.fl_init(0.0, 1.0, 8, "conservative") == (0, 7, 1)
    assert oracle.fl_init(0.0, 1.0, 8, "neutral") == (0, 8, 0)
    assert oracle.fl_init(0.0, 1.0, 8, "aggressive") == (0, 8, 0)
    # signed: psi = min(2/128, 1/127) = 1/127 -> beta_hat = log2(127) = 6.989
    assert oracle.fl_init(-2.0, 1.0, 8, "conservative") == (1, 6, 2)
    assert oracle.fl_init(-2.0, 1.0, 8, "neutral") == (1, 7, 1)
    # exact power of two: psi = min(0.5/128, 0.5/127) = 2^-8 -> beta = 8 for every strategy
    for st in ("conservative", "neutral", "aggressive"):
        assert oracle.fl_init(-0.5, 0.5, 8, st)[1] == 8


# ---------------------------------------------------------------- integer C-Block
def _im2col_conv(x, w, stride, pad):
    N, H, W, C = x.shape
    K, R, S, _ = w.shape
    xp = np.zeros((N, H + 2 * pad, W + 2 * pad, C), np.int64)
    xp[:, pad:pad + H, pad:pad + W] = x
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    cols = np.empty((N, P, Q, R, S, C), np.int64)
    for r in range(R):
        for s in range(S):
            cols[:, :, :, r, s, :] = xp[:, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride, :]
    return np.matmul(cols.reshape(N * P * Q, -1), w.reshape(K, -1).astype(np.int64).T).reshape(N, P, Q, K)


@pytest.mark.parametrize("shape", [(2, 9, 9, 5, 7, 3, 1, 1), (1, 23, 23, 3, 4, 11, 4, 2), (2, 8, 8, 16, 6, 1, 2, 0),
                                   (3, 6, 6, 4, 5, 6, 1, 0), (1, 7, 7, 3, 2, 7, 2, 3)])
def test_conv_matches_im2col_matmul(shape):
    N, H, W, C, K, R, st, pad = shape
    rng = np.random.default_rng(sum(shape))
    x = rng.integers(0, 256, size=(N, H, W, C))
    w = rng.integers(-128, 128, size=(K, R, R, C))
    assert np.array_equal(oracle.conv2d(x, w, st, pad), _im2col_conv(x, w, st, pad))


def test_conv_one_hot_weights_select_inputs():
    rng = np.random.default_rng(5)
    x = rng.integers(-32768, 32768, size=(2, 5, 5, 4))
    w = np.zeros((4, 3, 3, 4), np.int64)
    for k in range(4):
        w[k, 1, 1, k] = 1
    assert np.array_equal(oracle.conv2d(x, w, 1, 1), x)


def test_requant_matches_quantizing_the_exact_value():
    rng = np.random.default_rng(7)
    acc = rng.integers(-2 ** 40, 2 ** 40, size=400)
    acc[:8] = [0, 1, -1, 2 ** 10 + 2 ** 9, -(2 ** 10 + 2 ** 9), 3 * 2 ** 9, 5 * 2 ** 9, -7 * 2 ** 9]
    for s, fl, k, S in [(20, 10, 8, 1), (20, 8, 16, 1), (13, 3, 6, 0), (5, 9, 8, 1), (30, 30, 12, 1), (10, 0, 4, 0)]:
        got = oracle.requant(acc, s, k, S, fl)
        for a, g in zip(acc.tolist(), got.tolist()):
            y = Fraction(a) * Fraction(2) ** (fl - s)
            m = oracle.frac_round_half_even(y)
            assert g == min(max(m, -S * 2 ** (k - S)), 2 ** (k - S) - 1)


def test_bias_alignment_preserves_value():
    rng = np.random.default_rng(8)
    acc = rng.integers(-2 ** 30, 2 ** 30, size=100)
    b = rng.integers(-2 ** 15, 2 ** 15, size=100)
    for s, flb in [(12, 4), (12, 12), (5, 19), (0, 3)]:
        v, s2 = oracle.add_bias(acc, s, b, flb)
        for a, bb, vv in zip(acc.tolist(), b.tolist(), v.tolist()):
            assert Fraction(vv, 2 ** s2) == Fraction(a, 2 ** s) + Fraction(bb, 2 ** flb)


def test_scale_layer_cblock_equals_exact_bn_value():
    """CONV-Scale-ReLU (Sec. IV-B): the integer C-Block value times 2^-s equals, as an exact rational,
    relu(aleph1 * (acc 2^-s_acc + B 2^-FL_b) + aleph2) for every alignment case of both additions."""
    rng = np.random.default_rng(18)
    K = 7
    acc = rng.integers(-2 ** 28, 2 ** 28, size=(9, K))
    b = rng.integers(-2 ** 15, 2 ** 15, size=K)
    sc = rng.integers(-2 ** 15, 2 ** 15, size=K)
    sh = rng.integers(-2 ** 15, 2 ** 15, size=K)
    for s_acc, flb, fls, flh, relu in [(12, 4, 14, 20, True), (12, 18, 9, 3, False), (5, 5, 15, 30, True),
                                       (10, 2, 0, 22, False)]:
        v, s = oracle.cblock(acc, s_acc, b, flb, relu, scale=sc, fl_scale=fls, shift=sh, fl_shift=flh)
        for i in range(acc.shape[0]):
            for k in range(K):
                x = Fraction(int(acc[i, k]), 2 ** s_acc) + Fraction(int(b[k]), 2 ** flb)
                y = Fraction(int(sc[k]), 2 ** fls) * x + Fraction(int(sh[k]), 2 ** flh)
                if relu:
                    y = max(y, Fraction(0))
                assert Fraction(int(v[i, k]), 2 ** s) == y
        # and the FxP-QLayer of it equals Q of the exact value
        q = oracle.requant(v, s, 8, 1, 3)
        for i in range(acc.shape[0]):
            for k in range(K):
                yv = Fraction(int(v[i, k]), 2 ** s) * 8
                fl, cl = yv.numerator // yv.denominator, yv - yv.numerator // yv.denominator
                r = fl + (1 if cl > Fraction(1, 2) or (cl == Fraction(1, 2) and fl % 2) else 0)
                assert q[i, k] == min(max(r, -128), 127)


def test_bn_to_scale_matches_the_formula():
    """Eq. BatchNorm_s1_s2: aleph1 = gamma / sqrt(var + eps), aleph2 = beta - gamma mean / sqrt(var + eps),
    within fp32 rounding of the float64 formula, and BN(a) = aleph1 a + aleph2."""
    rng = np.random.default_rng(19)
    g = rng.uniform(0.5, 2.0, 64).astype(np.float32)
    be = rng.normal(0, 0.5, 64).astype(np.float32)
    mu = rng.normal(0, 1, 64).astype(np.float32)
    var = rng.uniform(0.1, 4.0, 64).astype(np.float32)
    a1, a2 = oracle.bn_to_scale(g, be, mu, var)
    r64 = np.sqrt(var.astype(np.float64) + 1e-5)
    np.testing.assert_allclose(a1, g / r64, rtol=4e-7)
    np.testing.assert_allclose(a2, be - g * mu.astype(np.float64) / r64, rtol=1e-5, atol=1e-6)
    x = rng.normal(0, 1, 64)
    bn = g * (x - mu) / r64 + be
    np.testing.assert_allclose(a1 * x + a2, bn, rtol=1e-5, atol=1e-5)


def test_maxpool_matches_window_max():
    rng = np.random.default_rng(9)
    x = rng.integers(0, 256, size=(2, 13, 11, 5))
    for k, st, pad in [(3, 2, 0), (2, 2, 0), (3, 2, 1), (3, 1, 1)]:
        got = oracle.maxpool(x, k, st, pad)
        xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)), constant_values=-1)
        win = np.lib.stride_tricks.sliding_window_view(xp, (k, k), axis=(1, 2))[:, ::st, ::st]
        want = win.max(axis=(-1, -2))
        assert np.array_equal(got, want[:, :got.shape[1], :got.shape[2]])
        # unsigned post-ReLU codes: ignoring padded taps equals zero padding
        xz = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)), constant_values=0)
        winz = np.lib.stride_tricks.sliding_window_view(xz, (k, k), axis=(1, 2))[:, ::st, ::st]
        assert np.array_equal(got, winz.max(axis=(-1, -2))[:, :got.shape[1], :got.shape[2]])


def test_eltwise_and_avgpool_exact():
    rng = np.random.default_rng(10)
    a = rng.integers(-128, 128, size=(2, 3, 3, 4))
    b = rng.integers(0, 64, size=(2, 3, 3, 4))
    v, fl = oracle.eltwise_add(a, 3, b, 6, relu=True)
    for x, y, z in zip(a.ravel().tolist(), b.ravel().tolist(), v.ravel().tolist()):
        assert Fraction(z, 2 ** fl) == max(Fraction(x, 8) + Fraction(y, 64), 0)
    x = rng.integers(0, 256, size=(2, 7, 7, 3))
    r = oracle.quantize(np.array([1 / 49], np.float32), 16, 0, 21)[0]
    v, s = oracle.avgpool_global(x, 4, int(r), 21)
    for n in range(2):
        for c in range(3):
            assert Fraction(int(v[n, c]), 2 ** s) == Fraction(int(x[n, :, :, c].sum()), 16) * Fraction(int(r), 2 ** 21)


def test_reciprocal_format_of_avgpool():
    # 1/49 as a 16-bit unsigned parameter: the FL search picks FL = 21 (largest unsaturated grid)
    _, best, S, _ = oracle.fl_search(np.array([1 / 49], np.float32), -1, 16, 16, -8, 23)
    assert S == 0 and best[0] == 21


# ---------------------------------------------------------------- small network, exact semantics
def _tiny_layers():
    return [
        {"type": "conv", "name": "c1", "C": 3, "K": 6, "R": 3, "stride": 1, "pad": 1, "relu": True, "src": None},
        {"type": "maxpool", "name": "p1", "k": 2, "stride": 2, "pad": 0},
        {"type": "conv", "name": "c2", "C": 6, "K": 5, "R": 3, "stride": 1, "pad": 1, "relu": False, "src": None},
        {"type": "eltwise", "name": "e", "a": "c2", "b": "c2b", "relu": True},
        {"type": "conv", "name": "fc", "C": 5, "K": 4, "R": 4, "stride": 1, "pad": 0, "relu": False, "src": "e"},
    ]


def test_tiny_network_layers_equal_quantized_exact_reals():
    layers = _tiny_layers()
    # second branch feeding the eltwise: a 1x1 conv on p1
    layers.insert(3, {"type": "conv", "name": "c2b", "C": 6, "K": 5, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": "p1"})
    layers[2]["src"] = "p1"
    rng = np.random.default_rng(13)
    weights = {}
    for L in layers:
        if L["type"] == "conv":
            fan = L["C"] * L["R"] ** 2
            weights[L["name"]] = ((rng.standard_normal((L["K"], L["R"], L["R"], L["C"])) * np.sqrt(2 / fan)).astype(np.float32),
                                  (rng.standard_normal(L["K"]) * 0.01).astype(np.float32))
    plan = {"input": 8, "c1": {"w": 6, "b": 16, "a": 5}, "c2": {"w": 7, "b": 16, "a": 6},
            "c2b": {"w": 5, "b": 16, "a": 7}, "e": {"a": 6}, "fc": {"w": 8, "b": 16}}
    imgs = synth.images(2, 77, hw=8)
    fmts, qp = onet.calibrate(layers, weights, imgs, plan)
    env = onet.forward_trace(layers, fmts, qp, imgs)

    def val(codes, fl):
        return [Fraction(int(c)) * Fraction(2) ** (-fl) for c in np.asarray(codes).ravel()]

    def check_q(codes, fmt, exact_vals):
        k, S, fl = fmt
        want = [min(max(oracle.frac_round_half_even(v * Fraction(2) ** fl), -S * 2 ** (k - S)), 2 ** (k - S) - 1)
                for v in exact_vals]
        assert np.asarray(codes).ravel().tolist() == want

    # each conv C-Block's output codes = Q(exact real conv + bias, ReLU) under its format
    for nm, src in [("c1", "input"), ("c2", "p1"), ("c2b", "p1")]:
        L = next(l for l in layers if l["name"] == nm)
        x, fx = env[src]
        wq, bq = qp[nm]
        fw, fb = fmts[nm]["w"], fmts[nm]["b"]
        acc = oracle.conv2d(x, wq, L["stride"], L["pad"])
        exact = [Fraction(int(a), 2 ** (fx[2] + fw[2])) + Fraction(int(bq[i % L["K"]])) * Fraction(2) ** (-fb[2])
                 for i, a in enumerate(acc.ravel().tolist())]
        if L["relu"]:
            exact = [max(e, 0) for e in exact]
        check_q(env[nm][0], fmts[nm]["a"], exact)
    # eltwise: Q(relu(a + b)) of the real values
    ea = val(env["c2"][0], fmts["c2"]["a"][2])
    eb = val(env["c2b"][0], fmts["c2b"]["a"][2])
    check_q(env["e"][0], fmts["e"]["a"], [max(p + q, 0) for p, q in zip(ea, eb)])
    # maxpool keeps the input format
    assert env["p1"][1] == fmts["c1"]["a"]
    # calibration picked the argmin of the L2 error of the calibration output (checked for c1)
    L = layers[0]
    x, fx = env["input"]
    acc = oracle.conv2d(x, qp["c1"][0], 1, 1)
    v, s = oracle.cblock(acc, fx[2] + fmts["c1"]["w"][2], qp["c1"][1], fmts["c1"]["b"][2], True)
    vf = oracle.to_f32(v, s)
    k, S, fl_c = fmts["c1"]["a"]
    assert S == (1 if vf.min() < 0 else 0)  # sign strategy of Sec. IV-A.3
    errs = [frac_l2(vf.ravel(), k, S, fl) for fl in range(-8, 24)]  # exact L of every candidate FL
    assert fl_c == -8 + min(range(32), key=lambda i: (errs[i], i))  # smallest L, exact ties to the smaller FL


# ---------------------------------------------------------------- architecture size pins
def test_architecture_size_pins():
    w = {L["name"]: L for L in synth.alexnet() if L["type"] == "conv"}
    # AlexNet CONV-1 weights: 4.25 KB per bit -> 96*3*11*11 = 34848 weights
    assert w["conv1"]["K"] * w["conv1"]["C"] * w["conv1"]["R"] ** 2 == 34848
    assert round(34848 / 8 / 1024, 2) == 4.25
    # AlexNet FC-6: 4.72 MB per bit -> 9216 x 4096
    assert w["fc6"]["C"] * w["fc6"]["R"] ** 2 == 9216 and w["fc6"]["K"] == 4096
    assert round(9216 * 4096 / 8 / 1e6, 2) == 4.72
    v = {L["name"]: L for L in synth.vgg16() if L["type"] == "conv"}
    # VGG-16 FC-6: 102.76 M multiplies per image
    assert round(v["fc6"]["C"] * v["fc6"]["R"] ** 2 * v["fc6"]["K"] / 1e6, 2) == 102.76
    # per-image MACs: VGG-16 15.3-15.5 G, ResNet-18 1.8 G
    assert 15.3e9 <= synth.macs_per_image("vgg16") <= 15.5e9
    assert abs(synth.macs_per_image("resnet18") - 1.8e9) < 0.05e9
    assert sum(1 for L in synth.vgg16() if L["type"] == "conv") == 16


def _bn_net(with_bn: bool):
    layers = [
        {"type": "conv", "name": "c1", "C": 3, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": True, "src": None},
        {"type": "conv", "name": "c2", "C": 8, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": False, "src": None},
        {"type": "conv", "name": "fc", "C": 8, "K": 4, "R": 6, "stride": 1, "pad": 0, "relu": False, "src": None},
    ]
    if with_bn:
        layers[0]["bn"] = layers[1]["bn"] = True
    return layers


def test_scale_layer_with_unit_gain_is_the_folded_bias_net():
    """Special case of the BN rewrite (Sec. IV-A.1): with gamma = sqrt(var + eps) (so aleph1 = 1 exactly,
    quantized to code 1 at FL 0) and mean = 0 (aleph2 = beta), a bias-free CONV -> Scale -> ReLU network
    is the folded network CONV(+bias beta) -> ReLU, bit for bit: same formats, same codes, same logits."""
    rng = np.random.default_rng(21)
    folded, withbn = _bn_net(False), _bn_net(True)
    W, Wbn, bn = {}, {}, {}
    for L in folded:
        fan = L["C"] * L["R"] ** 2
        w = (rng.standard_normal((L["K"], L["R"], L["R"], L["C"])) * np.sqrt(2 / fan)).astype(np.float32)
        b = (rng.standard_normal(L["K"]) * 0.05).astype(np.float32)
        W[L["name"]] = (w, b)
        if L["name"] == "fc":
            Wbn["fc"] = (w, b)
            continue
        Wbn[L["name"]] = (w, None)
        var = rng.uniform(0.5, 2.0, L["K"]).astype(np.float32)
        gamma = np.sqrt(var + np.float32(1e-5)).astype(np.float32)
        bn[L["name"]] = (gamma, b, np.zeros(L["K"], np.float32), var)
    a1, a2 = oracle.bn_to_scale(*bn["c1"])
    assert np.all(a1 == 1.0) and np.array_equal(a2, W["c1"][1])
    plan = {"input": 8, "c1": {"w": 6, "b": 16, "s": 16, "h": 16, "a": 7},
            "c2": {"w": 7, "b": 16, "s": 16, "h": 16, "a": 8}, "fc": {"w": 8, "b": 16}}
    imgs = synth.images(3, 5, hw=6)
    f0, q0 = onet.calibrate(folded, W, imgs, plan)
    f1, q1 = onet.calibrate(withbn, Wbn, imgs, plan, bn)
    for nm in ("c1", "c2"):
        assert f1[nm]["s"] == (16, 0, 0) and np.all(q1[nm][2] == 1)
        assert f1[nm]["h"] == f0[nm]["b"] and np.array_equal(q1[nm][3], q0[nm][1])
        assert f1[nm]["a"] == f0[nm]["a"]
    l0, s0 = onet.forward(folded, f0, q0, imgs)
    l1, s1 = onet.forward(withbn, f1, q1, imgs)
    assert s0 == s1 and np.array_equal(l0, l1)


def test_scale_layer_gain_applies_before_relu_and_requant():
    """A Scale layer with gain -1 (gamma = -sqrt(var + eps)) and no shift flips the sign of the conv value
    before ReLU: the C-Block output equals relu(-conv), not -relu(conv)."""
    rng = np.random.default_rng(22)
    acc = rng.integers(-2 ** 20, 2 ** 20, size=(5, 4))
    v, s = oracle.cblock(acc, 10, None, 0, True, scale=np.full(4, -1), fl_scale=0, shift=np.zeros(4, np.int64),
                         fl_shift=0)
    assert s == 10 and np.array_equal(v, np.maximum(-acc, 0))


def test_memory_footprint_closed_forms():
    """Eq. mfp: nu * k / 2^23 MB, so 2^20 8-bit codes are exactly 1 MB and FP32 over k bits is 32 / k."""
    assert oracle.mfp(2 ** 20, 8) == 1.0
    assert oracle.mfp(2 ** 23, 1) == 1.0
    for k in range(2, 17):
        assert oracle.mfp(12345, 32) / oracle.mfp(12345, k) == pytest.approx(32 / k, rel=1e-15)


def _act_elems(layers, hw=224, cin=3):
    """Output elements per image of every layer (true channels), by plain shape propagation."""
    shapes = {"input": (hw, cin)}
    prev = "input"
    for L in layers:
        src = L.get("src") or prev
        h, c = shapes[L["a"] if L["type"] == "eltwise" else src]
        if L["type"] == "conv":
            shapes[L["name"]] = ((h + 2 * L["pad"] - L["R"]) // L["stride"] + 1, L["K"])
        elif L["type"] == "maxpool":
            shapes[L["name"]] = ((h + 2 * L["pad"] - L["k"]) // L["stride"] + 1, c)
        elif L["type"] == "avgpool":
            shapes[L["name"]] = (1, c)
        else:
            shapes[L["name"]] = (h, c)
        prev = L["name"]
    return {nm: h * h * c for nm, (h, c) in shapes.items()}


def test_memory_model_vgg16_fp32_textbook_figures():
    """VGG-16 in FP32: RO_R is its textbook 138,357,544 parameters at 32 bits; RW_R is conv1_2's input
    plus output (two 224 x 224 x 64 maps), the largest pair of any layer."""
    layers = synth.vgg16()
    elems = _act_elems(layers)
    rw = oracle.rw_r(layers, elems, {nm: 32 for nm in elems})
    assert rw == pytest.approx(2 * 224 * 224 * 64 * 32 / 2 ** 23, rel=1e-15)
    params = []
    for L in layers:
        if L["type"] == "conv":
            params += [(L["K"] * L["R"] * L["R"] * L["C"], 32), (L["K"], 32)]
    assert sum(n for n, _ in params) == 138357544
    assert oracle.ro_r(params) == pytest.approx(138357544 * 32 / 2 ** 23, rel=1e-15)


def test_memory_model_resnet18_residual_inputs():
    """ResNet-18: an eltwise layer reads both its operands (Sec. V-E.2); in FP32 the largest read-write pair
    is pool1 (conv1's 112 x 112 x 64 output in, 56 x 56 x 64 out), above any residual add's three maps."""
    layers = synth.resnet18()
    elems = _act_elems(layers)
    bits = {nm: 32 for nm in elems}
    assert oracle.rw_r(layers, elems, bits) == pytest.approx((112 * 112 * 64 + 56 * 56 * 64) * 32 / 2 ** 23)
    # an eltwise alone: its two inputs and its output
    one = [L for L in layers if L["name"] == "res1a"]
    assert oracle.rw_r(one, elems, bits) == pytest.approx(3 * 56 * 56 * 64 * 32 / 2 ** 23)


def test_pack_codes_worked_example_and_round_trip():
    """Packed k-bit storage: signed 3-bit codes (1, -1, 2) are the fields 001, 111, 010, so the bit-0 word
    is 0b011 = 3, the bit-1 word 0b110 = 6 and the bit-2 word 0b010 = 2; every code of every format
    survives the round trip, and the footprint is ceil(n / 32) * k words."""
    w = oracle.pack_codes([1, -1, 2], 3)
    assert w.tolist() == [3, 6, 2]
    assert oracle.unpack_codes(w, 3, 3, 1).tolist() == [1, -1, 2]
    rng = np.random.default_rng(41)
    for k in (2, 3, 5, 8, 11, 16):
        for S in (0, 1):
            n = 70
            c = rng.integers(oracle.qmin(k, S), oracle.qmax(k, S) + 1, size=n)
            c[:2] = [oracle.qmin(k, S), oracle.qmax(k, S)]
            words = oracle.pack_codes(c, k)
            assert words.size == 3 * k
            assert np.array_equal(oracle.unpack_codes(words, n, k, S), c)
            # bit b of the stream counts the codes whose field has bit b set
            for b in range(k):
                ones = sum(bin(int(x)).count("1") for x in words[b::k])
                assert ones == sum(((int(v) & ((1 << k) - 1)) >> b) & 1 for v in c)


# ---------------------------------------------------------------- score variants: binary quantizer, L1
def frac_val(x, k, S, fl):
    """Exact value of Q(x): code * 2^-FL, or for the signed 1-bit binary quantizer the decoded sign."""
    if k == 1 and S == 1:
        return (Fraction(-1) if F(x) < 0 else Fraction(1)) * Fraction(2) ** (-fl)
    return Fraction(frac_q(x, k, S, fl)) * Fraction(2) ** (-fl)


def test_binary_quantizer_worked_example():
    """Eq. fp_1_bit_quantization: -1 for x < 0, 0 for x >= 0 (-0.0 included); decoded 0 -> +1, so the values
    are +-2^-FL and the L2 / L1 errors are sums of (|x| - 2^-FL)^2 / ||x| - 2^-FL|."""
    x = np.array([-0.5, -0.0, 0.0, 3.0, -1e-30, 0.25], np.float32)
    assert oracle.quantize(x, 1, 1, 2).tolist() == [-1, 0, 0, 0, -1, 0]
    assert oracle.value(oracle.quantize(x, 1, 1, 2), 1, 1, 2).tolist() == [-0.25, 0.25, 0.25, 0.25, -0.25, 0.25]
    c = Fraction(1, 4)
    want2 = sum((abs(F(v)) - c) ** 2 for v in x)
    want1 = sum(abs(abs(F(v)) - c) for v in x)
    assert oracle.l2_error(x, 1, 1, 2) == float(want2)
    assert oracle.l1_error(x, 1, 1, 2) == float(want1)


def test_l1_bruteforce_all_candidates_and_argmin():
    """The L1 score (Eq. MAE without the 1/N) of every (k, FL), k = 1..16 and both sign strategies, against
    an exact Fraction brute force; argmin ties go to the smallest FL."""
    for seed in (23, 24):
        xs = _adversarial(seed, 10)[:16]
        for S in (1, 0):
            err, best, s_used, _ = oracle.fl_search(xs, S, 1, 16, -8, 23, score="l1")
            assert s_used == S
            for ki, k in enumerate(range(1, 17)):
                exact = [sum(abs(F(x) - frac_val(x, k, S, fl)) for x in xs) for fl in range(-8, 24)]
                assert err[ki].tolist() == [float(e) for e in exact], (k, S)
                assert best[ki] == -8 + exact.index(min(exact))


def test_l2_one_bit_row_bruteforce():
    """The k = 1 row of the L2 search: the binary quantizer for S = 1, the two levels {0, 1} for S = 0."""
    xs = _adversarial(25, 10)[:16]
    for S in (1, 0):
        err, best, _, _ = oracle.fl_search(xs, S, 1, 1, -8, 23)
        exact = [sum((F(x) - frac_val(x, 1, S, fl)) ** 2 for x in xs) for fl in range(-8, 24)]
        assert err[0].tolist() == [float(e) for e in exact]


def test_l1_closed_forms_and_cauchy_schwarz():
    """L1 is zero on the grid, |x - Q(x)| for one element, and L1^2 <= n * L2 (Cauchy-Schwarz)."""
    codes = np.arange(-128, 128)
    for fl in (-3, 0, 5):
        assert oracle.l1_error((codes * 2.0 ** -fl).astype(np.float32), 8, 1, fl) == 0.0
    for x in (0.3, -0.7, 5.25, -100.0):
        for k, S, fl in ((8, 1, 4), (2, 0, 1), (1, 1, 3)):
            assert oracle.l1_error(np.array([x], np.float32), k, S, fl) == float(abs(F(np.float32(x)) - frac_val(np.float32(x), k, S, fl)))
    xs = _adversarial(26, 200)
    for k, fl in ((4, 2), (8, 6), (1, 0)):
        l1, l2 = oracle.l1_error(xs, k, 1, fl), oracle.l2_error(xs, k, 1, fl)
        assert l1 * l1 <= xs.size * l2 * (1 + 1e-12)


# ---------------------------------------------------------------- forward optimizer (Alg. 1, cost F)
from oracle import qopt  # noqa: E402


def test_qparams_opt_hand_traced_search():
    """Alg. 1 on the convex cost (FL - 7)^2 from FL 4 with K = 1: direction -1 tries 3 and stops; direction
    +1 improves at 5, 6, 7 (each success extends the limit by one), tries 8 and stops."""
    calls = []

    def cost(fl):
        calls.append(fl)
        return float((fl - 7) ** 2)

    best, c, trace = qopt.qparams_opt(cost, 4, K=1)
    assert (best, c) == (7, 0.0)
    assert trace == [(4, 9.0), (3, 16.0), (5, 4.0), (6, 1.0), (7, 0.0), (8, 1.0)]
    # K = 2 also looks two steps to the left without an improvement; a tie is not an improvement
    best, c, trace = qopt.qparams_opt(lambda fl: float(abs(fl - 4) // 2), 4, K=2)
    assert best == 4 and [f for f, _ in trace] == [4, 3, 2, 5, 6]


def test_unclass_and_mispred_hand_example():
    """Eqs. unclassified_samples / mispredicted_classes: sample 0 ties two classes, sample 1 none, sample 2
    ties all three: UnClass = 2/3, MisPred = (1 + 0 + 2) / (3 * 3)."""
    lg = np.array([[1.0, 1.0, 0.0], [2.0, 0.0, 0.0], [5.0, 5.0, 5.0]])
    assert qopt.ties(lg).tolist() == [2, 1, 3]
    uc, mp = qopt.unclass_mispred(lg)
    assert uc == pytest.approx(2 / 3) and mp == pytest.approx(3 / 9)


def test_fp_conv_equals_integer_conv_on_integer_data():
    rng = np.random.default_rng(51)
    x = rng.integers(-20, 20, size=(2, 7, 6, 5))
    w = rng.integers(-9, 9, size=(4, 3, 3, 5))
    for st, pad in ((1, 1), (2, 0)):
        assert np.array_equal(qopt.f_conv(x, w, None, st, pad, False), oracle.conv2d(x, w, st, pad).astype(np.float64))


def _qopt_tiny():
    layers = [
        {"type": "conv", "name": "c1", "C": 3, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": True, "src": None},
        {"type": "maxpool", "name": "p1", "k": 2, "stride": 2, "pad": 0},
        {"type": "conv", "name": "c2", "C": 8, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": False, "src": "p1"},
        {"type": "eltwise", "name": "e", "a": "c2", "b": "p1", "relu": True},
        {"type": "avgpool", "name": "gap", "src": "e"},
        {"type": "conv", "name": "fc", "C": 8, "K": 10, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": "gap"},
    ]
    rng = np.random.default_rng(52)
    W = {}
    for L in layers:
        if L["type"] == "conv":
            fan = L["C"] * L["R"] ** 2
            W[L["name"]] = ((rng.standard_normal((L["K"], L["R"], L["R"], L["C"])) * np.sqrt(2 / fan)).astype(np.float32),
                            (rng.standard_normal(L["K"]) * 0.05).astype(np.float32))
    plan = {"input": 6, "c1": {"w": 5, "b": 8, "a": 5}, "c2": {"w": 4, "b": 8, "a": 6}, "e": {"a": 5},
            "gap": {"a": 6, "r": 16}, "fc": {"w": 6, "b": 8}}
    return layers, W, plan, synth.images(4, 53, hw=8)


def test_mixed_forward_fully_fixed_point_equals_integer_network():
    """With every data-structure fixed point, the mixed forward's logits equal the integer network's (oracle
    net) at the same formats, value for value; pi sums to one per layer."""
    layers, W, plan, imgs = _qopt_tiny()
    net = qopt.Net(layers, W, imgs, plan)
    last = net.order[-1]
    net_fmts = {"input": net.fmt[("input", "a")]}
    for L in layers:
        nm = L["name"]
        d = {}
        for j in ("w", "b", "a"):
            if (nm, j) in net.fmt:
                d[j] = net.fmt[(nm, j)]
        if L["type"] == "avgpool":
            d["r"] = net._recip(nm, 16)[0]
        net_fmts[nm] = d
    for ds in net.order[:-1]:
        net.done.add(ds)
    X, logits = net.forward(last, net.fmt[last][2])
    qparams = {}
    for L in layers:
        if L["type"] == "conv":
            nm = L["name"]
            qparams[nm] = (oracle.quantize(W[nm][0], *net_fmts[nm]["w"]).reshape(W[nm][0].shape),
                           oracle.quantize(W[nm][1], *net_fmts[nm]["b"]))
    want, s = onet.forward(layers, net_fmts, qparams, imgs)
    assert np.array_equal(logits, want.astype(np.float64) * 2.0 ** -s)
    # the importance weights of a layer's data-structures sum to one
    sts = [qopt.ds_stats(X[("c1", j)][0], j == "a") for j in ("a", "w", "b")]
    den = sum(s_ * n for s_, n, _ in sts)
    assert sum(s_ * n / den for s_, n, _ in sts) == pytest.approx(1.0)


def test_forward_optimizer_cost_is_zero_for_on_grid_data():
    """L is zero for data on the grid, so E vanishes for a data-structure whose every term is exact: a
    network of one 1x1 conv with power-of-two weights and integer images has E = 0 for its bias."""
    layers = [{"type": "conv", "name": "fc", "C": 3, "K": 4, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": None}]
    W = {"fc": (np.array([1, 0.5, -2, 0.25] * 3, np.float32).reshape(4, 1, 1, 3), np.array([1, 2, 3, 4], np.float32))}
    imgs = np.random.default_rng(54).integers(-3, 4, size=(2, 3, 2, 2)).astype(np.float32)
    net = qopt.Net(layers, W, imgs, {"input": 8, "fc": {"w": 8, "b": 8}})
    F_, E, uc, mp = net.cost(("fc", "b"), net.fmt[("fc", "b")][2])
    assert E == 0.0
    assert F_ == uc + mp


# ---------------------------------------------------------------- forward optimizer: E, pi, sigma, R
def _pop_sigma(vals):
    """Population standard deviation from the exact mean and variance (Fractions), then one sqrt."""
    fr = [F(v) for v in vals]
    m = sum(fr) / len(fr)
    return float(sum((v - m) ** 2 for v in fr) / len(fr)) ** 0.5


def test_ds_stats_population_sigma_and_per_sample_activations():
    """Eq. importance's sigma is the population deviation; activations take it per sample (averaged over
    the calibration samples) with nu the per-sample size; Eq. data_range's R = max - min."""
    s, n, R = qopt.ds_stats(np.array([1.0, 2.0, 3.0, 6.0]), per_sample=False)
    assert s == pytest.approx(3.5 ** 0.5, rel=1e-15) and n == 4 and R == 5.0  # sample deviation: sqrt(14/3)
    s, n, R = qopt.ds_stats(np.array([[0.0, 2.0], [1.0, 5.0]]), per_sample=True)
    assert s == pytest.approx(1.5, rel=1e-15) and n == 2 and R == 5.0  # per-tensor: sqrt(3.5), nu 4


def _two_layer_net():
    """conv c1 (1x1, 1 -> 2 channels, no ReLU) then fc (1x1 over 2x2 maps of 2 channels -> 2 classes),
    hand-sized weights, two 2x2 single-channel images."""
    layers = [{"type": "conv", "name": "c1", "C": 1, "K": 2, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": None},
              {"type": "conv", "name": "fc", "C": 2, "K": 2, "R": 2, "stride": 1, "pad": 0, "relu": False, "src": None}]
    W = {"c1": (np.array([0.8125, -0.40625], np.float32).reshape(2, 1, 1, 1), np.array([0.1, -0.3], np.float32)),
         "fc": (np.array([0.3, -0.7, 0.45, 0.2, -0.15, 0.6, 0.05, -0.35,
                          0.25, 0.5, -0.6, 0.1, 0.7, -0.2, 0.35, 0.15], np.float32).reshape(2, 2, 2, 2),
                np.array([0.02, -0.01], np.float32))}
    imgs = np.array([[[[1.3, -0.7], [0.4, 2.1]]], [[[-1.6, 0.9], [0.25, -0.45]]]], np.float32)
    plan = {"input": 6, "c1": {"w": 4, "b": 5, "a": 5}, "fc": {"w": 5, "b": 6}}
    return layers, W, imgs, plan


def _fq(v, fmt):
    k, S, fl = fmt
    return Fraction(frac_q(v, k, S, fl)) * Fraction(2) ** (-fl)


def _term(vals, fmt, per_sample, nsamp):
    """(sigma * nu, L / R) of one data-structure straight from Eqs. importance, DSB_QE and data_range."""
    flat = [float(v) for v in np.asarray(vals, np.float64).ravel()]
    if per_sample:
        m = len(flat) // nsamp
        sig = sum(_pop_sigma(flat[i * m:(i + 1) * m]) for i in range(nsamp)) / nsamp
        nu = m
    else:
        sig, nu = _pop_sigma(flat), len(flat)
    L = sum((F(v) - _fq(v, fmt)) ** 2 for v in flat)
    R = F(max(flat)) - F(min(flat))
    return sig * nu, (float(L / R) if R else 0.0)


def _E(layer_terms):
    """Eq. CPB_QE: per layer, pi_j = sigma_j nu_j / sum (sigma nu), E = sum pi_j L_j / R_j."""
    E = 0.0
    for terms in layer_terms:
        den = sum(sn for sn, _ in terms)
        E += sum(sn / den * lr for sn, lr in terms)
    return E


def test_cost_E_from_the_equations_with_a_later_layer_fp32():
    """E for c1's weights at candidate FLs: the input is fixed point (optimized before), c1's weights take
    the candidate, c1's bias and activations and all of fc are FP32 -- and each term's L is taken under
    its own QPs (candidate, or the initial QPs of the preprocessor)."""
    layers, W, imgs, plan = _two_layer_net()
    net = qopt.Net(layers, W, imgs, plan)
    x = np.transpose(imgs.astype(np.float64), (0, 2, 3, 1))  # NHWC, one channel
    fin = net.fmt[("input", "a")]
    xq = [[_fq(v, fin) for v in img.ravel()] for img in x]
    w1, b1 = W["c1"]
    for cand in (net.fmt[("c1", "w")][2] - 1, net.fmt[("c1", "w")][2], net.fmt[("c1", "w")][2] + 2):
        fw = (net.fmt[("c1", "w")][0], net.fmt[("c1", "w")][1], cand)
        wq = [_fq(v, fw) for v in w1.ravel()]
        # c1's output (FP32 bias, no ReLU): sample-major, pixel, channel
        y = [[float(xq[n][p] * wq[c] + F(b1[c])) for p in range(4) for c in range(2)] for n in range(2)]
        c1_terms = [_term(y, net.fmt[("c1", "a")], True, 2), _term(w1, fw, False, 1),
                    _term(b1, net.fmt[("c1", "b")], False, 1)]
        fc_terms = [_term(W["fc"][0], net.fmt[("fc", "w")], False, 1), _term(W["fc"][1], net.fmt[("fc", "b")], False, 1)]
        want = _E([c1_terms, fc_terms])
        _, E, _, _ = net.cost(("c1", "w"), cand)
        assert E == pytest.approx(want, rel=1e-12)


def test_cost_E_in_a_mixed_state_with_a_quantized_prefix():
    """E for fc's weights once input, c1's w, b and a are fixed point at their QPs: only layer fc's terms
    count, fc's input is c1's quantized output, and fc's bias keeps its initial QPs (FP32 values)."""
    layers, W, imgs, plan = _two_layer_net()
    net = qopt.Net(layers, W, imgs, plan)
    for ds in net.order[:4]:
        net.done.add(ds)
    cur = ("fc", "w")
    assert net.order[4] == cur
    for cand in (net.fmt[cur][2], net.fmt[cur][2] + 1):
        fw = (net.fmt[cur][0], net.fmt[cur][1], cand)
        _, E, uc, mp = net.cost(cur, cand)
        want = _E([[_term(W["fc"][0], fw, False, 1), _term(W["fc"][1], net.fmt[("fc", "b")], False, 1)]])
        assert E == pytest.approx(want, rel=1e-12)
    # the logits of this forward: quantized input, c1 weights, bias and output, candidate fc weights
    x = np.transpose(imgs.astype(np.float64), (0, 2, 3, 1))
    fin, f1w, f1b, f1a = (net.fmt[d] for d in net.order[:4])
    fw = net.fmt[cur]
    w1, b1 = W["c1"]
    wf, bf = W["fc"]
    logits = []
    for n in range(2):
        h = [[_fq(_fq(x[n].ravel()[p], fin) * _fq(w1.ravel()[c], f1w) + _fq(b1[c], f1b), f1a) for c in range(2)]
             for p in range(4)]
        logits.append([sum(h[p][c] * _fq(wf[o].reshape(4, 2)[p, c], fw) for p in range(4) for c in range(2)) + F(bf[o])
                       for o in range(2)])
    X, lg = net.forward(cur, fw[2])
    assert np.array_equal(lg, np.array([[float(v) for v in row] for row in logits]))
