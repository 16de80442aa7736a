"""GPU parity of the C-Block kernels (conv / FC with the fused epilogue, max-pool, eltwise,
avg-pool) against the CPU oracle: bit-exact codes, accumulators and fp32 calibration images."""
import os

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", params=["tc", "tc_rows", "tc_bn256", "simt"])
def F(request):
    """Runs every case on the tensor-core kernel (default: patch tiles where the layer allows
    them), on the tensor-core kernel with 128-row tiles only, on the tensor-core kernel with
    256-column tiles wherever K > 128, and on the CUDA-core kernel."""
    import os
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import fxpq
    old = os.environ.get("FXPQ_CONV_PATH")
    os.environ["FXPQ_CONV_PATH"] = request.param
    yield fxpq
    if old is None:
        os.environ.pop("FXPQ_CONV_PATH", None)
    else:
        os.environ["FXPQ_CONV_PATH"] = old


def rand_codes(rng, shape, k, S):
    lo, hi = oracle.qmin(k, S), oracle.qmax(k, S)
    c = rng.integers(lo, hi + 1, size=shape)
    # make the extremes appear
    flat = c.reshape(-1)
    flat[: min(4, flat.size)] = [lo, hi, lo, hi][: min(4, flat.size)]
    return c


def to_f16_planes(codes, k, Cp):
    """Storage encoding of a code tensor [..., C] as a plane-major fp16 code tensor [..., Cp] (zero padded)."""
    c = np.zeros(codes.shape[:-1] + (Cp,), np.int64)
    c[..., : codes.shape[-1]] = codes
    if k <= 8:
        return torch.from_numpy(c.astype(np.float16)).cuda()
    hi = c >> 8
    lo = c - (hi << 8)
    return torch.from_numpy(np.stack([hi, lo]).astype(np.float16)).cuda()


def run_conv(F, x, fx, w, fw, b, fb, stride, pad, relu, mode, fy, Cp, w_l1=0, scale=None, packed_w=None):
    """packed_w: one-plane weight codes [K, R, S, C] whose packed records (fxpq_pack_weights) go with the
    descriptor (normally w itself)."""
    N, H, W, C = x.shape
    K, R, S, _ = w.shape
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    xd = to_f16_planes(x, fx.bits, Cp)
    wd = to_f16_planes(w, fw.bits, Cp)
    bd = torch.from_numpy(b.astype(np.int32)).cuda() if b is not None else None
    if mode == F.OUT_CODES:
        y = torch.empty(N * P * Q * K * (2 if fy.bits > 8 else 1), dtype=torch.float16, device="cuda")
    elif mode == F.OUT_ACC64:
        y = torch.empty(N * P * Q * K, dtype=torch.int64, device="cuda")
    else:
        y = torch.empty(N * P * Q * K, dtype=torch.float32, device="cuda")
    sd = hd = fs = fh = None
    if scale is not None:
        m, fs, h, fh = scale
        sd = torch.from_numpy(m.astype(np.int32)).cuda()
        hd = torch.from_numpy(h.astype(np.int32)).cuda()
    wp = None
    if packed_w is not None:
        wp = F.pack_weights(to_f16_planes(packed_w, fw.bits, Cp), fw, K, R * S * Cp)
    d = F.conv_desc(N, H, W, C, Cp, K, R, S, stride, pad, relu, mode, fx, fw, fb, fy, w_l1,
                    scale=sd, fmt_scale=fs, shift=hd, fmt_shift=fh, wpacked=wp)
    nws = F.fxpq_conv_workspace(d)
    ws = torch.empty(nws, dtype=torch.uint8, device="cuda") if nws else None
    s = F.fxpq_conv_fwd(d, xd, wd, bd, y, ws=ws)
    torch.cuda.synchronize()
    assert F.fxpq_get_device_status() == 0
    if mode == F.OUT_CODES:
        return F.codes_to_int(y.cpu(), fy, (N, P, Q, K)).numpy(), s
    return y.cpu().numpy().reshape(N, P, Q, K), s


def oracle_conv(x, fx, w, fw, b, fb, stride, pad, relu, mode, fy, scale=None):
    acc = oracle.conv2d(x, w, stride, pad)
    if scale is None:
        v, s = oracle.cblock(acc, fx.fl + fw.fl, b, fb.fl if fb is not None else 0, relu)
    else:
        m, fs, h, fh = scale
        v, s = oracle.cblock(acc, fx.fl + fw.fl, b, fb.fl if fb is not None else 0, relu,
                             scale=m, fl_scale=fs.fl, shift=h, fl_shift=fh.fl)
    if mode == 0:
        return oracle.requant(v, s, fy.bits, fy.is_signed, fy.fl), s
    if mode == 1:
        return v, s
    return oracle.to_f32(v, s), s


CASES = [
    # N, H, C, K, R, stride, pad, (kx,Sx,flx), (kw,Sw,flw), (kb,flb) or None, relu, mode, (ky,Sy,fly)
    (2, 9, 8, 16, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),
    (3, 13, 24, 72, 5, 2, 2, (8, 0, 2), (8, 1, 9), (16, 19), True, 0, (8, 0, 5)),
    (2, 39, 3, 96, 11, 4, 2, (8, 1, 5), (8, 1, 8), (16, 18), True, 0, (8, 0, 2)),
    (2, 14, 64, 32, 1, 2, 0, (6, 0, 3), (7, 1, 8), (16, 17), False, 0, (7, 1, 4)),
    (3, 6, 64, 24, 6, 1, 0, (8, 0, 4), (4, 1, 6), (16, 16), True, 0, (8, 0, 1)),
    (2, 11, 16, 16, 3, 1, 1, (16, 1, 12), (16, 1, 14), (16, 20), True, 0, (16, 0, 9)),
    (1, 10, 8, 8, 3, 1, 1, (16, 1, 12), (16, 1, 14), (16, 20), False, 1, None),
    (2, 9, 16, 40, 3, 1, 1, (5, 1, 2), (4, 1, 3), (16, 9), False, 1, None),        # delta < 0: acc shifted left
    (2, 9, 16, 40, 3, 1, 0, (8, 0, 4), (8, 1, 7), None, True, 2, None),            # no bias, fp32 calibration image
    (2, 8, 32, 16, 3, 2, 1, (8, 0, 6), (8, 1, 8), (16, 22), False, 2, None),
    (4, 7, 8, 8, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (4, 0, 20)),      # left-shift requant + saturate
    (1, 5, 3, 8, 3, 1, 1, (3, 1, 1), (3, 1, 2), (16, 10), True, 0, (2, 0, 0)),
    # bias finer than the accumulator (delta < 0) on the 32-bit epilogue: fractional bias parts, ties
    (2, 9, 16, 40, 3, 1, 1, (5, 1, 2), (4, 1, 3), (16, 9), False, 0, (6, 1, 1)),
    (2, 9, 16, 40, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 19), True, 0, (8, 0, 6)),
    (2, 7, 8, 16, 3, 1, 1, (3, 1, 0), (3, 1, 0), (16, 3), False, 0, (8, 1, -1)),
    (3, 12, 64, 136, 3, 1, 1, (8, 0, 6), (8, 1, 9), (16, 24), True, 0, (8, 0, 12)),
    # stride 1, Cp % 64 == 0: patch tiles (TMA windows with zero-filled padding) on the tensor cores
    (2, 16, 64, 128, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),       # 16 x 8 patches
    (2, 28, 64, 72, 3, 1, 1, (8, 0, 5), (8, 1, 8), (16, 17), True, 0, (8, 0, 4)),        # 28 x 4: 112 rows, ragged K
    (2, 18, 64, 64, 3, 1, 0, (7, 0, 3), (6, 1, 7), (16, 14), False, 0, (8, 1, 2)),       # no padding
    (2, 16, 64, 64, 5, 1, 2, (8, 0, 4), (8, 1, 9), (16, 18), True, 0, (8, 0, 6)),        # 5 x 5 taps
    (2, 10, 128, 64, 3, 1, 1, (8, 0, 4), (8, 1, 7), None, True, 2, None),               # 10 x 10 patch, fp32 image
    (2, 10, 128, 64, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), False, 1, None),          # int64 accumulators
    (1, 16, 64, 64, 3, 1, 1, (16, 1, 12), (16, 1, 14), (16, 20), True, 0, (16, 0, 9)),   # two limbs, two planes out
    (2, 16, 64, 40, 3, 1, 1, (5, 1, 2), (4, 1, 3), (16, 9), False, 0, (6, 1, 1)),        # bias finer than acc
    (1, 16, 256, 128, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),      # several exact groups
    # K > 128: 256-column tiles under tc_bn256 (one exact group: two accumulator buffers; several:
    # one buffer plus integer running sums)
    (2, 8, 64, 256, 3, 1, 1, (6, 0, 2), (6, 1, 5), (16, 12), True, 0, (8, 0, 3)),
    (1, 16, 256, 256, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),
    (2, 9, 16, 264, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),        # ragged K, row tiles
    (2, 8, 64, 256, 3, 1, 1, (8, 0, 4), (8, 1, 7), None, True, 2, None),               # fp32 image
    (2, 8, 64, 256, 3, 1, 1, (8, 0, 4), (8, 1, 7), (16, 15), False, 1, None),          # int64 accumulators
    # 8-channel stride-1 inputs: patch tiles with one box per tap (VGG conv1_1-like, two limbs)
    (2, 20, 3, 16, 5, 1, 2, (16, 1, 12), (16, 1, 14), (16, 20), True, 0, (8, 0, 3)),
    (3, 16, 3, 64, 3, 1, 1, (16, 1, 11), (16, 1, 14), (16, 22), True, 0, (4, 0, 2)),
    # window mode (8 stored channels, stride 1, K <= 64): ragged patches, 1x1 taps, one plane, ACC64
    (2, 20, 3, 64, 3, 1, 1, (16, 1, 11), (16, 1, 13), (16, 21), True, 0, (8, 0, 3)),
    (2, 12, 8, 24, 1, 1, 0, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),
    (1, 19, 5, 40, 3, 1, 1, (7, 1, 3), (6, 1, 6), (16, 12), False, 0, (8, 1, 2)),
    (2, 17, 3, 32, 3, 1, 1, (16, 1, 11), (16, 1, 14), (16, 22), True, 1, None),
    # FC-like layers (few output rows, long reductions): the split reduction across SMs, one- and
    # two-limb, every output mode, with biases coarser and finer than the accumulator
    (3, 7, 512, 200, 7, 1, 0, (8, 0, 4), (6, 1, 8), (16, 15), True, 0, (8, 0, 3)),
    (2, 7, 512, 96, 7, 1, 0, (8, 0, 4), (16, 1, 15), (16, 22), False, 1, None),
    (5, 1, 4096, 136, 1, 1, 0, (5, 0, 2), (7, 1, 9), (16, 8), False, 2, None),
    (4, 1, 4096, 1000, 1, 1, 0, (16, 0, 12), (16, 1, 18), (16, 20), False, 1, None),
    (9, 3, 512, 64, 3, 1, 0, (7, 0, 3), (5, 1, 6), (16, 4), True, 0, (6, 0, 1)),
    # 1x1 stride-1 layers without padding: 128-row tiles whose A tile is one 2-D TMA box of [M][Cp]
    # (ragged M, M below one tile, two-limb activations with int64 sums, 256 output channels)
    (3, 9, 64, 72, 1, 1, 0, (8, 0, 4), (8, 1, 7), (16, 15), True, 0, (8, 0, 3)),
    (2, 20, 128, 128, 1, 1, 0, (16, 1, 12), (8, 1, 7), (16, 20), False, 1, None),
    (1, 11, 192, 256, 1, 1, 0, (7, 0, 3), (6, 1, 6), (16, 12), True, 0, (8, 0, 2)),
    (2, 13, 40, 24, 1, 1, 0, (8, 0, 4), (8, 1, 7), None, True, 2, None),
    # window mode, two limbs, one-plane codes: the 32-bit epilogue (shift >= 17, bias not finer), its
    # shift-17 edge and no ReLU with signed codes, and the 64-bit fallback for a finer bias
    (2, 20, 3, 48, 3, 1, 1, (16, 1, 9), (16, 1, 12), (16, 18), False, 0, (6, 1, 2)),
    (1, 18, 3, 64, 3, 1, 1, (16, 1, 9), (16, 1, 10), (16, 17), True, 0, (8, 0, 2)),
    (2, 20, 3, 64, 3, 1, 1, (16, 1, 11), (16, 1, 13), (16, 30), False, 0, (8, 1, 3)),
    # 64-channel window mode (stride 1, one plane, Cp % 16 == 0 and <= 64, K <= 64, one exact group):
    # ragged maps, every supported Cp, no padding, 2 x 2 taps, every output mode
    (2, 19, 64, 64, 3, 1, 1, (8, 0, 4), (7, 1, 8), (16, 15), True, 0, (8, 0, 3)),
    (3, 12, 32, 48, 3, 1, 1, (6, 0, 2), (5, 1, 5), (16, 10), False, 0, (8, 1, 2)),
    (2, 10, 16, 64, 3, 1, 0, (8, 0, 4), (8, 1, 7), None, True, 2, None),
    (1, 9, 48, 24, 2, 1, 0, (4, 0, 1), (8, 1, 9), (16, 12), True, 1, None),
    # the fp32 image of a C-Block output (calibration) from both window instances: two limbs with and
    # without ReLU, and the 64-channel window
    (2, 20, 3, 64, 3, 1, 1, (16, 1, 11), (16, 1, 13), (16, 21), True, 2, None),
    (1, 18, 3, 48, 3, 1, 1, (16, 1, 9), (16, 1, 10), (16, 17), False, 2, None),
    (2, 19, 64, 64, 3, 1, 1, (8, 0, 4), (7, 1, 8), (16, 15), True, 2, None),
    # the 32-bit window epilogue at its smallest shift (16: the tie is decided by the low 16 bits alone),
    # and one below it (15: the 64-bit path)
    (1, 16, 3, 32, 3, 1, 1, (16, 1, 9), (16, 1, 10), (16, 15), False, 0, (8, 1, 3)),
    (1, 16, 3, 32, 3, 1, 1, (16, 1, 9), (16, 1, 10), (16, 15), True, 0, (8, 1, 4)),
]


def run_case(F, case, use_l1=False):
    N, H, C, K, R, st, pad, tx, tw, tb, relu, mode, ty = case
    rng = np.random.default_rng(H * 131 + K)
    fx, fw = F.fmt(*tx), F.fmt(*tw)
    fb = F.fmt(tb[0], 1, tb[1]) if tb else None
    fy = F.fmt(*ty) if ty else None
    x = rand_codes(rng, (N, H, H, C), tx[0], tx[1])
    w = rand_codes(rng, (K, R, R, C), tw[0], tw[1])
    w = np.where(rng.random(w.shape) < 0.8, w // 4, w)
    b = rand_codes(rng, (K,), tb[0], 1) if tb else None
    Cp = (C + 7) // 8 * 8
    w_l1 = int(np.abs(w).reshape(K, -1).sum(axis=1).max()) if use_l1 else 0
    got, s = run_conv(F, x, fx, w, fw, b, fb, st, pad, relu, mode, fy, Cp, w_l1)
    want, ws = oracle_conv(x, fx, w, fw, b, fb, st, pad, relu, mode, fy)
    assert s == ws
    assert np.array_equal(got, want)


@pytest.mark.parametrize("case", [c for c in CASES if c[8][0] <= 8])
def test_conv_parity_l1_bound(F, case):
    """The weight-code L1 bound lets the tensor-core path take the whole reduction as one exact
    fp32 group (and a 32-bit epilogue) where the wordlength bound alone would split it."""
    run_case(F, case, use_l1=True)


@pytest.mark.parametrize("case", CASES)
def test_conv_parity(F, case):
    run_case(F, case)


WINDOW_TWO_LIMB = [c for c in CASES if c[2] <= 8 and c[3] <= 64 and c[5] == 1 and c[7][0] > 8 and c[8][0] > 8]


@pytest.mark.parametrize("alt", ["tc_win64"])
@pytest.mark.parametrize("case", WINDOW_TWO_LIMB)
def test_window_epilogue_alternatives(F, case, alt):
    """Window mode's two-limb epilogue in its 64-bit form on the same cases as the default (32-bit
    where the bounds allow)."""
    if os.environ.get("FXPQ_CONV_PATH") != "tc":
        pytest.skip("alternative forms of the default tensor-core path")
    os.environ["FXPQ_CONV_PATH"] = alt
    try:
        run_case(F, case)
    finally:
        os.environ["FXPQ_CONV_PATH"] = "tc"


def test_code_l1max(F):
    """max over rows of sum |code| on one-plane fp16 codes, against numpy; the zero-row case."""
    rng = np.random.default_rng(11)
    for rows, L_, lo, hi in ((37, 8 * 163, -128, 127), (1, 8, 0, 255), (300, 4608, -8, 7)):
        c = rng.integers(lo, hi + 1, size=(rows, L_))
        c[rows // 2, :] = hi if abs(hi) > abs(lo) else lo  # the extreme row
        d = torch.from_numpy(c.astype(np.float16)).cuda()
        out = torch.full((1,), -1, dtype=torch.int64, device="cuda")
        F.fxpq_code_l1max(d, rows, L_, out)
        assert int(out.item()) == int(np.abs(c).sum(axis=1).max())
    out = torch.full((1,), -1, dtype=torch.int64, device="cuda")
    F.fxpq_code_l1max(torch.empty(8, dtype=torch.float16, device="cuda"), 0, 8, out)
    assert int(out.item()) == 0


def test_gemm_entry_point(F):
    rng = np.random.default_rng(3)
    M, N, Kd = 37, 48, 200
    fx, fw, fb, fy = F.fmt(8, 0, 5), F.fmt(8, 1, 9), F.fmt(16, 1, 20), F.fmt(8, 0, 4)
    x = rand_codes(rng, (M, Kd), 8, 0)
    w = rand_codes(rng, (N, Kd), 8, 1) // 3
    b = rand_codes(rng, (N,), 16, 1)
    y = torch.empty(M * N, dtype=torch.float16, device="cuda")
    s = F.fxpq_gemm(to_f16_planes(x, 8, Kd), fx, to_f16_planes(w, 8, Kd), fw, torch.from_numpy(b.astype(np.int32)).cuda(),
                    fb, M, N, Kd, True, F.OUT_CODES, fy, y)
    want, ws = oracle_conv(x.reshape(M, 1, 1, Kd), fx, w.reshape(N, 1, 1, Kd), fw, b, fb, 1, 0, True, 0, fy)
    assert s == ws
    assert np.array_equal(F.codes_to_int(y.cpu(), fy, (M, N)).numpy(), want.reshape(M, N))


@pytest.mark.parametrize("k,st,pad,bits", [(3, 2, 0, 8), (2, 2, 0, 6), (3, 2, 1, 8), (3, 2, 1, 12), (3, 1, 1, 4)])
def test_maxpool_parity(F, k, st, pad, bits):
    rng = np.random.default_rng(k + st + pad + bits)
    N, H, C = 2, 15, 24
    x = rand_codes(rng, (N, H, H, C), bits, 0)
    f = F.fmt(bits, 0, 3)
    P = (H + 2 * pad - k) // st + 1
    y = torch.empty(N * P * P * C * (2 if bits > 8 else 1), dtype=torch.float16, device="cuda")
    F.fxpq_maxpool(to_f16_planes(x, bits, C), N, H, H, C, f, k, st, pad, y)
    got = F.codes_to_int(y.cpu(), f, (N, P, P, C)).numpy()
    assert np.array_equal(got, oracle.maxpool(x, k, st, pad))


@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("fa,fb,relu", [((8, 1, 5), (7, 1, 3), True), ((6, 0, 2), (8, 1, 6), False),
                                        ((16, 1, 10), (8, 0, 4), True)])
def test_eltwise_parity(F, mode, fa, fb, relu):
    rng = np.random.default_rng(sum(fa) + sum(fb) + mode)
    npix, C = 333, 16
    a = rand_codes(rng, (npix, C), fa[0], fa[1])
    b = rand_codes(rng, (npix, C), fb[0], fb[1])
    FA, FB, FY = F.fmt(*fa), F.fmt(*fb), F.fmt(7, 0 if relu else 1, 4)
    if mode == 0:
        y = torch.empty(npix * C, dtype=torch.float16, device="cuda")
    elif mode == 1:
        y = torch.empty(npix * C, dtype=torch.int64, device="cuda")
    else:
        y = torch.empty(npix * C, dtype=torch.float32, device="cuda")
    s = F.fxpq_eltwise(to_f16_planes(a, fa[0], C), FA, to_f16_planes(b, fb[0], C), FB, npix, C, relu, mode, FY, y)
    v, ws = oracle.eltwise_add(a, fa[2], b, fb[2], relu)
    assert s == ws
    if mode == 0:
        assert np.array_equal(F.codes_to_int(y.cpu(), FY, (npix, C)).numpy(), oracle.requant(v, ws, 7, FY.is_signed, 4))
    elif mode == 1:
        assert np.array_equal(y.cpu().numpy().reshape(npix, C), v)
    else:
        assert np.array_equal(y.cpu().numpy().reshape(npix, C), oracle.to_f32(v, ws))


@pytest.mark.parametrize("s,fy", [(20, (8, 0, 6)), (11, (16, 1, 3)), (5, (4, 1, 9)), (30, (8, 1, 30)), (0, (6, 1, -2))])
def test_qlayer_parity(F, s, fy):
    rng = np.random.default_rng(s + 100)
    v = rng.integers(-2 ** 40, 2 ** 40, size=1001)
    v[:6] = [0, 1, -1, 3 << 9, -(3 << 9), 5 << 9]
    vd = torch.from_numpy(v).cuda()
    FY = F.fmt(*fy)
    y = torch.empty(v.size * (2 if fy[0] > 8 else 1), dtype=torch.float16, device="cuda")
    F.fxpq_qlayer(vd, s, F.OUT_CODES, FY, y)
    assert np.array_equal(F.codes_to_int(y.cpu(), FY, (v.size,)).numpy(), oracle.requant(v, s, *fy))
    small = v >> 12  # the fp32 image needs |v| < 2^53 on the oracle side
    f = torch.empty(v.size, dtype=torch.float32, device="cuda")
    F.fxpq_qlayer(torch.from_numpy(small).cuda(), s, F.OUT_F32, None, f)
    assert np.array_equal(f.cpu().numpy(), oracle.to_f32(small, s))


@pytest.mark.parametrize("bits", [5, 8, 11])
def test_avgpool_parity(F, bits):
    rng = np.random.default_rng(bits)
    N, H, C = 3, 7, 40
    x = rand_codes(rng, (N, H, H, C), bits, 0)
    fx, fr, fy = F.fmt(bits, 0, 4), F.fmt(16, 0, 21), F.fmt(8, 0, 5)
    rc = int(oracle.quantize(np.array([1 / 49], np.float32), 16, 0, 21)[0])
    y = torch.empty(N * C, dtype=torch.float16, device="cuda")
    s = F.fxpq_avgpool(to_f16_planes(x, bits, C), N, H, H, C, fx, rc, fr, F.OUT_CODES, fy, y)
    v, ws = oracle.avgpool_global(x, 4, rc, 21)
    assert s == ws
    assert np.array_equal(F.codes_to_int(y.cpu(), fy, (N, C)).numpy(), oracle.requant(v, ws, 8, 0, 5))


# Scale layer cases: a CASES geometry, then (k, FL) of aleph1 and of aleph2 (both signed)
SCALE_CASES = [
    (CASES[0], (16, 14), (16, 12)),     # 8-bit, bias; 64-bit epilogue with the Scale layer
    (CASES[8], (16, 13), (16, 10)),     # no bias (ResNet-style conv), fp32 calibration image
    (CASES[7], (12, 9), (16, 30)),      # ACC64; aleph2 finer than the product (delta2 < 0)
    (CASES[10], (16, 14), (16, 12)),    # requantizing left shift and saturation
    (CASES[12], (8, 5), (16, 3)),       # bias finer than the accumulator, then the Scale layer
    (CASES[16], (16, 14), (16, 11)),    # patch tiles
    (CASES[22], (16, 15), (16, 13)),    # two limbs in, two planes out
    (CASES[25], (16, 14), (16, 12)),    # 256-column tiles
    (CASES[32], (16, 14), (16, 12)),    # window mode, two-limb fast epilogue
    (CASES[35], (16, 14), (16, 12)),    # window mode, ACC64
    (CASES[41], (16, 14), (16, 12)),    # 1x1: A tiles as 2-D TMA boxes
    (CASES[48], (16, 14), (16, 12)),    # 64-channel window mode
    (CASES[36], (16, 14), (16, 12)),    # split reduction
    (CASES[39], (16, 13), (16, 10)),    # split reduction, two limbs, ACC64
]


@pytest.mark.parametrize("sc", SCALE_CASES)
def test_conv_scale_layer_parity(F, sc):
    """CONV (+bias) -> Scale (aleph1, aleph2) -> ReLU -> FxP-QLayer (Sec. IV-A.1, IV-B), bit-exact."""
    case, (ks, fls), (kh, flh) = sc
    N, H, C, K, R, st, pad, tx, tw, tb, relu, mode, ty = case
    rng = np.random.default_rng(H * 131 + K + 7)
    fx, fw = F.fmt(*tx), F.fmt(*tw)
    fb = F.fmt(tb[0], 1, tb[1]) if tb else None
    fy = F.fmt(*ty) if ty else None
    x = rand_codes(rng, (N, H, H, C), tx[0], tx[1])
    w = rand_codes(rng, (K, R, R, C), tw[0], tw[1])
    w = np.where(rng.random(w.shape) < 0.8, w // 4, w)
    b = rand_codes(rng, (K,), tb[0], 1) if tb else None
    m = rand_codes(rng, (K,), ks, 1)
    h = rand_codes(rng, (K,), kh, 1)
    scale = (m, F.fmt(ks, 1, fls), h, F.fmt(kh, 1, flh))
    Cp = (C + 7) // 8 * 8
    got, s = run_conv(F, x, fx, w, fw, b, fb, st, pad, relu, mode, fy, Cp, scale=scale)
    want, ws = oracle_conv(x, fx, w, fw, b, fb, st, pad, relu, mode, fy,
                           scale=(m, scale[1], h, scale[3]))
    assert s == ws
    assert np.array_equal(got, want)


# ---------------------------------------------------------------- exactness at the fp32 group bound
def _edge_case(kind, K):
    """Codes that drive every exact fp32 group of the tensor-core path to its planner bound, with odd
    partial sums (an accumulator that dropped low bits would change them).

    "wordlength": 8-bit unsigned x = 255, 8-bit signed w = -128 or 127: the bound alone makes groups of
      512 taps (255 * 128 * 512 = 16,711,680 < 2^24), and one weight per channel is nudged by one so
      that every group sum is odd.
    "limbs": 16-bit codes whose low limbs are all 255: lo x lo products of 65,025 in groups of 256
      taps (16,646,400).
    "l1": 8-bit unsigned x = 255 with sum |w[o]| = 65,793, so that max|x| * w_l1 = 2^24 - 1: the L1
      bound makes the whole reduction one group and channels of one sign reach exactly +-(2^24 - 1).
    """
    N, H, C, R = 2, 5, 64, 3  # 3 x 3 taps over 64 channels: 576 taps per output, no padding
    taps = R * R * C
    rng = np.random.default_rng({"wordlength": 1, "limbs": 2, "l1": 3}[kind] * 100 + K)
    if kind == "limbs":
        hi_x = rng.integers(-100, 100, size=(N, H, H, C))
        x = hi_x * 256 + 255
        hi_w = rng.integers(-100, 100, size=(K, taps))
        lo_w = np.full((K, taps), 255)
        lo_w[:, [0, 256, 512]] = 254  # one even product per 256-tap group: odd group sums
        w = (hi_w * 256 + lo_w).reshape(K, R, R, C)
        return x, (16, 1, 12), w, (16, 1, 14), (16, 1, 20)
    x = np.full((N, H, H, C), 255)
    x[0, 0, 0, :5] = [254, 253, 1, 0, 128]  # a few other codes so the rows differ
    if kind == "wordlength":
        sign = np.where(np.arange(K) % 2 == 0, -1, 1)
        w = np.where(sign[:, None] < 0, -128, 127) * np.ones((K, taps), np.int64)
        w[:, 7] -= sign  # -127 / 126: odd group sums
        return x, (8, 0, 4), w.reshape(K, R, R, C), (8, 1, 7), (16, 1, 15)
    # l1: per channel sum |w| = 65793 = 513 * 128 + 63 * 2 + 3, one sign per channel
    mag = np.concatenate([np.full(513, 128), np.full(62, 2), [5]])
    assert mag.sum() == 65793 and mag.size == taps
    w = np.empty((K, taps), np.int64)
    for o in range(K):
        m = rng.permutation(mag)
        w[o] = -m if o % 3 == 0 else np.minimum(m, 127)
    # positive channels cannot reach 128: keep them at 127 (their bound is then lower); the negative
    # channels carry the exact 2^24 - 1 sums
    return x, (8, 0, 4), w.reshape(K, R, R, C), (8, 1, 7), (16, 1, 15)


@pytest.mark.parametrize("kind", ["wordlength", "limbs", "l1"])
@pytest.mark.parametrize("K,mode", [(64, 1), (128, 1), (256, 1), (128, 0)])
def test_conv_exact_at_group_bound(F, kind, K, mode):
    x, tx, w, tw, tb = _edge_case(kind, K)
    fx, fw = F.fmt(*tx), F.fmt(*tw)
    fb = F.fmt(tb[0], 1, tb[1])
    b = np.zeros(K, np.int64)
    b[::5] = 3
    fy = F.fmt(8, 1, -12) if mode == 0 else None
    Cp = x.shape[-1]
    w_l1 = int(np.abs(w).reshape(K, -1).sum(axis=1).max()) if kind == "l1" else 0
    if kind == "l1":
        assert 255 * w_l1 == 2 ** 24 - 1
    got, s = run_conv(F, x, fx, w, fw, b, fb, 1, 0, False, mode, fy, Cp, w_l1)
    want, ws = oracle_conv(x, fx, w, fw, b, fb, 1, 0, False, mode, fy)
    assert s == ws
    assert np.array_equal(got, want)
    if mode == 1:
        acc = oracle.conv2d(x, w, 1, 0)
        if kind == "l1":
            assert np.abs(acc).max() == 2 ** 24 - 1  # the exact edge is reached
        if kind == "wordlength":
            assert np.any(acc % 2 == 1) and np.abs(acc).max() > 2 ** 24  # odd sums; the full reduction exceeds one group


def test_bounded_wait_runs_out_and_the_context_stays_usable(F):
    """A bounded mbarrier wait of the tensor-core kernels given up after a short limit on a barrier that
    nothing arrives on: FXPQ_ERR_TIMEOUT is latched and read once, and a normal launch afterwards is
    bit-exact (no fault, no hang)."""
    from paper_2203_12091_gb300 import _lib as L
    assert F.fxpq_get_device_status() == 0
    assert L.lib().fxpq_selftest_wait_timeout(20000, None) == L.OK
    assert F.fxpq_get_device_status() == L.ERR_TIMEOUT
    assert F.fxpq_get_device_status() == 0  # read once: the word is cleared
    run_case(F, CASES[0])
    run_case(F, CASES[16])  # a patch-tile case on the tensor cores
    assert F.fxpq_get_device_status() == 0


# ----------------------------------------------------------------------------- packed k-bit weights
@pytest.mark.parametrize("k,S", [(1, 0), (1, 1), (2, 1), (3, 1), (4, 0), (5, 1), (7, 1), (8, 1), (8, 0)])
@pytest.mark.parametrize("K,Lw", [(5, 100), (300, 64), (1, 8)])
def test_pack_weights_layout(F, k, S, K, Lw):
    """fxpq_pack_weights: the oracle's k-bit packing (Sec. V-E.2) of the codes rearranged as
    [ceil(L / 64)][K rounded up to 256][64], zero past L and past K, each 256-channel tile's words
    plane-major."""
    rng = np.random.default_rng(100 * k + K + Lw + S)
    c = rand_codes(rng, (K, Lw), k, S)
    fw = F.fmt(k, S, 3)
    packed = F.pack_weights(torch.from_numpy(c.astype(np.float16)).cuda(), fw, K, Lw)
    n_kb, K_pad = (Lw + 63) // 64, (K + 255) // 256 * 256
    r = np.zeros((n_kb, K_pad, 64), np.int64)
    for kb in range(n_kb):
        seg = c[:, 64 * kb:64 * kb + 64]
        r[kb, :K, :seg.shape[1]] = seg
    # pack_codes' records (kb, o, h) of k words, then each 256-channel tile's words plane-major
    want = oracle.pack_codes(r, k).reshape(n_kb, K_pad // 256, 256, 2, k).transpose(0, 1, 4, 2, 3).reshape(-1)
    assert packed.numel() == F.fxpq_packed_weights_bytes(fw, K, Lw) == want.size * 4
    assert np.array_equal(packed.cpu().numpy().view(np.uint32), want)


PACKED_CASES = [
    # N, H, C, K, R, (kx,Sx,flx), (kb,flb) or None, relu, mode, (ky,Sy,fly), packed records read: FC layers
    # (R = H, pad 0) and 1x1 layers; every weight wordlength runs on each
    (3, 7, 64, 304, 7, (8, 0, 4), (16, 15), True, 0, (8, 0, 3), True),      # FC, ragged K, split reduction
    (64, 1, 1024, 512, 1, (5, 0, 2), (16, 12), True, 0, (8, 0, 3), True),   # FC at batch 64
    (2, 9, 64, 272, 1, (8, 0, 4), (16, 15), False, 0, (8, 1, 3), True),     # 1x1, two row tiles, signed out
    (3, 1, 40, 264, 1, (7, 0, 3), None, True, 2, None, True),               # reduction of 40: a partial k-block
    (2, 3, 128, 136, 3, (6, 0, 2), (16, 10), False, 1, None, True),         # FC over a 3x3 map, int64 sums out
    (64, 18, 64, 256, 1, (8, 0, 4), (16, 15), True, 0, (8, 0, 3), False),   # 1x1, enough tiles: fp16 codes read
]
# (the C-Block takes weights of 2..16 bits: 1-bit codes exist only as stored tensors)
PACKED_W = [(2, 1, 2), (2, 0, 1), (3, 1, 3), (4, 1, 5), (4, 0, 4), (5, 1, 6), (6, 1, 7), (7, 1, 8), (8, 1, 9),
            (8, 0, 8)]


@pytest.mark.parametrize("tw", PACKED_W)
@pytest.mark.parametrize("case", PACKED_CASES)
def test_conv_packed_weights(F, case, tw):
    """FC and 1x1 layers with packed k-bit weights (k = 2..8): bit-exact against the oracle and equal to
    the layer reading fp16 codes.  Then the packed records of a weight tensor with one channel changed go
    with the original fp16 codes: where the tensor-core path reads the records (layers split across
    the SMs, on every path but tc_rows and simt) the output follows the changed codes, which shows the
    kernel consumed them; elsewhere it follows the fp16 codes."""
    N, H, C, K, R, tx, tb, relu, mode, ty, reads_packed = case
    rng = np.random.default_rng(H * 7 + K + tw[0] * 31 + tw[1])
    fx, fw = F.fmt(*tx), F.fmt(*tw)
    fb = F.fmt(tb[0], 1, tb[1]) if tb else None
    fy = F.fmt(*ty) if ty else None
    x = rand_codes(rng, (N, H, H, C), tx[0], tx[1])
    w = rand_codes(rng, (K, R, R, C), tw[0], tw[1])
    b = rand_codes(rng, (K,), tb[0], 1) if tb else None
    Cp = (C + 7) // 8 * 8
    w_l1 = int(np.abs(w).reshape(K, -1).sum(axis=1).max())
    want, ws = oracle_conv(x, fx, w, fw, b, fb, 1, 0, relu, mode, fy)
    got, s = run_conv(F, x, fx, w, fw, b, fb, 1, 0, relu, mode, fy, Cp, w_l1, packed_w=w)
    assert s == ws
    assert np.array_equal(got, want)
    # output channel K-1 set to the largest (else the smallest) code in the packed copy only (the L1
    # bound passed covers both tensors): its outputs change, and they follow the packed copy wherever
    # the kernel reads it
    for code in (oracle.qmax(tw[0], tw[1]), oracle.qmin(tw[0], tw[1])):
        w2 = w.copy()
        w2[K - 1] = code
        want2, _ = oracle_conv(x, fx, w2, fw, b, fb, 1, 0, relu, mode, fy)
        if not np.array_equal(want2, want):
            break
    assert not np.array_equal(want2, want)
    w_l1_2 = max(w_l1, int(np.abs(w2).reshape(K, -1).sum(axis=1).max()))
    got2, _ = run_conv(F, x, fx, w, fw, b, fb, 1, 0, relu, mode, fy, Cp, w_l1_2, packed_w=w2)
    if os.environ.get("FXPQ_CONV_PATH") in ("tc_rows", "simt") or not reads_packed:
        assert np.array_equal(got2, want)
    else:
        assert np.array_equal(got2, want2)
