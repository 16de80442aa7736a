"""CPU oracle for the dynamic fixed-point network-evaluation path of FxP-QNet
(Shawahna et al., IEEE Access 2022, arXiv 2203.12091).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  It shares no code with the CUDA library (``paper_2203_12091_gb300``)
and never imports it; the two meet only through the seeded generators in
``synth``, which hold none of the method's arithmetic.

Everything here is the paper's definition written out plainly:

* Q (Sec. IV-B, Eq. fp_k_bit_quantization / clip / quantization_levels):
  ``code = clip(round_half_even(x * 2^FL), Qmin, Qmax)``.
* L (Sec. IV-C, Eq. DSB_QE): ``sum (x - code * 2^-FL)^2``, summed exactly and
  rounded once (C core, Kulisch accumulator).
* FL search: L for every candidate (k, FL), argmin per k, exact ties to the
  smallest FL (Alg. 1 only moves on a strict improvement).
* Initial QPs (Sec. IV-A.3, Eq. initial_quantization_parameters).
* C-Block arithmetic (Sec. IV-B, the C-Block paragraph and its figure):
  exact integer MAC, bias aligned by a left shift of delta = FL_a + FL_w - FL_b,
  ReLU, then the FxP-QLayer's right shift with round-half-even and clip.
* MAX-POOL without a QLayer, AVG-POOL with the reciprocal quantized like a
  parameter, Eltwise add with FL alignment (Sec. IV-A.2).
* Scale layer (BN rewritten as aleph1 * A + aleph2, Sec. IV-A.1) in the C-Block.
* Memory model MFP / RW_R / RO_R / COMP (Sec. V-E.2) and the packed k-bit code
  storage whose footprint it counts.

Parity status of every function is pinned by ``tests/test_oracle_pins.py``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from fractions import Fraction

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fxpq_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the C core with gcc (plain -O2, OpenMP across independent outer loops only)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _L():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        f32p = ctypes.POINTER(ctypes.c_float)
        i32p = ctypes.POINTER(ctypes.c_int32)
        i64p = ctypes.POINTER(ctypes.c_int64)
        f64p = ctypes.POINTER(ctypes.c_double)
        I, L = ctypes.c_int, ctypes.c_int64
        lib.ora_quantize.argtypes = [f32p, L, I, I, I, i32p]
        lib.ora_quantize.restype = None
        lib.ora_l2_error.argtypes = [f32p, L, I, I, I]
        lib.ora_l2_error.restype = ctypes.c_double
        lib.ora_exact_sum.argtypes = [f64p, L]
        lib.ora_exact_sum.restype = ctypes.c_double
        lib.ora_l1_error.argtypes = [f32p, L, I, I, I]
        lib.ora_l1_error.restype = ctypes.c_double
        lib.ora_fl_search.argtypes = [f32p, L, I, I, I, I, I, f64p, i32p, f64p, I]
        lib.ora_fl_search.restype = I
        lib.ora_conv2d.argtypes = [i32p, I, I, I, I, i32p, I, I, I, I, I, I, I, i64p]
        lib.ora_conv2d.restype = None
        _lib = lib
    return _lib


def _p(a, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


# --------------------------------------------------------------------------
# Quantizer (Sec. IV-B)
# --------------------------------------------------------------------------
def qmin(k: int, S: int) -> int:
    """Eq. (quantization_levels): Qmin = -S * 2^(k-S)."""
    return -S * (1 << (k - S))


def qmax(k: int, S: int) -> int:
    """Eq. (quantization_levels): Qmax = 2^(k-S) - 1."""
    return (1 << (k - S)) - 1


def quantize(x, k: int, S: int, fl: int) -> np.ndarray:
    """Eq. (fp_k_bit_quantization): codes of fp32 ``x`` in S(alpha, FL) / U(alpha, FL), k = alpha + FL.
    k = 1 with S = 1 is the binary quantizer of Eq. (fp_1_bit_quantization): -1 for x < 0, else 0."""
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    out = np.empty(x.size, dtype=np.int32)
    _L().ora_quantize(_p(x, ctypes.c_float), x.size, k, S, fl, _p(out, ctypes.c_int32))
    return out.astype(np.int64)


def value(codes, k: int, S: int, fl: int) -> np.ndarray:
    """The values codes stand for (fp64, exact): code * 2^-FL, or for the binary quantizer (k = 1,
    S = 1) the decoded sign, 0 -> +1 and -1 -> -1, times 2^-FL (Eq. fp_1_bit_quantization)."""
    c = np.asarray(codes, dtype=np.int64)
    if k == 1 and S == 1:
        c = 2 * c + 1
    return np.ldexp(c.astype(np.float64), -fl)


def l2_error(x, k: int, S: int, fl: int) -> float:
    """Eq. (DSB_QE): ||X - X~||_2^2, exact sum rounded once to a double."""
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    return float(_L().ora_l2_error(_p(x, ctypes.c_float), x.size, k, S, fl))


def l1_error(x, k: int, S: int, fl: int) -> float:
    """Eq. (MAE) as a sum: sum |X - X~| (the MAE is this over N), exact sum rounded once."""
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    return float(_L().ora_l1_error(_p(x, ctypes.c_float), x.size, k, S, fl))


def exact_sum(v) -> float:
    v = np.ascontiguousarray(v, dtype=np.float64).reshape(-1)
    return float(_L().ora_exact_sum(_p(v, ctypes.c_double), v.size))


def fl_search(x, S: int, k_lo: int, k_hi: int, fl_lo: int, fl_hi: int, score: str = "l2"):
    """Score every (k, FL) candidate by Eq. (DSB_QE) (score "l2") or by the L1 error of Eq. (MAE) as a
    sum (score "l1"); argmin FL per k (ties -> smallest FL).

    S = -1 selects the sign strategy of Sec. IV-A.3 (S = 1 iff min(X) < 0).
    Returns (err[nk, nfl] float64, best_fl[nk] int32, S_used, stats dict).
    """
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    nk, nfl = k_hi - k_lo + 1, fl_hi - fl_lo + 1
    err = np.empty(nk * nfl, dtype=np.float64)
    best = np.empty(nk, dtype=np.int32)
    st = np.empty(4, dtype=np.float64)
    s_used = _L().ora_fl_search(_p(x, ctypes.c_float), x.size, S, k_lo, k_hi, fl_lo, fl_hi,
                                _p(err, ctypes.c_double), _p(best, ctypes.c_int32), _p(st, ctypes.c_double),
                                {"l2": 0, "l1": 1}[score])
    stats = {"min": st[0], "max": st[1], "sum": st[2], "sumsq": st[3], "n": x.size}
    return err.reshape(nk, nfl), best, int(s_used), stats


def fl_init(xmin: float, xmax: float, k: int, strategy: str):
    """Initial QPs (Sec. IV-A.3): sign strategy, scalar psi, beta_hat = -log2(psi) and
    beta = floor / round / ceil for the conservative / neutral / aggressive strategy.

    Reading: where one of the two candidates of the signed psi is not positive it is
    dropped (the printed min() assumes both are positive).  Round is half-to-even.
    Returns (S, beta, alpha) with alpha = k - beta (k = alpha + beta, Sec. II-A).
    """
    S = 1 if xmin < 0 else 0
    if S == 0:
        psi = xmax / (2.0 ** k - 1.0)
        cands = [psi] if psi > 0 else []
    else:
        cands = [c for c in (xmin / -(2.0 ** (k - 1)), xmax / (2.0 ** (k - 1) - 1.0)) if c > 0]
    if not cands:
        raise ValueError("fl_init: data-structure has no positive scale")
    psi = min(cands)
    beta_hat = -np.log2(psi)
    if strategy == "conservative":
        beta = int(np.floor(beta_hat))
    elif strategy == "neutral":
        beta = int(np.round(beta_hat))  # numpy rounds halves to even
    elif strategy == "aggressive":
        beta = int(np.ceil(beta_hat))
    else:
        raise ValueError(strategy)
    return S, beta, k - beta


# --------------------------------------------------------------------------
# Integer C-Block arithmetic (Sec. IV-B)
# --------------------------------------------------------------------------
def conv2d(x_nhwc, w_krsc, stride: int, pad: int) -> np.ndarray:
    """Exact int64 MAC of codes: acc[n,p,q,k] = sum_{r,s,c} x[n, p*st+r-pad, q*st+s-pad, c] * w[k,r,s,c]."""
    x = np.ascontiguousarray(x_nhwc, dtype=np.int32)
    w = np.ascontiguousarray(w_krsc, dtype=np.int32)
    N, H, W, C = x.shape
    K, R, S, C2 = w.shape
    assert C == C2
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    acc = np.empty((N, P, Q, K), dtype=np.int64)
    _L().ora_conv2d(_p(x, ctypes.c_int32), N, H, W, C, _p(w, ctypes.c_int32), K, R, S, stride, pad, P, Q,
                    _p(acc, ctypes.c_int64))
    return acc


def fc(x_nc, w_kc) -> np.ndarray:
    """FC layer = 1x1 convolution over a 1x1 map."""
    x = np.asarray(x_nc)
    N, C = x.shape
    w = np.asarray(w_kc)
    return conv2d(x.reshape(N, 1, 1, C), w.reshape(w.shape[0], 1, 1, C), 1, 0).reshape(N, -1)


def rne_shift(v, sh: int) -> np.ndarray:
    """round(v / 2^sh) with halves to even, sh >= 1, exact in int64."""
    v = np.asarray(v, dtype=np.int64)
    q = v >> sh  # floor division (arithmetic shift)
    rem = v - (q << sh)
    half = np.int64(1) << np.int64(sh - 1)
    up = (rem > half) | ((rem == half) & ((q & 1) == 1))
    return q + up.astype(np.int64)


def _check_range(v, bits: int):
    m = int(np.max(np.abs(v))) if np.size(v) else 0
    assert m < (1 << bits), f"integer range exceeded ({m} >= 2^{bits})"


def requant(acc, s_acc: int, k: int, S: int, fl_out: int) -> np.ndarray:
    """FxP-QLayer (Sec. IV-B): shift the value acc * 2^-s_acc to FL_out, rounding half to even
    on the dropped bits, then clip to [Qmin, Qmax]."""
    acc = np.asarray(acc, dtype=np.int64)
    sh = s_acc - fl_out
    if sh > 0:
        q = rne_shift(acc, sh)
    else:
        _check_range(acc, 62 + sh)
        q = acc << np.int64(-sh)
    return np.clip(q, qmin(k, S), qmax(k, S))


def add_bias(acc, s_acc: int, bias, fl_b: int):
    """Bias alignment (Sec. IV-B): delta = s_acc - FL_b; B is shifted left by delta.
    Reading for delta < 0: the accumulator is shifted left instead (no bits dropped)."""
    acc = np.asarray(acc, dtype=np.int64)
    b = np.asarray(bias, dtype=np.int64)
    d = s_acc - fl_b
    if d >= 0:
        _check_range(b, 62 - d)
        return acc + (b << np.int64(d)), s_acc
    _check_range(acc, 62 + d)
    return (acc << np.int64(-d)) + b, fl_b


def scale_layer(v, s_v: int, scale, fl_scale: int, shift, fl_shift: int):
    """Scale layer on integers (Sec. IV-A.1, Eq. BatchNorm: BN(A) = aleph1 * A + aleph2, with aleph1 and
    aleph2 quantized like weights and biases; Sec. IV-B: an integer multiplier and accumulator).  The
    per-channel (last axis) product aleph1_code * v has scale s_v + FL_aleph1; aleph2 is aligned to it
    like a bias (add_bias, with the same reading when its FL is finer).  Returns (value, scale)."""
    v = np.asarray(v, dtype=np.int64)
    m = np.asarray(scale, dtype=np.int64)
    _check_range(v, 62 - int(np.max(np.abs(m), initial=0)).bit_length())
    p = v * m
    s_p = s_v + fl_scale
    if shift is None:
        return p, s_p
    return add_bias(p, s_p, shift, fl_shift)


def cblock(acc, s_acc: int, bias, fl_b, relu: bool, scale=None, fl_scale: int = 0, shift=None, fl_shift: int = 0):
    """C-Block output before its FxP-QLayer: MAC result + aligned bias, the optional Scale layer
    (CONV-Scale-ReLU, Sec. IV-B), then ReLU.  Returns (int64 value, its scale exponent)."""
    if bias is not None:
        acc, s_acc = add_bias(acc, s_acc, bias, fl_b)
    if scale is not None:
        acc, s_acc = scale_layer(acc, s_acc, scale, fl_scale, shift, fl_shift)
    if relu:
        acc = np.maximum(acc, 0)
    return acc, s_acc


def bn_to_scale(gamma, beta, mean, var, eps=1e-5):
    """Preprocessor (Sec. IV-A.1, Eq. BatchNorm_s1_s2): a BN layer becomes a Scale layer with
    aleph1 = gamma / sqrt(var + eps) and aleph2 = beta - gamma * mean / sqrt(var + eps), in fp32 in that
    order of operations."""
    g, b, mu, v = (np.asarray(t, dtype=np.float32) for t in (gamma, beta, mean, var))
    r = np.sqrt(v + np.float32(eps))
    a1 = (g / r).astype(np.float32)
    a2 = (b - (g * mu) / r).astype(np.float32)
    return a1, a2


def maxpool(x_nhwc, k: int, stride: int, pad: int) -> np.ndarray:
    """MAX-POOL on codes; taps outside the map are ignored; no QLayer follows (Sec. IV-A.2)."""
    x = np.asarray(x_nhwc, dtype=np.int64)
    N, H, W, C = x.shape
    P = (H + 2 * pad - k) // stride + 1
    Q = (W + 2 * pad - k) // stride + 1
    out = np.full((N, P, Q, C), np.iinfo(np.int64).min, dtype=np.int64)
    for r in range(k):
        for s in range(k):
            for p in range(P):
                h = p * stride + r - pad
                if h < 0 or h >= H:
                    continue
                for q in range(Q):
                    w = q * stride + s - pad
                    if w < 0 or w >= W:
                        continue
                    out[:, p, q, :] = np.maximum(out[:, p, q, :], x[:, h, w, :])
    return out


def eltwise_add(a, fl_a: int, b, fl_b: int, relu: bool):
    """Eltwise C-Block: both inputs aligned to the finer scale max(FL_a, FL_b) by an exact
    left shift, added, optional ReLU.  Returns (int64 value, its scale exponent)."""
    fl = max(fl_a, fl_b)
    a = np.asarray(a, dtype=np.int64) << np.int64(fl - fl_a)
    b = np.asarray(b, dtype=np.int64) << np.int64(fl - fl_b)
    v = a + b
    if relu:
        v = np.maximum(v, 0)
    return v, fl


def avgpool_global(x_nhwc, fl_x: int, recip_code: int, fl_r: int):
    """AVG-POOL over the whole map: sum of codes times the quantized reciprocal of the
    patch size (handled like a parameter, Sec. IV-A.2).  Returns (int64 [N, C], scale)."""
    x = np.asarray(x_nhwc, dtype=np.int64)
    s = x.sum(axis=(1, 2))
    return s * np.int64(recip_code), fl_x + fl_r


def to_f32(v, s: int) -> np.ndarray:
    """fp32 nearest-even image of the exact value v * 2^-s (|v| < 2^53)."""
    v = np.asarray(v, dtype=np.int64)
    _check_range(v, 53)
    return (v.astype(np.float64) * (2.0 ** -s)).astype(np.float32)


# --------------------------------------------------------------------------
# Memory model and packed code storage (Sec. V-E.2, Eq. mfp, RW_R, RO_R, compression)
# --------------------------------------------------------------------------
def mfp(nu: int, k) -> float:
    """Memory footprint in MB of a data-structure of nu elements at k bits (k = 32 for FP32)."""
    return nu * k / 2.0 ** 23


def rw_r(layers, act_elems, act_bits) -> float:
    """Read-write requirement: the largest, over layers l, of the footprints of l's input activations
    (every layer feeding it; the network input for the first) plus l's own output activations.
    act_elems / act_bits: name -> elements per image / bits ("input" included)."""
    best = 0.0
    prev = "input"
    for L in layers:
        if L["type"] == "eltwise":
            inputs = [L["a"], L["b"]]
        else:
            inputs = [L.get("src") or prev]
        v = sum(mfp(act_elems[i], act_bits[i]) for i in inputs) + mfp(act_elems[L["name"]], act_bits[L["name"]])
        best = max(best, v)
        prev = L["name"]
    return best


def ro_r(params) -> float:
    """Read-only requirement: the sum of the footprints of every layer's parameters.
    params: list of (elements, bits) pairs (weights and biases of each layer with parameters)."""
    return sum(mfp(nu, k) for nu, k in params)


def pack_codes(codes, k: int) -> np.ndarray:
    """Packed storage of k-bit codes (1 <= k <= 16), k bits per code: the codes are taken in groups of 32
    (the last group zero-padded) and group g occupies k uint32 words, word g*k + b holding bit b of the
    k-bit two's-complement field of code 32g + i at bit i."""
    c = np.asarray(codes, dtype=np.int64).reshape(-1)
    ng = (c.size + 31) // 32
    out = np.zeros(ng * k, dtype=np.uint32)
    for e in range(c.size):
        field = int(c[e]) & ((1 << k) - 1)
        g, i = divmod(e, 32)
        for b in range(k):
            if (field >> b) & 1:
                out[g * k + b] |= np.uint32(1 << i)
    return out


def unpack_codes(words, n: int, k: int, S: int) -> np.ndarray:
    """Inverse of pack_codes: n codes, sign-extended from k bits when S = 1."""
    w = np.asarray(words, dtype=np.uint32)
    out = np.zeros(n, dtype=np.int64)
    for e in range(n):
        g, i = divmod(e, 32)
        field = 0
        for b in range(k):
            field |= ((int(w[g * k + b]) >> i) & 1) << b
        if S and field >= 1 << (k - 1):
            field -= 1 << k
        out[e] = field
    return out


# --------------------------------------------------------------------------
# Exact rational helpers used only by the pins (Python Fractions)
# --------------------------------------------------------------------------
def frac_round_half_even(y: Fraction) -> int:
    f = y.numerator // y.denominator
    d = y - f
    if d > Fraction(1, 2):
        return f + 1
    if d < Fraction(1, 2):
        return f
    return f if f % 2 == 0 else f + 1
