"""The C-Block epilogue arithmetic of the kernels, run on the CPU against the oracle.

`tests/epilogue_host.cu` plans each case with the library's host planner and evaluates the kernels'
inline epilogue functions (generic 64-bit, 32-bit CUDA-core, 32-bit and 64-bit tensor-core) on the
host; every code they produce must equal the oracle's C-Block value (Sec. IV-B: bias alignment, Scale
layer, ReLU) passed through its FxP-QLayer.  Random formats and values, plus targeted ties, biases
finer than the accumulator, large and small shifts, negative Scale gains and saturation.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "epilogue_host.cu")
BIN = os.path.join(ROOT, "tests", "_build", "epilogue_host")
NA = -(2 ** 31)


def _harness():
    from paper_2203_12091_gb300 import build as B
    if not shutil.which(B.nvcc()) and not os.path.exists(B.nvcc()):
        pytest.skip("nvcc not available")
    B.build()
    objs = sorted(os.path.join(B.BUILD, f) for f in os.listdir(B.BUILD) if f.endswith(".o"))
    deps = [SRC] + objs + [os.path.join(B.CSRC, f) for f in os.listdir(B.CSRC) if f.endswith(".cuh")]
    if not os.path.exists(BIN) or any(os.path.getmtime(d) > os.path.getmtime(BIN) for d in deps):
        os.makedirs(os.path.dirname(BIN), exist_ok=True)
        cmd = [B.nvcc(), *B.ARCH, "-O2", "-std=c++17", "--expt-relaxed-constexpr", f"-I{B.INCLUDE}", f"-I{B.CSRC}",
               SRC, *objs, "-o", BIN + ".tmp"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stdout + r.stderr
        os.replace(BIN + ".tmp", BIN)
    return BIN


def _scale_of(c):
    """Scale exponent of the value entering the FxP-QLayer, and its right shift (the oracle's rules)."""
    s = c["xfl"] + c["wfl"]
    if c["has_bias"] and s - c["bfl"] < 0:
        s = c["bfl"]
    if c["has_scale"]:
        s += c["sfl"]
        if s - c["hfl"] < 0:
            s = c["hfl"]
    return s, s - c["yfl"]


def _expected(c):
    acc = np.array([c["acc"]], dtype=np.int64)
    kw = {}
    if c["has_scale"]:
        kw = dict(scale=np.array([c["m"]]), fl_scale=c["sfl"], shift=np.array([c["h"]]), fl_shift=c["hfl"])
    v, s = oracle.cblock(acc, c["xfl"] + c["wfl"], np.array([c["bias"]]) if c["has_bias"] else None, c["bfl"],
                         bool(c["relu"]), **kw)
    return int(oracle.requant(v, s, c["yb"], c["ys"], c["yfl"])[0])


def _cases(n, seed):
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        xb, wb = int(rng.integers(2, 17)), int(rng.integers(2, 17))
        xs, ws = int(rng.integers(0, 2)), 1
        c = dict(xb=xb, xs=xs, xfl=int(rng.integers(-4, 16)), wb=wb, ws=ws, wfl=int(rng.integers(-2, 16)),
                 bb=int(rng.choice([8, 16, 32])), bs=1, bfl=int(rng.integers(-4, 36)),
                 yb=int(rng.integers(2, 17)), ys=int(rng.integers(0, 2)), yfl=int(rng.integers(-6, 20)),
                 relu=int(rng.integers(0, 2)), has_bias=int(rng.random() < 0.8), C=int(rng.choice([3, 8, 64, 576, 4608])),
                 w_l1=0, has_scale=int(rng.random() < 0.25), sb=16, ss=1, sfl=int(rng.integers(0, 16)),
                 hb=16, hs=1, hfl=int(rng.integers(0, 24)))
        bound = (2 ** (xb - xs)) * (2 ** (wb - ws)) * c["C"]
        bmax = 2 ** (c["bb"] - 1) - 1
        c["bias"] = int(rng.integers(-bmax, bmax + 1)) if rng.random() < 0.7 else int(rng.integers(-64, 65))
        c["m"] = int(rng.integers(-2 ** 15, 2 ** 15)) if rng.random() < 0.7 else int(rng.choice([-1, 1, 2, -3]))
        c["h"] = int(rng.integers(-2 ** 15, 2 ** 15))
        mode = rng.random()
        if mode < 0.4:
            acc = int(rng.integers(-bound, bound + 1))
        elif mode < 0.7:
            acc = int(rng.integers(-1000, 1001))
        else:
            # a tie of the FxP-QLayer's rounding (without bias and Scale the value is acc itself)
            c["has_bias"] = 0
            c["has_scale"] = 0
            _, sh = _scale_of(c)
            if sh < 1:
                acc = int(rng.integers(-bound, bound + 1))
            else:
                q = int(rng.integers(-64, 65))
                acc = (2 * q + 1) * (1 << (sh - 1))
                if abs(acc) > bound:
                    acc = int(rng.integers(-bound, bound + 1))
        c["acc"] = acc
        out.append(c)
    return out


ORDER = ["xb", "xs", "xfl", "wb", "ws", "wfl", "bb", "bs", "bfl", "yb", "ys", "yfl", "relu", "has_bias", "C",
         "w_l1", "acc", "bias", "has_scale", "sb", "ss", "sfl", "hb", "hs", "hfl", "m", "h"]


def _run(cases):
    exe = _harness()
    text = "\n".join(" ".join(str(c[k]) for k in ORDER) for c in cases) + "\n"
    r = subprocess.run([exe], input=text, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    rows = [list(map(int, line.split())) for line in r.stdout.strip().splitlines()]
    assert len(rows) == len(cases)
    return rows


def test_epilogue_paths_match_the_oracle():
    cases = _cases(6000, 11)
    rows = _run(cases)
    used = {"generic": 0, "code32": 0, "epi32": 0, "epi64": 0, "ties": 0}
    planned = 0
    for c, (st, v32, sh, generic, code32, epi32, epi64) in zip(cases, rows):
        if st != 0:
            continue  # the planner refused the layer's integer ranges (FXPQ_ERR_RANGE): nothing runs
        planned += 1
        want = _expected(c)
        for name, got in (("generic", generic), ("code32", code32), ("epi32", epi32), ("epi64", epi64)):
            if got != NA:
                used[name] += 1
                assert got == want, (name, c, got, want)
        _, sh_o = _scale_of(c)
        assert sh == sh_o, (c, sh, sh_o)
        if not c["has_bias"] and not c["has_scale"] and sh >= 1 and c["acc"] % (1 << sh) == 1 << (sh - 1):
            used["ties"] += 1
    assert planned > 4000
    # every path and the ties were exercised
    assert min(used.values()) > 200, used


def test_epilogue_edge_cases():
    base = dict(xb=8, xs=0, xfl=4, wb=8, ws=1, wfl=8, bb=16, bs=1, bfl=20, yb=8, ys=0, yfl=5, relu=1, has_bias=1,
                C=64, w_l1=0, acc=0, bias=0, has_scale=0, sb=16, ss=1, sfl=12, hb=16, hs=1, hfl=14, m=1, h=0)
    cases = []
    for acc in (0, 1, -1, 255 * 127 * 64, -255 * 128 * 64, 12345, -12345):
        for bias in (0, 1, -1, 32767, -32768, 255, -256):
            for relu in (0, 1):
                for yb, ys in ((8, 0), (8, 1), (16, 1), (2, 1)):
                    cases.append(dict(base, acc=acc, bias=bias, relu=relu, yb=yb, ys=ys))
    # shifts from 1 up to the 62-bit limit, bias finer and coarser than the accumulator
    for yfl in (-20, -10, 0, 11, 19):
        for bfl in (0, 8, 12, 30):
            cases.append(dict(base, yfl=yfl, bfl=bfl, acc=777777, bias=-12345))
    # Scale layers: gains of both signs, shifts finer and coarser than the product
    for m in (-1, 1, -32768, 32767):
        for hfl in (0, 20, 30):
            cases.append(dict(base, has_scale=1, m=m, hfl=hfl, acc=-54321, bias=999, h=-777))
    rows = _run(cases)
    for c, (st, v32, sh, generic, code32, epi32, epi64) in zip(cases, rows):
        if st != 0:
            continue
        want = _expected(c)
        for got in (generic, code32, epi32, epi64):
            assert got == NA or got == want, (c, got, want)
