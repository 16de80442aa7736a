"""C ABI checks that need no GPU: the library builds and loads, exports exactly what
include/fxpq.h declares, and its host-side validation and host-only helpers behave."""
import ctypes
import os
import re

import pytest

import oracle
from paper_2203_12091_gb300 import _lib as L
from paper_2203_12091_gb300 import build as B

HDR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "fxpq.h")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return L.lib()


def declared():
    src = open(HDR).read()
    return sorted(set(re.findall(r"FXPQ_API\s+[\w\s\*]*?\b(fxpq_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared()
    for must in ("fxpq_fl_search", "fxpq_quantize", "fxpq_conv_fwd", "fxpq_gemm", "fxpq_net_forward"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB], capture_output=True, text=True).stdout
    exported = set(re.findall(r"\sT\s(fxpq_\w+)", out))
    assert set(declared()) <= exported
    assert set(declared()) == set(L.declared_symbols())
    for n in declared():
        assert hasattr(lib, n)


def test_host_validation_rejects_bad_arguments(lib):
    f8 = L.Fmt(8, 1, 4)
    assert lib.fxpq_quantize(None, -1, f8, L.DT_I8, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_quantize(None, 4, L.Fmt(1, 1, 0), L.DT_I8, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_quantize(None, 4, L.Fmt(8, 1, 41), L.DT_I8, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_quantize(ctypes.c_void_p(256), 4, L.Fmt(9, 1, 0), L.DT_I8, ctypes.c_void_p(256), None) == L.ERR_INVALID_ARG
    assert lib.fxpq_quantize(ctypes.c_void_p(256), 4, L.Fmt(8, 0, 0), L.DT_I8, ctypes.c_void_p(256), None) == L.ERR_INVALID_ARG
    p = ctypes.c_void_p(256)
    ws = lib.fxpq_fl_search_workspace(100)
    assert ws > 0 and ws % 256 == 0
    # k out of range, FL span too wide, missing outputs, workspace too small / misaligned
    assert lib.fxpq_fl_search(p, 100, -1, 0, 8, 0, 10, p, p, None, p, ws, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search(p, 100, -1, 2, 17, 0, 10, p, p, None, p, ws, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search(p, 100, -1, 2, 8, -8, 24, p, p, None, p, ws, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search(p, 100, 2, 2, 8, 0, 10, p, p, None, p, ws, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search(p, 100, -1, 2, 8, 0, 10, None, p, None, p, ws, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_fl_search(p, 100, -1, 2, 8, 0, 10, p, p, None, p, ws - 1, None) == L.ERR_WORKSPACE
    assert lib.fxpq_fl_search(p, 100, -1, 2, 8, 0, 10, p, p, None, ctypes.c_void_p(258), ws, None) == L.ERR_WORKSPACE
    assert lib.fxpq_fl_search(p, 100, -1, 2, 8, 0, 10, p, p, None, None, ws, None) == L.ERR_WORKSPACE
    # conv: misaligned pointers, bad geometry, integer range
    d = L.ConvDesc(1, 8, 8, 8, 8, 8, 3, 3, 1, 1, 1, L.OUT_CODES, f8, f8, L.Fmt(16, 1, 8), f8)
    sc = L.I32()
    assert lib.fxpq_conv_fwd(ctypes.byref(d), ctypes.c_void_p(258), p, None, p, ctypes.byref(sc), None, 0, None) == L.ERR_INVALID_ARG
    d.Cp = 12
    assert lib.fxpq_conv_fwd(ctypes.byref(d), p, p, None, p, ctypes.byref(sc), None, 0, None) == L.ERR_INVALID_ARG
    d.Cp, d.K = 8, 12
    assert lib.fxpq_conv_fwd(ctypes.byref(d), p, p, None, p, ctypes.byref(sc), None, 0, None) == L.ERR_INVALID_ARG
    d.K = 8
    d.fmt_b = L.Fmt(32, 1, -30)  # delta = 8 - (-30) = 38: B << 38 of a 32-bit bias leaves int64
    assert lib.fxpq_conv_fwd(ctypes.byref(d), p, p, p, p, ctypes.byref(sc), None, 0, None) == L.ERR_RANGE
    assert lib.fxpq_maxpool(p, 1, 4, 4, 8, f8, 3, 2, 3, p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_eltwise(p, f8, p, L.Fmt(8, 1, 60), 4, 8, 0, 0, f8, p, None, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_avgpool(p, 1, 7, 7, 8, f8, 70000, L.Fmt(16, 0, 21), 0, f8, p, None, None) == L.ERR_INVALID_ARG


def test_net_planning_rejects_malformed_graphs(lib):
    ops = (L.OpDesc * 1)()
    ops[0].op = L.OP_MAXPOOL
    ops[0].last = 1
    net = L.Net(1, 2, 3, 8, 8, 8, L.Fmt(8, 1, 4), ctypes.cast(ops, ctypes.POINTER(L.OpDesc)))
    assert lib.fxpq_net_workspace(ctypes.byref(net), 4) == 0  # last op must be a conv
    ops[0].op = L.OP_CONV
    ops[0].K, ops[0].R, ops[0].S, ops[0].stride = 8, 3, 3, 1
    ops[0].d_w = 256
    assert lib.fxpq_net_workspace(ctypes.byref(net), 4) > 0
    ops[0].src0 = 1  # undefined source slot
    assert lib.fxpq_net_workspace(ctypes.byref(net), 4) == 0


@pytest.mark.parametrize("mn,mx,k", [(0.0, 1.0, 8), (-2.0, 1.0, 8), (-0.5, 0.5, 8), (0.0, 3.7, 4), (-1e-3, 2e-3, 16),
                                     (-5.0, -1.0, 6), (0.0, 1e-4, 8)])
def test_fl_init_matches_oracle(lib, mn, mx, k):
    for strat, name in enumerate(("conservative", "neutral", "aggressive")):
        st = L.Stats(mn, mx, 0, 0, 0.0, 0.0, 1)
        out = L.Fmt()
        code = lib.fxpq_fl_init(ctypes.byref(st), k, strat, ctypes.byref(out))
        try:
            S, beta, _ = oracle.fl_init(float(st.min), float(st.max), k, name)
        except ValueError:
            assert code == L.ERR_INVALID_ARG
            continue
        assert code == L.OK and (out.is_signed, out.fl, out.bits) == (S, beta, k)


def test_status_strings(lib):
    for c in range(8):
        assert lib.fxpq_status_string(c)
    assert lib.fxpq_launch_count() >= 0


def test_struct_layout_matches_header(tmp_path):
    """Every ctypes mirror of a header struct has the C compiler's size and field offsets."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no host C compiler")
    mirrors = {"fxpq_fmt": L.Fmt, "fxpq_stats": L.Stats, "fxpq_fl_search_item": L.FlSearchItem,
               "fxpq_quantize_item": L.QuantizeItem, "fxpq_conv_desc": L.ConvDesc, "fxpq_op_desc": L.OpDesc,
               "fxpq_conv_f32_desc": L.ConvF32Desc,
               "fxpq_net": L.Net}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "fxpq.h"', "int main(void) {"]
    for cname, py in mirrors.items():
        lines.append(f'printf("{cname} sizeof %zu\\n", sizeof({cname}));')
        for f, _ in py._fields_:
            lines.append(f'printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));')
    lines += ["return 0; }"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.dirname(HDR), str(src), "-o", str(exe)], check=True)
    got = {}
    for ln in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.splitlines():
        c, f, v = ln.split()
        got[(c, f)] = int(v)
    for cname, py in mirrors.items():
        assert got[(cname, "sizeof")] == ctypes.sizeof(py), cname
        for f, _ in py._fields_:
            assert got[(cname, f)] == getattr(py, f).offset, (cname, f)


@pytest.mark.parametrize("arch", ["vgg16", "resnet18_bn", "alexnet"])
def test_net_memory_matches_oracle(lib, arch):
    """fxpq_net_memory (host-only) against the oracle's RW_R / RO_R on a workload's bit plan."""
    import torch
    import synth
    from paper_2203_12091_gb300 import fxpq as F
    from paper_2203_12091_gb300.net import QNet
    layers = synth.ARCHS[arch]()
    plan = synth.bit_plan(arch, 3)
    q = QNet(layers)
    dummy = torch.zeros(8)
    q.fmts["input"] = {"a": F.fmt(plan["input"], 1, 0)}
    bits = {"input": plan["input"]}
    params = []
    prev = "input"
    for i, Lr in enumerate(layers):
        nm = Lr["name"]
        p = plan.get(nm, {})
        f = q.fmts.setdefault(nm, {})
        last = i == len(layers) - 1
        if "a" in p:
            f["a"] = F.fmt(p["a"], 1, 0)
        if Lr["type"] == "conv":
            f["w"] = F.fmt(p["w"], 1, 0)
            params.append((Lr["K"] * Lr["R"] * Lr["R"] * Lr["C"], p["w"]))
            if "b" in p:
                f["b"] = F.fmt(p["b"], 1, 0)
                params.append((Lr["K"], p["b"]))
            q.q[nm] = (dummy, dummy if "b" in p else None)
            if Lr.get("bn"):
                f["s"], f["h"] = F.fmt(p["s"], 1, 0), F.fmt(p["h"], 1, 0)
                q.qs[nm] = (dummy, dummy)
                params += [(Lr["K"], p["s"]), (Lr["K"], p["h"])]
        elif Lr["type"] == "avgpool":
            f["r"] = F.fmt(p["r"], 0, 0)
            q.q[nm] = (None, 1)
        bits[nm] = 32 if last else (bits[Lr.get("src") or prev] if Lr["type"] == "maxpool" else p["a"])
        prev = nm
    q._build_ops()
    rw, ro = F.fxpq_net_memory(q.net, False)
    rw32, ro32 = F.fxpq_net_memory(q.net, True)
    from tests.test_oracle_pins import _act_elems
    elems = _act_elems(layers)
    assert rw == pytest.approx(oracle.rw_r(layers, elems, bits), rel=1e-12)
    assert ro == pytest.approx(oracle.ro_r(params), rel=1e-12)
    assert rw32 == pytest.approx(oracle.rw_r(layers, elems, {nm: 32 for nm in bits}), rel=1e-12)
    assert ro32 == pytest.approx(oracle.ro_r([(n, 32) for n, _ in params]), rel=1e-12)


def test_new_entry_points_reject_bad_arguments(lib):
    """Every rejected call returns before any launch (no device is touched)."""
    p = ctypes.c_void_p(256)
    assert lib.fxpq_pack_codes(p, 10, L.Fmt(0, 1, 0), p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_pack_codes(p, 10, L.Fmt(17, 1, 0), p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_pack_codes(p, -1, L.Fmt(4, 1, 0), p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_pack_codes(p, 10, L.Fmt(4, 1, 0), ctypes.c_void_p(258), None) == L.ERR_INVALID_ARG
    assert lib.fxpq_unpack_codes(p, 10, L.Fmt(4, 2, 0), p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_unpack_codes(None, 10, L.Fmt(4, 1, 0), p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_bn_to_scale(p, p, p, p, -1, 1e-5, p, p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_bn_to_scale(p, p, p, p, 8, -1.0, p, p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_bn_to_scale(p, None, p, p, 8, 1e-5, p, p, None) == L.ERR_INVALID_ARG
    assert lib.fxpq_quantize(p, 4, L.Fmt(1, 2, 0), L.DT_I8, p, None) == L.ERR_INVALID_ARG
    item = L.FlSearchItem(256, 100, -1, 1, 8, 0, 10, 256, 256, None, 2)  # unknown score
    ws = lib.fxpq_fl_search_batch_workspace(1)
    arr = (L.FlSearchItem * 1)(item)
    assert lib.fxpq_fl_search_batch(ctypes.cast(arr, ctypes.c_void_p), 1, p, ws, None) == L.ERR_INVALID_ARG
    rw, ro = ctypes.c_double(), ctypes.c_double()
    assert lib.fxpq_net_memory(None, 0, ctypes.byref(rw), ctypes.byref(ro)) == L.ERR_INVALID_ARG
