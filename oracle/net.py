"""Oracle network executor: calibration and integer-only forward of a quantized CNN.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Readings of the paper used here, where it is silent or ambiguous (the CUDA path follows the same
readings):

* FxP-QLayers sit after the input and after every C-Block output, not after MAX-POOL and
  not after the last layer (Sec. IV-A.2).
* Calibration follows the forward optimizer's order (Sec. IV-C, last paragraphs): layer by
  layer; per layer the weights' FL, then the bias FL, then the output activation FL.  The
  activation FL is chosen by the FL search (Eq. DSB_QE) on the fp32 nearest-even image of the
  exact C-Block output (after bias and ReLU) of the calibration slice, computed with all
  preceding layers already quantized.
* The sign strategy is Sec. IV-A.3's: S = 1 iff the smallest value is negative.
* The AVG-POOL reciprocal 1/(patch size) is a 16-bit unsigned parameter whose FL is searched
  like any other parameter.
* A BN layer after a conv is rewritten as a Scale layer (Sec. IV-A.1): aleph1 and aleph2 come from
  bn_to_scale in fp32 and are then searched and quantized like weights and biases (aleph1 after
  the weights, aleph2 after it); the C-Block applies them after the (absent) bias and before ReLU.
"""
from __future__ import annotations

import numpy as np

from . import (avgpool_global, bn_to_scale, cblock, conv2d, eltwise_add, fl_search, maxpool, quantize,
               requant, to_f32)

FL_LO, FL_HI = -8, 23


def search_fmt(x, k: int):
    """(k, S, FL) of a data-structure: FL search over [FL_LO, FL_HI] at one wordlength k, S by min."""
    _, best, S, _ = fl_search(np.asarray(x, dtype=np.float32).reshape(-1), -1, k, k, FL_LO, FL_HI)
    return (k, S, int(best[0]))


def images_to_codes(images_nchw, fmt):
    k, S, fl = fmt
    x = np.ascontiguousarray(np.transpose(np.asarray(images_nchw, dtype=np.float32), (0, 2, 3, 1)))
    return quantize(x, k, S, fl).reshape(x.shape)


def _is_last(layers, i):
    return i == len(layers) - 1


def _layer_pass(layers, i, L, env, fmts, qparams, calibrating: bool, plan):
    """Run layer i on the codes in env; during calibration choose the output FL."""
    name = L["name"]
    prev = layers[i - 1]["name"] if i > 0 else "input"
    if L["type"] == "conv":
        src = L.get("src") or prev
        x, fx = env[src]
        wq, bq = qparams[name][:2]
        fw, fb = fmts[name]["w"], fmts[name].get("b", (0, 0, 0))
        if x.ndim == 2:
            x = x.reshape(x.shape[0], 1, 1, -1)
        acc = conv2d(x, wq, L["stride"], L["pad"])
        if L.get("bn"):
            sq, hq = qparams[name][2:]
            v, s = cblock(acc, fx[2] + fw[2], bq, fb[2], L["relu"], scale=sq, fl_scale=fmts[name]["s"][2],
                          shift=hq, fl_shift=fmts[name]["h"][2])
        else:
            v, s = cblock(acc, fx[2] + fw[2], bq, fb[2], L["relu"])
        if _is_last(layers, i):
            env[name] = (v.reshape(v.shape[0], -1), ("logits", None, s))
            return
    elif L["type"] == "maxpool":
        x, fx = env[prev]
        env[name] = (maxpool(x, L["k"], L["stride"], L["pad"]), fx)
        return
    elif L["type"] == "eltwise":
        (a, fa), (b, fb) = env[L["a"]], env[L["b"]]
        v, s = eltwise_add(a, fa[2], b, fb[2], L["relu"])
    elif L["type"] == "avgpool":
        x, fx = env[L.get("src") or prev]
        if calibrating:  # reciprocal of the patch size, searched like a parameter
            fmts[name]["r"] = search_fmt(np.array([1.0 / (x.shape[1] * x.shape[2])], dtype=np.float32), plan[name]["r"])
        rk, rS, rfl = fmts[name]["r"]
        rcode = int(quantize(np.array([1.0 / (x.shape[1] * x.shape[2])], dtype=np.float32), rk, rS, rfl)[0])
        v, s = avgpool_global(x, fx[2], rcode, rfl)
        v = v.reshape(v.shape[0], 1, 1, -1)
    else:
        raise ValueError(L["type"])
    if calibrating:
        fmts[name]["a"] = search_fmt(to_f32(v, s), plan[name]["a"])
    k, S, fl = fmts[name]["a"]
    env[name] = (requant(v, s, k, S, fl), fmts[name]["a"])


def quantize_params(layers, weights, plan, bn=None):
    """Weights then bias of every conv/FC layer: FL search at the planned wordlength, then Q.  A conv
    with a BN layer (bn[name] = (gamma, beta, mean, var)) has no bias; its Scale parameters aleph1
    ("s") and aleph2 ("h") follow the weights.  qparams[name] = (W, B or None[, aleph1, aleph2])."""
    fmts, qparams = {}, {}
    for L in layers:
        nm = L["name"]
        fmts[nm] = {}
        if L["type"] == "conv":
            w, b = weights[nm]
            fw = search_fmt(w, plan[nm]["w"])
            fmts[nm]["w"] = fw
            qw = quantize(w, *fw).reshape(w.shape)
            if b is not None:
                fb = search_fmt(b, plan[nm]["b"])
                fmts[nm]["b"] = fb
                qparams[nm] = (qw, quantize(b, *fb))
            else:
                qparams[nm] = (qw, None)
            if L.get("bn"):
                a1, a2 = bn_to_scale(*bn[nm])
                fs = search_fmt(a1, plan[nm]["s"])
                fh = search_fmt(a2, plan[nm]["h"])
                fmts[nm]["s"], fmts[nm]["h"] = fs, fh
                qparams[nm] = qparams[nm] + (quantize(a1, *fs), quantize(a2, *fh))
    return fmts, qparams


def calibrate(layers, weights, calib_images_nchw, plan, bn=None):
    """Forward-optimizer-order calibration on a slice.  Returns (fmts, qparams)."""
    fmts, qparams = quantize_params(layers, weights, plan, bn)
    fmts["input"] = search_fmt(calib_images_nchw, plan["input"])
    env = {"input": (images_to_codes(calib_images_nchw, fmts["input"]), fmts["input"])}
    for i, L in enumerate(layers):
        _layer_pass(layers, i, L, env, fmts, qparams, True, plan)
    return fmts, qparams


def forward(layers, fmts, qparams, images_nchw):
    """Integer-only forward with frozen formats.  Returns (logits int64 [N, classes], scale exponent)."""
    env = {"input": (images_to_codes(images_nchw, fmts["input"]), fmts["input"])}
    for i, L in enumerate(layers):
        _layer_pass(layers, i, L, env, fmts, qparams, False, None)
    logits, f = env[layers[-1]["name"]]
    return logits, f[2]


def forward_trace(layers, fmts, qparams, images_nchw):
    """As forward(), returning every layer's output codes (for per-layer parity tests)."""
    env = {"input": (images_to_codes(images_nchw, fmts["input"]), fmts["input"])}
    for i, L in enumerate(layers):
        _layer_pass(layers, i, L, env, fmts, qparams, False, None)
    return env
