"""Oracle of the forward optimizer: Alg. 1 (QParamsOpt) with the cost F of
Eq. quantization_parameters_optimization, applied in the forward optimizer's order (Sec. IV-C).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).  Plain numpy in float64; the FP32 parts of the
network are evaluated in float64 here (the GPU evaluates them in fp32; the tests compare within a
tolerance).

Readings of the paper used here, where it is silent or ambiguous (the CUDA path follows the same
readings):

* Data-structures: the network input's activations ("input", a only), then per layer in order its
  weights w, bias b (conv/FC only) and output activations a (not for MAX-POOL, which has no QLayer,
  and not for the last layer, which has none either).  a of a layer is its C-Block output.
* The mixed network while (d, l) is optimized: every data-structure optimized before (d, l) is fixed-
  point at its chosen QPs, d takes the candidate, every later one is FP32 (Sec. IV-C: "succeeding
  layers ... floating-point", "preceding layers ... fixed-point"; within a layer, w then b then a).
* E(d, l) sums pi * L / R over the data-structures of layers l, l+1, ... (Eq. CPB_QE): L is the
  quantization error of the data-structure's FP32 values in this forward under its QPs (the
  candidate for d, the chosen QPs for those already optimized, the initial QPs otherwise); R its
  range max - min (a term with R = 0 is 0); pi by Eq. importance with sigma the population standard
  deviation (for activations the mean over calibration samples of the per-sample deviation) and nu
  the element count (per sample for activations).
* UnClass / MisPred (Eqs. unclassified_samples, mispredicted_classes) from the logits: |C_i| is the
  number of classes tied at the largest logit of sample i; T_C the number of classes.
* Initial QPs (preprocessor, Eq. initial_quantization_parameters) from the ranges of the FP32
  network on the calibration slice and of the FP32 parameters, with a given rounding strategy.
* Alg. 1 moves FL by +-k at a fixed wordlength (alpha + beta constant), direction -1 first, and
  accepts a candidate only on a strict improvement; FLs outside [-32, 40] end that direction.
"""
from __future__ import annotations

import numpy as np

from . import conv2d, fl_init, qmax, qmin, rne_shift  # noqa: F401

FL_MIN, FL_MAX = -32, 40


# ------------------------------------------------------------------ fixed-point helpers (float64)
def q64(x, k: int, S: int, fl: int) -> np.ndarray:
    """Eq. fp_k_bit_quantization on float64 data (round half to even, clip); the binary quantizer for
    k = 1, S = 1."""
    x = np.asarray(x, dtype=np.float64)
    if k == 1 and S == 1:
        return np.where(x < 0, -1, 0).astype(np.int64)
    return np.clip(np.round(np.ldexp(x, fl)), qmin(k, S), qmax(k, S)).astype(np.int64)


def val64(codes, k: int, S: int, fl: int) -> np.ndarray:
    c = np.asarray(codes, dtype=np.int64)
    if k == 1 and S == 1:
        c = 2 * c + 1
    return np.ldexp(c.astype(np.float64), -fl)


def qerr(x, fmt) -> float:
    """L of Eq. DSB_QE: sum of (x - Q(x))^2."""
    k, S, fl = fmt
    d = np.asarray(x, np.float64) - val64(q64(x, k, S, fl), k, S, fl)
    return float(np.sum(d * d))


# ------------------------------------------------------------------ FP32 layers (evaluated in float64)
def f_conv(x, w, b, stride, pad, relu):
    """x NHWC, w KRSC (K, R, S, C), b [K] or None."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    N, H, W, C = x.shape
    K, R, S_, _ = w.shape
    P, Q = (H + 2 * pad - R) // stride + 1, (W + 2 * pad - S_) // stride + 1
    xp = np.zeros((N, H + 2 * pad, W + 2 * pad, C))
    xp[:, pad:pad + H, pad:pad + W, :] = x
    cols = np.empty((N, P, Q, R, S_, C))
    for r in range(R):
        for s in range(S_):
            cols[:, :, :, r, s, :] = xp[:, r:r + stride * P:stride, s:s + stride * Q:stride, :]
    y = cols.reshape(N * P * Q, -1) @ w.reshape(K, -1).T
    if b is not None:
        y = y + np.asarray(b, np.float64)
    if relu:
        y = np.maximum(y, 0.0)
    return y.reshape(N, P, Q, K)


def f_maxpool(x, k, stride, pad):
    N, H, W, C = x.shape
    P, Q = (H + 2 * pad - k) // stride + 1, (W + 2 * pad - k) // stride + 1
    out = np.full((N, P, Q, C), -np.inf)
    for r in range(k):
        for s in range(k):
            for p in range(P):
                h = p * stride + r - pad
                if h < 0 or h >= H:
                    continue
                for q in range(Q):
                    ww = q * stride + s - pad
                    if 0 <= ww < W:
                        out[:, p, q, :] = np.maximum(out[:, p, q, :], x[:, h, ww, :])
    return out


def f_avgpool(x):
    return np.mean(np.asarray(x, np.float64), axis=(1, 2), keepdims=True)


# ------------------------------------------------------------------ data-structure statistics
def ds_stats(x, per_sample: bool):
    """(sigma, nu, R) of a data-structure: Eq. importance's dispersion and size, Eq. data_range."""
    x = np.asarray(x, np.float64)
    if per_sample:
        flat = x.reshape(x.shape[0], -1)
        sigma = float(np.mean(np.std(flat, axis=1)))
        nu = flat.shape[1]
    else:
        sigma = float(np.std(x))
        nu = x.size
    return sigma, nu, float(np.max(x) - np.min(x))


def ties(logits) -> np.ndarray:
    """|C_i|: classes tied at the largest logit, per sample."""
    lg = np.asarray(logits)
    return np.sum(lg == lg.max(axis=1, keepdims=True), axis=1)


def unclass_mispred(logits):
    c = ties(logits)
    n, tc = c.size, np.asarray(logits).shape[1]
    return float(np.mean(c > 1)), float(np.sum(c - 1)) / (n * tc)


# ------------------------------------------------------------------ the mixed forward and its cost
def data_structures(layers):
    """Forward optimizer order: ("input", "a"), then per layer w, b, a (where present)."""
    out = [("input", "a")]
    for i, L in enumerate(layers):
        last = i == len(layers) - 1
        if L["type"] == "conv":
            out += [(L["name"], "w"), (L["name"], "b")]
            if not last:
                out.append((L["name"], "a"))
        elif L["type"] in ("eltwise", "avgpool") and not last:
            out.append((L["name"], "a"))
    return out


class Net:
    """A network with FP32 parameters and a calibration slice; the fixed-point state of every
    data-structure (its QPs and whether it is quantized yet)."""

    def __init__(self, layers, weights, images_nchw, plan, strategy="conservative", recip_fmt_bits=16):
        self.layers = layers
        self.W = weights
        self.x0 = np.transpose(np.asarray(images_nchw, np.float64), (0, 2, 3, 1))
        self.plan = plan
        self.order = data_structures(layers)
        self.fmt = {}
        self.done = set()
        # AVG-POOL's reciprocal 1/(H W) is a parameter quantized at a fixed 16-bit format by the FL
        # search (not optimized here)
        self.recip = {}
        acts = self.fp32_forward()
        for nm, j in self.order:
            if j == "a":
                x = acts[nm]
                k = plan["input"] if nm == "input" else plan[nm]["a"]
            else:
                x = weights[nm][0] if j == "w" else weights[nm][1]
                k = plan[nm][j]
            S, beta, _ = fl_init(float(np.min(x)), float(np.max(x)), k, strategy)
            self.fmt[(nm, j)] = (k, S, beta)

    def _recip(self, nm, hw):
        from . import fl_search
        from . import quantize as qz
        r = np.array([1.0 / hw], np.float32)
        _, best, S, _ = fl_search(r, -1, 16, 16, -8, 23)
        fmt = (16, S, int(best[0]))
        return fmt, int(qz(r, *fmt)[0])

    def fp32_forward(self):
        """Activations (C-Block outputs) of the all-FP32 network: name -> float64 NHWC."""
        env = {"input": self.x0}
        prev = "input"
        for L in self.layers:
            nm = L["name"]
            if L["type"] == "conv":
                x = env[L.get("src") or prev]
                w, b = self.W[nm]
                env[nm] = f_conv(x, w, b, L["stride"], L["pad"], L["relu"])
            elif L["type"] == "maxpool":
                env[nm] = f_maxpool(env[prev], L["k"], L["stride"], L["pad"])
            elif L["type"] == "eltwise":
                v = env[L["a"]] + env[L["b"]]
                env[nm] = np.maximum(v, 0.0) if L["relu"] else v
            elif L["type"] == "avgpool":
                env[nm] = f_avgpool(env[L.get("src") or prev])
            prev = nm
        return env

    def forward(self, cur, cand_fl):
        """The mixed forward while data-structure `cur` = (name, j) takes FL cand_fl.

        Returns (X: data-structure -> (float64 values, fmt, per_sample) for the cost's terms, logits)."""
        pos = self.order.index(cur)
        fixed = set(self.order[:pos])  # optimized before cur: fixed point at their chosen QPs

        def fmt_of(ds):
            if ds == cur:
                k, S, _ = self.fmt[ds]
                return (k, S, cand_fl)
            return self.fmt[ds]

        def is_q(ds):
            return ds in fixed or ds == cur

        X = {}
        # each env entry: float64 values (the exact value of the codes when quantized)
        if is_q(("input", "a")):
            f = fmt_of(("input", "a"))
            env = {"input": val64(q64(self.x0, *f), *f)}
        else:
            env = {"input": self.x0}
        X[("input", "a")] = (self.x0, fmt_of(("input", "a")), True)
        prev = "input"
        logits = None
        for i, L in enumerate(self.layers):
            nm = L["name"]
            last = i == len(self.layers) - 1
            if L["type"] == "conv":
                x = env[L.get("src") or prev]
                w, b = self.W[nm]
                wv = val64(q64(w, *fmt_of((nm, "w"))), *fmt_of((nm, "w"))) if is_q((nm, "w")) else w
                bv = val64(q64(b, *fmt_of((nm, "b"))), *fmt_of((nm, "b"))) if is_q((nm, "b")) else b
                y = f_conv(x, wv, bv, L["stride"], L["pad"], L["relu"])
                X[(nm, "w")] = (w, fmt_of((nm, "w")), False)
                X[(nm, "b")] = (b, fmt_of((nm, "b")), False)
            elif L["type"] == "maxpool":
                y = f_maxpool(env[prev], L["k"], L["stride"], L["pad"])
            elif L["type"] == "eltwise":
                y = env[L["a"]] + env[L["b"]]
                if L["relu"]:
                    y = np.maximum(y, 0.0)
            else:  # avgpool: the reciprocal of the patch size is a quantized parameter once the layer is
                x = env[L.get("src") or prev]
                hw = x.shape[1] * x.shape[2]
                if is_q((nm, "a")):
                    rf, rc = self._recip(nm, hw)
                    y = np.sum(x, axis=(1, 2), keepdims=True) * val64(rc, *rf)
                else:
                    y = f_avgpool(x)
            if last:
                logits = y.reshape(y.shape[0], -1)
            elif L["type"] != "maxpool":
                X[(nm, "a")] = (y, fmt_of((nm, "a")), True)
                if is_q((nm, "a")):
                    f = fmt_of((nm, "a"))
                    y = val64(q64(y, *f), *f)
            env[nm] = y
            prev = nm
        return X, logits

    def cost(self, cur, cand_fl):
        """F = E + UnClass + MisPred for data-structure cur at FL cand_fl; returns (F, E, UnClass, MisPred)."""
        X, logits = self.forward(cur, cand_fl)
        name = cur[0]
        start = 0 if name == "input" else 1 + [L["name"] for L in self.layers].index(name)
        names = ["input"] + [L["name"] for L in self.layers]
        E = 0.0
        for li in range(start, len(names)):
            nm = names[li]
            terms = [(j, X[(nm, j)]) for j in ("a", "w", "b") if (nm, j) in X]
            if not terms:
                continue
            st = {j: ds_stats(v, ps) for j, (v, f, ps) in terms}
            den = sum(s * n for s, n, _ in st.values())
            for j, (v, f, ps) in terms:
                s, n, R = st[j]
                if den == 0.0 or R == 0.0:
                    continue
                E += (s * n / den) * qerr(v, f) / R
        uc, mp = unclass_mispred(logits)
        return E + uc + mp, E, uc, mp


def qparams_opt(cost_fn, init: int, K: int = 1):
    """Alg. 1 around the initial FL `init` with cost_fn(FL) -> F (Sec. IV-C): the FL moves away from init in
    each direction at a fixed wordlength; a candidate is accepted only when its cost is strictly below the
    best so far, and each acceptance lets its direction go one step beyond the K steps it always takes;
    FLs outside [FL_MIN, FL_MAX] end a direction.  Returns (best FL, best cost, [(FL, cost)] in the order
    visited)."""
    best_fl, best = init, cost_fn(init)
    trace = [(init, best)]
    for d in (-1, 1):
        steps, k = K, 1
        while k <= steps and FL_MIN <= init + d * k <= FL_MAX:
            fl = init + d * k
            c = cost_fn(fl)
            trace.append((fl, c))
            if c < best:
                best, best_fl = c, fl
                steps += 1
            k += 1
    return best_fl, best, trace


def forward_optimize(net: Net, K: int = 1, upto=None):
    """The forward optimizer: Alg. 1 on every data-structure in order (the first `upto` of them if
    given); each chosen FL is fixed before the next.  Returns [(data-structure, best FL, cost, trace)]."""
    out = []
    for cur in net.order[: upto if upto is not None else len(net.order)]:
        fl, c, tr = qparams_opt(lambda f: net.cost(cur, f)[0], net.fmt[cur][2], K)
        k, S, _ = net.fmt[cur]
        net.fmt[cur] = (k, S, fl)
        net.done.add(cur)
        out.append((cur, fl, c, tr))
    return out
