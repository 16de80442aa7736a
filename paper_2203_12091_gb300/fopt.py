"""The forward optimizer (Sec. IV-C): Alg. 1 (QParamsOpt) on every data-structure in the order input,
then per layer weights, bias, activations, each candidate scored by the cost
F = E + UnClass + MisPred (Eq. quantization_parameters_optimization) on a calibration slice.

While data-structure d of layer l is optimized, every data-structure optimized before it is fixed
point at its chosen QPs, d takes the candidate, and every later one is FP32: the forward runs the
integer C-Blocks (fxpq_conv_fwd, fxpq_eltwise, fxpq_avgpool, fxpq_maxpool) up to the point where FP32
takes over (fxpq_dequantize), then the FP32 layers (fxpq_conv_f32, ...).  E sums, over the
data-structures of layers l, l+1, ..., the importance pi (Eq. importance) times the quantization
error L (Eq. DSB_QE) over the range R (Eq. data_range), each from fxpq_ds_stats on the data-structure's
FP32 values in that forward; UnClass and MisPred count top-1 ties of the logits (fxpq_top1_ties).
The initial QPs come from the preprocessor (Eq. initial_quantization_parameters, fxpq_fl_init) on the
ranges of the FP32 network.  Every arithmetic step runs in libfxpq.so; this module sequences the calls
and combines a handful of per-data-structure scalars on the host.
"""
from __future__ import annotations

import math

import torch

from . import _lib as L
from . import fxpq as F
from .net import pad8, search_fmt

FL_MIN, FL_MAX = -32, 40
STRATEGY = {"conservative": 0, "neutral": 1, "aggressive": 2}


def data_structures(layers):
    """Forward optimizer order: ("input", "a"), then per layer w, b, a (where present; MAX-POOL and the last
    layer have no activation QLayer)."""
    out = [("input", "a")]
    for i, L_ in enumerate(layers):
        last = i == len(layers) - 1
        if L_["type"] == "conv":
            out += [(L_["name"], "w"), (L_["name"], "b")]
            if not last:
                out.append((L_["name"], "a"))
        elif L_["type"] in ("eltwise", "avgpool") and not last:
            out.append((L_["name"], "a"))
    return out


class _Q:
    """A fixed-point tensor: fp16 code tensor [N, H, W, Cp], its format and true channel count."""

    def __init__(self, t, fmt, H, W, C, Cp):
        self.t, self.fmt, self.H, self.W, self.C, self.Cp = t, fmt, H, W, C, Cp


class _F:
    """An FP32 tensor [N, H, W, C]."""

    def __init__(self, t, H, W, C):
        self.t, self.H, self.W, self.C = t, H, W, C


class ForwardOptimizer:
    def __init__(self, layers, weights_dev, images, plan, strategy="conservative", stream=None):
        """weights_dev: name -> (fp32 KRSC weight, fp32 bias) device tensors; images: fp32 NCHW device
        tensor (the calibration slice); plan: wordlengths (as for the network)."""
        self.layers, self.W, self.plan, self.stream = layers, weights_dev, plan, stream
        self.dev = images.device
        self.N, self.cin, self.hw = images.shape[0], images.shape[1], images.shape[2]
        self.x0 = images.contiguous()
        self.x0_nhwc = torch.empty(self.N * self.hw * self.hw * self.cin, dtype=torch.float32, device=self.dev)
        F.fxpq_nchw_to_nhwc_f32(self.x0, self.N, self.cin, self.hw, self.hw, self.x0_nhwc, stream)
        self.order = data_structures(layers)
        self.names = ["input"] + [L_["name"] for L_ in layers]
        self._stats_out = torch.empty(3 + 2 * max(self.N, 1), dtype=torch.float64, device=self.dev)
        self._stats_ws = torch.empty(2, dtype=torch.int32, device=self.dev)
        self._recip = {}
        self.fmt = {}
        acts = self._fp32_forward()
        for nm, j in self.order:
            if j == "a":
                x = acts[nm].t
                k = plan["input"] if nm == "input" else plan[nm]["a"]
                n_s, nu = self.N, x.numel() // self.N
            else:
                x = self.W[nm][0] if j == "w" else self.W[nm][1]
                k = plan[nm][j]
                n_s, nu = 1, x.numel()
            st = self._stats(x.reshape(-1), n_s, nu, F.fmt(k, 1, 0))
            stats = L.Stats(st["min"], st["max"], 0, 0, 0.0, 0.0, x.numel())
            self.fmt[(nm, j)] = F.fxpq_fl_init(stats, k, STRATEGY[strategy])

    # ------------------------------------------------------------------ device statistics
    def _stats(self, x, n_samples, nu, fmt):
        out = self._stats_out[: 3 + 2 * n_samples]
        F.fxpq_ds_stats(x, n_samples, nu, fmt, out, self._stats_ws, self.stream)
        return _decode(out.cpu().tolist(), 0, n_samples, nu)

    # ------------------------------------------------------------------ helpers
    def _src(self, i, L_):
        s = L_.get("src")
        return s if s is not None else self.names[i]

    def _empty(self, n, dtype=torch.float32):
        return torch.empty(max(n, 1), dtype=dtype, device=self.dev)

    def _to_f(self, v):
        if isinstance(v, _F):
            return v
        y = self._empty(self.N * v.H * v.W * v.C)
        F.fxpq_dequantize(v.t, self.N * v.H * v.W, v.Cp, v.C, v.fmt, y, self.stream)
        return _F(y, v.H, v.W, v.C)

    def _recip_of(self, nm, hw):
        if nm not in self._recip:
            r = torch.tensor([1.0 / hw], dtype=torch.float32, device=self.dev)
            f = search_fmt(r, self.plan[nm]["r"], self.stream)
            c = self._empty(1, torch.int32)
            F.fxpq_quantize(r, f, L.DT_I32, c, self.stream)
            self._recip[nm] = (f, int(c.item()))
        return self._recip[nm]

    def _q_params(self, nm, fw, fb, Cp):
        w, b = self.W[nm]
        K, R, _, C = w.shape
        wq = self._empty(K * R * R * Cp * F.planes(fw), torch.float16)
        F.fxpq_quantize_rows(w, K * R * R, C, fw, Cp, wq, self.stream)
        bq = None
        if fb is not None:
            bq = self._empty(K, torch.int32)
            F.fxpq_quantize(b, fb, L.DT_I32, bq, self.stream)
        return wq, bq

    # ------------------------------------------------------------------ the all-FP32 network
    def _fp32_forward(self):
        env = {"input": _F(self.x0_nhwc, self.hw, self.hw, self.cin)}
        for i, L_ in enumerate(self.layers):
            env[L_["name"]] = self._f_layer(i, L_, env, None)
        return env

    def _f_layer(self, i, L_, env, wq_override):
        """One layer in FP32 on FP32 inputs (dequantized where needed)."""
        nm, typ = L_["name"], L_["type"]
        if typ == "conv":
            x = self._to_f(env[self._src(i, L_)])
            w, b = self.W[nm]
            K, R = L_["K"], L_["R"]
            P = (x.H + 2 * L_["pad"] - R) // L_["stride"] + 1
            y = self._empty(self.N * P * P * K)
            F.fxpq_conv_f32(self.N, x.H, x.W, x.C, K, R, R, L_["stride"], L_["pad"], L_["relu"], x.t, w, b, y,
                            self.stream)
            return _F(y, P, P, K)
        if typ == "maxpool":
            x = self._to_f(env[self._src(i, L_)])
            P = (x.H + 2 * L_["pad"] - L_["k"]) // L_["stride"] + 1
            y = self._empty(self.N * P * P * x.C)
            F.fxpq_maxpool_f32(x.t, self.N, x.H, x.W, x.C, L_["k"], L_["stride"], L_["pad"], y, self.stream)
            return _F(y, P, P, x.C)
        if typ == "eltwise":
            a, b = self._to_f(env[L_["a"]]), self._to_f(env[L_["b"]])
            y = self._empty(self.N * a.H * a.W * a.C)
            F.fxpq_eltwise_f32(a.t, b.t, self.N * a.H * a.W * a.C, L_["relu"], y, self.stream)
            return _F(y, a.H, a.W, a.C)
        x = self._to_f(env[self._src(i, L_)])  # avgpool
        y = self._empty(self.N * x.C)
        F.fxpq_avgpool_f32(x.t, self.N, x.H, x.W, x.C, y, self.stream)
        return _F(y, 1, 1, x.C)

    # ------------------------------------------------------------------ the mixed forward
    def forward(self, cur, cand_fl):
        """Forward of the calibration slice while data-structure cur = (name, j) takes FL cand_fl.
        Returns (X: data-structure -> (fp32 device values, fmt, n_samples, nu) for the cost, logits)."""
        pos = self.order.index(cur)
        fixed = set(self.order[:pos])

        def fmt_of(ds):
            if ds == cur:
                f = self.fmt[ds]
                return F.fmt(f.bits, f.is_signed, cand_fl)
            return self.fmt[ds]

        def is_q(ds):
            return ds in fixed or ds == cur

        X = {}
        if is_q(("input", "a")):
            f = fmt_of(("input", "a"))
            cp = pad8(self.cin)
            t = self._empty(self.N * self.hw * self.hw * cp * F.planes(f), torch.float16)
            F.fxpq_quantize_images(self.x0, f, cp, t, self.stream)
            env = {"input": _Q(t, f, self.hw, self.hw, self.cin, cp)}
        else:
            env = {"input": _F(self.x0_nhwc, self.hw, self.hw, self.cin)}
        X[("input", "a")] = (self.x0_nhwc, fmt_of(("input", "a")), self.N, self.hw * self.hw * self.cin)
        logits = None
        for i, L_ in enumerate(self.layers):
            nm, typ = L_["name"], L_["type"]
            last = i == len(self.layers) - 1
            if typ == "conv":
                X[(nm, "w")] = (self.W[nm][0], fmt_of((nm, "w")), 1, self.W[nm][0].numel())
                X[(nm, "b")] = (self.W[nm][1], fmt_of((nm, "b")), 1, self.W[nm][1].numel())
            qa = (nm, "a") in self.fmt
            if typ == "maxpool":
                src = env[self._src(i, L_)]
                if isinstance(src, _Q):
                    P = (src.H + 2 * L_["pad"] - L_["k"]) // L_["stride"] + 1
                    y = self._empty(self.N * P * P * src.Cp * F.planes(src.fmt), torch.float16)
                    F.fxpq_maxpool(src.t, self.N, src.H, src.W, src.Cp, src.fmt, L_["k"], L_["stride"], L_["pad"], y,
                                   self.stream)
                    env[nm] = _Q(y, src.fmt, P, P, src.C, src.Cp)
                else:
                    env[nm] = self._f_layer(i, L_, env, None)
                continue
            if typ == "conv" and is_q((nm, "w")):
                env[nm], xa, lg = self._conv_q(i, L_, env, fmt_of, is_q, last)
            elif typ in ("eltwise", "avgpool") and qa and is_q((nm, "a")):
                env[nm], xa = self._other_q(i, L_, env, fmt_of((nm, "a")))
                lg = None
            else:
                y = self._f_layer(i, L_, env, None)
                env[nm], xa, lg = y, y.t, (y.t if last else None)
            if last:
                logits = lg
            else:
                X[(nm, "a")] = (xa, fmt_of((nm, "a")), self.N, env_size(env[nm]))
        return X, logits

    def _conv_q(self, i, L_, env, fmt_of, is_q, last):
        """A conv whose weights are fixed point: (output entry, FP32 values of its C-Block output, logits)."""
        nm = L_["name"]
        src = env[self._src(i, L_)]
        assert isinstance(src, _Q), "a fixed-point layer reads fixed-point activations"
        K, R = L_["K"], L_["R"]
        P = (src.H + 2 * L_["pad"] - R) // L_["stride"] + 1
        npix = self.N * P * P
        fw = fmt_of((nm, "w"))
        qb = is_q((nm, "b"))
        fb = fmt_of((nm, "b")) if qb else None
        wq, bq = self._q_params(nm, fw, fb, src.Cp)
        qa = (not last) and is_q((nm, "a"))
        if not qb:
            # weights fixed, bias FP32: exact contraction to fp32, then the FP32 bias and ReLU
            y = self._empty(npix * K)
            d = F.conv_desc(self.N, src.H, src.W, src.Cp, src.Cp, K, R, R, L_["stride"], L_["pad"], False, F.OUT_F32,
                            src.fmt, fw, None, None)
            F.fxpq_conv_fwd(d, src.t, wq, None, y, self.stream)
            F.fxpq_bias_relu_f32(y, npix, K, self.W[nm][1], L_["relu"], self.stream)
            return _F(y, P, P, K), y, (y if last else None)
        # weights and bias fixed: the exact C-Block value
        acc = self._empty(npix * K, torch.int64)
        d = F.conv_desc(self.N, src.H, src.W, src.Cp, src.Cp, K, R, R, L_["stride"], L_["pad"], L_["relu"],
                        F.OUT_ACC64, src.fmt, fw, fb, None)
        s = F.fxpq_conv_fwd(d, src.t, wq, bq, acc, self.stream)
        xf = self._empty(npix * K)
        F.fxpq_qlayer(acc, s, F.OUT_F32, None, xf, self.stream)
        if last:
            return _F(xf, P, P, K), xf, acc
        if not qa:
            return _F(xf, P, P, K), xf, None
        fy = fmt_of((nm, "a"))
        codes = self._empty(npix * K * F.planes(fy), torch.float16)
        F.fxpq_qlayer(acc, s, F.OUT_CODES, fy, codes, self.stream)
        return _Q(codes, fy, P, P, K, K), xf, None

    def _other_q(self, i, L_, env, fy):
        """Eltwise / avg-pool with its output QLayer: (codes entry, FP32 values of the C-Block output)."""
        nm = L_["name"]
        if L_["type"] == "eltwise":
            a, b = env[L_["a"]], env[L_["b"]]
            npix = self.N * a.H * a.W
            acc = self._empty(npix * a.Cp, torch.int64)
            s = F.fxpq_eltwise(a.t, a.fmt, b.t, b.fmt, npix, a.Cp, L_["relu"], F.OUT_ACC64, None, acc, self.stream)
            H, C, Cp = a.H, a.C, a.Cp
        else:
            x = env[self._src(i, L_)]
            rf, rc = self._recip_of(nm, x.H * x.W)
            npix = self.N
            acc = self._empty(npix * x.Cp, torch.int64)
            s = F.fxpq_avgpool(x.t, self.N, x.H, x.W, x.Cp, x.fmt, rc, rf, F.OUT_ACC64, None, acc, self.stream)
            H, C, Cp = 1, x.C, x.Cp
        xf = self._empty(npix * Cp)
        F.fxpq_qlayer(acc, s, F.OUT_F32, None, xf, self.stream)
        codes = self._empty(npix * Cp * F.planes(fy), torch.float16)
        F.fxpq_qlayer(acc, s, F.OUT_CODES, fy, codes, self.stream)
        return _Q(codes, fy, H, H, C, Cp), xf

    # ------------------------------------------------------------------ the cost
    def cost(self, cur, cand_fl):
        """F = E + UnClass + MisPred for cur at FL cand_fl: (F, E, UnClass, MisPred)."""
        X, logits = self.forward(cur, cand_fl)
        start = self.names.index(cur[0])
        # every statistic and the tie counts into one device buffer, read back once
        layers = []
        off = 0
        for nm in self.names[start:]:
            terms = [(j, X[(nm, j)]) for j in ("a", "w", "b") if (nm, j) in X]
            if terms:
                layers.append([(j, t, f, n_s, nu, off + 0) for j, (t, f, n_s, nu) in terms])
                for _, _, _, n_s, _, _ in layers[-1]:
                    off += 3 + 2 * n_s
        n_cls = self.layers[-1]["K"]
        buf = torch.empty(off + self.N, dtype=torch.float64, device=self.dev)
        o = 0
        for terms in layers:
            for i, (j, t, f, n_s, nu, _) in enumerate(terms):
                terms[i] = (j, t, f, n_s, nu, o)
                F.fxpq_ds_stats(t.reshape(-1), n_s, nu, f, buf[o:o + 3 + 2 * n_s], self._stats_ws, self.stream)
                o += 3 + 2 * n_s
        counts = buf[off:].view(torch.int32)[: self.N]
        F.fxpq_top1_ties(logits, self.N, n_cls, counts, self.stream)
        hb = buf.cpu()
        h = hb[:off].tolist()
        E = 0.0
        for terms in layers:
            st = {j: _decode(h, o, n_s, nu) for j, _, _, n_s, nu, o in terms}
            den = sum(v["sigma"] * v["nu"] for v in st.values())
            for j, *_ in terms:
                v = st[j]
                R = v["max"] - v["min"]
                if den == 0.0 or R == 0.0:
                    continue
                E += (v["sigma"] * v["nu"] / den) * v["L"] / R
        c = hb[off:].view(torch.int32)[: self.N]
        uc = float((c > 1).sum()) / self.N
        mp = float((c - 1).sum()) / (self.N * n_cls)
        return E + uc + mp, E, uc, mp

    # ------------------------------------------------------------------ Alg. 1 and the forward optimizer
    def qparams_opt(self, cur, K=1):
        init = self.fmt[cur].fl
        best_fl, cost_best = init, self.cost(cur, init)[0]
        trace = [(init, cost_best)]
        for i in (-1, 1):
            k, j = 1, 0
            while k <= K + j:
                fl = init + i * k
                if fl < FL_MIN or fl > FL_MAX:
                    break
                c = self.cost(cur, fl)[0]
                trace.append((fl, c))
                if c < cost_best:
                    cost_best, best_fl, j = c, fl, j + 1
                k += 1
        return best_fl, cost_best, trace

    def run(self, K=1, upto=None):
        """Alg. 1 on every data-structure in order (the first `upto`), fixing each chosen FL before the next.
        Returns [(data-structure, best FL, cost, trace)]."""
        out = []
        for cur in self.order[: upto if upto is not None else len(self.order)]:
            fl, c, tr = self.qparams_opt(cur, K)
            f = self.fmt[cur]
            self.fmt[cur] = F.fmt(f.bits, f.is_signed, fl)
            out.append((cur, fl, c, tr))
        return out


def env_size(v):
    return v.H * v.W * v.C


def _decode(h, o, n_samples, nu):
    """L, range ends and the mean per-sample dispersion (Eq. importance) of one fxpq_ds_stats record."""
    sig = 0.0
    for s in range(n_samples):
        m1, m2 = h[o + 3 + 2 * s] / nu, h[o + 4 + 2 * s] / nu
        sig += math.sqrt(max(m2 - m1 * m1, 0.0))
    return {"L": h[o], "min": h[o + 1], "max": h[o + 2], "sigma": sig / n_samples, "nu": nu}
