"""The forward optimizer (Sec. IV-C): Alg. 1 (QParamsOpt) on every data-structure in the order input,
then per layer weights, bias, activations, each candidate scored by the cost
F = E + UnClass + MisPred (Eq. quantization_parameters_optimization) on a calibration slice.

While data-structure d of layer l is optimized, every data-structure optimized before it is fixed
point at its chosen QPs, d takes the candidate, and every later one is FP32: the forward runs the
integer C-Blocks (fxpq_conv_fwd, fxpq_eltwise, fxpq_avgpool, fxpq_maxpool) up to the point where FP32
takes over (fxpq_dequantize), then the FP32 layers (fxpq_conv_f32, ...).  E sums, over the
data-structures of layers l, l+1, ..., the importance pi (Eq. importance) times the quantization
error L (Eq. DSB_QE) over the range R (Eq. data_range), from the statistics of the data-structure's
FP32 values in that forward (fxpq_ds_stats_batch); UnClass and MisPred count top-1 ties of the logits
(fxpq_top1_ties); fxpq_fopt_cost forms F on the device.  The candidates of one data-structure share
their forward: the layers before its layer run once, its layer once per candidate, every later layer
once over the candidates stacked along the batch.  The initial QPs come from the preprocessor (Eq.
initial_quantization_parameters, fxpq_fl_init) on the ranges of the FP32 network.  Every arithmetic
step runs in libfxpq.so; this module sequences the calls and reads back one cost per candidate.
"""
from __future__ import annotations

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
        self._recip = {}
        self.fmt = {}
        # initial QPs (preprocessor) from the ranges of the FP32 network: one statistics batch, one read-back
        acts = self._fp32_forward()
        items, ks, off = [], [], 0
        rec = torch.empty(sum(3 + 2 * (self.N if j == "a" else 1) for _, j in self.order), dtype=torch.float64,
                          device=self.dev)
        for nm, j in self.order:
            if j == "a":
                x = acts[nm].t
                k = plan["input"] if nm == "input" else plan[nm]["a"]
                n_s, nu = self.N, x.numel() // self.N
            else:
                x = self.W[nm][0] if j == "w" else self.W[nm][1]
                k = plan[nm][j]
                n_s, nu = 1, x.numel()
            items.append((x.reshape(-1), n_s, nu, F.fmt(k, 1, 0), rec[off:off + 3 + 2 * n_s]))
            ks.append((off, k, x.numel()))
            off += 3 + 2 * n_s
        F.fxpq_ds_stats_batch(items, stream)
        h = rec.cpu().tolist()
        for (nm, j), (o, k, n) in zip(self.order, ks):
            stats = L.Stats(h[o + 1], h[o + 2], 0, 0, 0.0, 0.0, n)
            self.fmt[(nm, j)] = F.fxpq_fl_init(stats, k, STRATEGY[strategy])

    # ------------------------------------------------------------------ helpers
    def _src(self, i, L_):
        s = L_.get("src")
        return s if s is not None else self.names[i]

    def _empty(self, n, dtype=torch.float32):
        return torch.empty(max(n, 1), dtype=dtype, device=self.dev)

    def _to_f(self, v, nb=None):
        if isinstance(v, _F):
            return v
        nb = self.N if nb is None else nb
        y = self._empty(nb * v.H * v.W * v.C)
        F.fxpq_dequantize(v.t, nb * v.H * v.W, v.Cp, v.C, v.fmt, y, self.stream)
        return _F(y, v.H, v.W, v.C)

    def _stack(self, entries):
        """One FP32 entry holding the given entries (each over the N calibration samples) one after the other
        along the batch: candidate c's samples are rows c N .. (c + 1) N - 1."""
        fs = [self._to_f(e) for e in entries]
        n = fs[0].t.numel()
        y = self._empty(n * len(fs))
        for c, f in enumerate(fs):
            y[c * n:(c + 1) * n].copy_(f.t[:n])  # device-to-device copies
        return _F(y, fs[0].H, fs[0].W, fs[0].C)

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
            env[L_["name"]] = self._f_layer(i, L_, env)
        return env

    def _f_layer(self, i, L_, env, nb=None):
        """One layer in FP32 on FP32 inputs (dequantized where needed), over nb samples (N by default)."""
        nm, typ = L_["name"], L_["type"]
        N = self.N if nb is None else nb
        if typ == "conv":
            x = self._to_f(env[self._src(i, L_)], N)
            w, b = self.W[nm]
            K, R = L_["K"], L_["R"]
            P = (x.H + 2 * L_["pad"] - R) // L_["stride"] + 1
            y = self._empty(N * P * P * K)
            F.fxpq_conv_f32(N, x.H, x.W, x.C, K, R, R, L_["stride"], L_["pad"], L_["relu"], x.t, w, b, y,
                            self.stream)
            return _F(y, P, P, K)
        if typ == "maxpool":
            x = self._to_f(env[self._src(i, L_)], N)
            P = (x.H + 2 * L_["pad"] - L_["k"]) // L_["stride"] + 1
            y = self._empty(N * P * P * x.C)
            F.fxpq_maxpool_f32(x.t, N, x.H, x.W, x.C, L_["k"], L_["stride"], L_["pad"], y, self.stream)
            return _F(y, P, P, x.C)
        if typ == "eltwise":
            a, b = self._to_f(env[L_["a"]], N), self._to_f(env[L_["b"]], N)
            y = self._empty(N * a.H * a.W * a.C)
            F.fxpq_eltwise_f32(a.t, b.t, N * a.H * a.W * a.C, L_["relu"], y, self.stream)
            return _F(y, a.H, a.W, a.C)
        x = self._to_f(env[self._src(i, L_)], N)  # avgpool
        y = self._empty(N * x.C)
        F.fxpq_avgpool_f32(x.t, N, x.H, x.W, x.C, y, self.stream)
        return _F(y, 1, 1, x.C)

    # ------------------------------------------------------------------ the mixed forward
    def _q_input(self, f):
        cp = pad8(self.cin)
        t = self._empty(self.N * self.hw * self.hw * cp * F.planes(f), torch.float16)
        F.fxpq_quantize_images(self.x0, f, cp, t, self.stream)
        return _Q(t, f, self.hw, self.hw, self.cin, cp)

    def _fixed_layer(self, i, L_, env):
        """A layer before the current data-structure's: every data-structure of it is fixed point."""
        nm = L_["name"]
        if L_["type"] == "maxpool":
            src = env[self._src(i, L_)]
            P = (src.H + 2 * L_["pad"] - L_["k"]) // L_["stride"] + 1
            y = self._empty(self.N * P * P * src.Cp * F.planes(src.fmt), torch.float16)
            F.fxpq_maxpool(src.t, self.N, src.H, src.W, src.Cp, src.fmt, L_["k"], L_["stride"], L_["pad"], y,
                           self.stream)
            return _Q(y, src.fmt, P, P, src.C, src.Cp)
        if L_["type"] == "conv":
            return self._conv_q(i, L_, env, lambda ds: self.fmt[ds], lambda ds: True, False)[0]
        return self._other_q(i, L_, env, self.fmt[(nm, "a")])[0]

    def _forward_candidates(self, cur, fls):
        """The calibration slice through the mixed network for each candidate FL of cur (Sec. IV-C: the
        data-structures optimized before cur fixed point, cur at the candidate, every later one FP32).

        The layers before cur's layer are the same for every candidate and run once; cur's layer runs
        once per candidate; every later layer runs once over the candidates stacked along the batch.
        Returns (terms: per candidate {data-structure: (fp32 values, fmt, n_samples, nu)}, stacked
        logits [n_cand N, classes] (fp32, or exact int64 when cur's layer is the last one))."""
        N, nc = self.N, len(fls)
        pos = self.order.index(cur)
        fixed = set(self.order[:pos])
        cl = self.names.index(cur[0]) - 1  # cur's layer; -1: the input QLayer

        def fmt_for(fl):
            def fmt_of(ds):
                if ds == cur:
                    f = self.fmt[ds]
                    return F.fmt(f.bits, f.is_signed, fl)
                return self.fmt[ds]
            return fmt_of

        def is_q(ds):
            return ds in fixed or ds == cur

        terms = [dict() for _ in range(nc)]
        env = {}
        logits = None
        if cl < 0:
            outs = [self._q_input(fmt_for(fl)(cur)) for fl in fls]
            for c, fl in enumerate(fls):
                terms[c][cur] = (self.x0_nhwc, fmt_for(fl)(cur), N, self.hw * self.hw * self.cin)
            stacked = {"input": self._stack(outs)}
        else:
            env["input"] = self._q_input(self.fmt[("input", "a")])
            for i in range(cl):
                env[self.layers[i]["name"]] = self._fixed_layer(i, self.layers[i], env)
            L_ = self.layers[cl]
            nm = L_["name"]
            last = cl == len(self.layers) - 1
            outs, lgs = [], []
            for c, fl in enumerate(fls):
                fo = fmt_for(fl)
                if L_["type"] == "conv":
                    y, xa, lg = self._conv_q(cl, L_, env, fo, is_q, last)
                    terms[c][(nm, "w")] = (self.W[nm][0], fo((nm, "w")), 1, self.W[nm][0].numel())
                    terms[c][(nm, "b")] = (self.W[nm][1], fo((nm, "b")), 1, self.W[nm][1].numel())
                else:
                    y, xa = self._other_q(cl, L_, env, fo((nm, "a")))
                    lg = None
                if last:
                    lgs.append(lg)
                else:
                    terms[c][(nm, "a")] = (xa, fo((nm, "a")), N, env_size(y))
                    outs.append(y)
            if last:
                n = lgs[0].numel()
                logits = torch.empty(n * nc, dtype=lgs[0].dtype, device=self.dev)
                for c, lg in enumerate(lgs):
                    logits[c * n:(c + 1) * n].copy_(lg.reshape(-1)[:n])
                return terms, logits
            stacked = {nm: self._stack(outs)}
        # every later layer in FP32 over the stacked batch; an entry of the prefix is repeated on first use
        senv = _Stacked(self, env, nc, stacked)
        for i in range(cl + 1, len(self.layers)):
            L_ = self.layers[i]
            nm = L_["name"]
            y = self._f_layer(i, L_, senv, N * nc)
            senv[nm] = y
            n = N * env_size(y)
            if L_["type"] == "conv":
                for c in range(nc):
                    terms[c][(nm, "w")] = (self.W[nm][0], self.fmt[(nm, "w")], 1, self.W[nm][0].numel())
                    terms[c][(nm, "b")] = (self.W[nm][1], self.fmt[(nm, "b")], 1, self.W[nm][1].numel())
            if i == len(self.layers) - 1:
                logits = y.t
            elif L_["type"] != "maxpool":
                for c in range(nc):
                    terms[c][(nm, "a")] = (y.t[c * n:(c + 1) * n], self.fmt[(nm, "a")], N, env_size(y))
        return terms, logits

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
    def costs(self, cur, fls):
        """(F, E, UnClass, MisPred) for each candidate FL of data-structure cur (Eq.
        quantization_parameters_optimization): the candidates' mixed forwards together, the statistics of
        every term of layers cur's and later (Eq. CPB_QE) in one batch, the tie counts of the logits, and
        every candidate's cost on the device; one read-back."""
        terms, logits = self._forward_candidates(cur, fls)
        nc = len(fls)
        start = self.names.index(cur[0])
        layout = []  # (data-structure, n_samples, nu, record offset, layer) -- the same for every candidate
        off = 0
        for li, nm in enumerate(self.names[start:]):
            for j in ("a", "w", "b"):
                if (nm, j) in terms[0]:
                    _, _, n_s, nu = terms[0][(nm, j)]
                    layout.append(((nm, j), n_s, nu, off, li))
                    off += 3 + 2 * n_s
        n_cls = self.layers[-1]["K"]
        stats = self._empty(off * nc, torch.float64)
        items = [(terms[c][ds][0].reshape(-1), n_s, nu, terms[c][ds][1], stats[c * off + o:c * off + o + 3 + 2 * n_s])
                 for c in range(nc) for ds, n_s, nu, o, _ in layout]
        F.fxpq_ds_stats_batch(items, self.stream)
        ties = self._empty(nc * self.N, torch.int32)
        F.fxpq_top1_ties(logits, nc * self.N, n_cls, ties, self.stream)
        cost = self._empty(4 * nc, torch.float64)
        F.fxpq_fopt_cost(stats, off, [(o, nu, n_s, li) for _, n_s, nu, o, li in layout], ties, self.N, n_cls, nc, cost,
                         self.stream)
        h = cost.cpu().tolist()
        return [tuple(h[4 * c:4 * c + 4]) for c in range(nc)]

    def cost(self, cur, cand_fl):
        """F, E, UnClass, MisPred for one candidate FL."""
        return self.costs(cur, [cand_fl])[0]

    # ------------------------------------------------------------------ Alg. 1 and the forward optimizer
    def qparams_opt(self, cur, K=1):
        """Alg. 1 for data-structure cur: its FL moves away from the initial one in each direction at a fixed
        wordlength, and a candidate is accepted only when it lowers the best cost so far.  Each direction
        takes at least K steps (fewer only at the ends of the FL range), so the initial FL and those 2K
        neighbours are scored as one batch; every accepted step lets its direction go one step further.
        Returns (best FL, its cost, [(FL, cost)] in the order the algorithm visits them)."""
        init = self.fmt[cur].fl
        ring = [init] + [init + d * k for d in (-1, 1) for k in range(1, K + 1) if FL_MIN <= init + d * k <= FL_MAX]
        seen = {fl: c[0] for fl, c in zip(ring, self.costs(cur, ring))}
        best_fl, best = init, seen[init]
        trace = [(init, best)]
        for d in (-1, 1):
            reach, k = K, 1
            while k <= reach and FL_MIN <= init + d * k <= FL_MAX:
                fl = init + d * k
                if fl not in seen:
                    seen[fl] = self.cost(cur, fl)[0]
                trace.append((fl, seen[fl]))
                if seen[fl] < best:
                    best, best_fl, reach = seen[fl], fl, reach + 1
                k += 1
        return best_fl, best, trace

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


class _Stacked(dict):
    """Entries over the candidates' stacked batch; an entry of the candidate-independent prefix is repeated
    once per candidate on first use."""

    def __init__(self, opt, base, nc, init):
        super().__init__(init)
        self.opt, self.base, self.nc = opt, base, nc

    def __missing__(self, key):
        v = self.opt._stack([self.base[key]] * self.nc)
        self[key] = v
        return v


def env_size(v):
    return v.H * v.W * v.C
