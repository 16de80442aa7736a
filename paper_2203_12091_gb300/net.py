"""Host-side planning of an integer-only network: parameter quantization, calibration of the
activation formats, and the op list handed to ``fxpq_net_forward`` (Sec. IV-A.2).

A layer list is a list of dicts (the format the workload generators produce):
  {"type": "conv", "name", "C", "K", "R", "stride", "pad", "relu", "src"[, "bn"]}   (FC = conv over the map)
  {"type": "maxpool", "name", "k", "stride", "pad"}
  {"type": "eltwise", "name", "a", "b", "relu"}
  {"type": "avgpool", "name", "src"}
``src`` (or ``a``/``b``) names the producing layer; ``None`` means the previous layer, and
"input" is the network input.  The last layer must be a conv/FC: it has no FxP-QLayer.

A conv with "bn" is followed by a BatchNorm layer, which becomes a Scale layer (Sec. IV-A.1): its
aleph1 / aleph2 are computed by ``fxpq_bn_to_scale``, searched and quantized like weights and biases,
and applied in the conv's epilogue.

Calibration follows the forward optimizer's order (Sec. IV-C): layer by layer, weights' FL, then
bias FL, then the output activation FL; each FL comes from ``fxpq_fl_search`` at the planned
wordlength over FL in [-8, 23], sign strategy by Sec. IV-A.3; activation FLs are searched on the
fp32 image of the exact C-Block output of the calibration slice, with every preceding layer
already quantized.  Every arithmetic step runs in libfxpq.so; this module only sequences calls
and reads back the chosen formats.
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib as L
from . import fxpq as F

FL_LO, FL_HI = -8, 23
BN_EPS = 1e-5  # the BatchNorm epsilon of the rewritten layers (Caffe's and torchvision's default)


def pad8(c: int) -> int:
    return (c + 7) // 8 * 8


REC = 64  # bytes per search result record: int32 best FL at 0, fxpq_stats at 8


def launch_searches(items, res, stream=None):
    """FL searches at one wordlength each, as one batch (fxpq_fl_search_batch), results into the device
    uint8 buffer `res` (REC bytes per item); nothing is read back."""
    dev = items[0][0].device
    nfl = FL_HI - FL_LO + 1
    err = torch.empty(len(items) * nfl, dtype=torch.float64, device=dev)
    ws = F.workspace(F.fxpq_fl_search_batch_workspace(len(items)), dev)
    base = res.data_ptr()
    batch = []
    for i, (x, k) in enumerate(items):
        x = x.reshape(-1)
        batch.append(L.FlSearchItem(x.data_ptr(), x.numel(), -1, k, k, FL_LO, FL_HI, err.data_ptr() + 8 * nfl * i,
                                    base + REC * i, base + REC * i + 8))
    F.fxpq_fl_search_batch(batch, ws, stream)


def decode_fmts(host: bytes, ks):
    """The chosen (k, S, FL) per search from the read-back result records (sign strategy of Sec. IV-A.3)."""
    out = []
    for i, k in enumerate(ks):
        best = int.from_bytes(host[REC * i:REC * i + 4], "little", signed=True)
        st = L.Stats.from_buffer_copy(host[REC * i + 8:REC * i + 8 + ctypes.sizeof(L.Stats)])
        out.append(F.fmt(k, st.is_signed, best))
    return out


def search_fmts(items, stream=None):
    """FL searches at one wordlength each, as one batch; one device-to-host read.

    items: list of (tensor, k).  Returns the chosen (k, S, FL) per item."""
    if not items:
        return []
    res = torch.empty(len(items) * REC, dtype=torch.uint8, device=items[0][0].device)
    launch_searches(items, res, stream)
    return decode_fmts(bytes(res.cpu().numpy().tobytes()), [k for _, k in items])


def search_fmt(x: torch.Tensor, k: int, stream=None) -> L.Fmt:
    """FL search at one wordlength; returns the chosen (k, S, FL).  Synchronises once."""
    return search_fmts([(x, k)], stream)[0]


class QNet:
    """A quantized network on one device: code tensors, formats, and the fxpq_net op list."""

    def __init__(self, layers, hw=224, cin=3, pack_weights=False):
        self.layers = layers
        self.hw, self.cin = hw, cin
        self.cp_in = pad8(cin)
        self.fmts = {}
        self.q = {}  # name -> (weight fp16 codes, bias int32 codes or None)
        # name -> packed k-bit weights (fxpq_pack_weights) of FC and 1x1 layers with k <= 8, which the
        # contraction reads instead of the fp16 codes (Sec. V-E.2: k bits per read-only value); built
        # when pack_weights is set (they halve or better the FC layers' weight reads, while the
        # in-kernel expansion costs FC time at present)
        self.qp = {}
        self.pack_weights = pack_weights
        self.qs = {}  # BN conv name -> (aleph1 int32 codes, aleph2 int32 codes)
        self.w_l1 = {}  # conv name -> max over output channels of sum |weight code| (0: unknown)
        self.names = ["input"] + [L_["name"] for L_ in layers]
        self.slot = {nm: i for i, nm in enumerate(self.names)}
        self.shapes = {}

    # ------------------------------------------------------------------ parameters
    def _src(self, i, L_, key="src"):
        s = L_.get(key)
        return s if s is not None else (self.names[i] if i > 0 else "input")

    def quantize_params(self, weights_dev, plan, stream=None, bn_dev=None):
        """weights_dev: name -> (fp32 KRSC weight, fp32 bias or None) device tensors; plan: wordlengths;
        bn_dev: BN conv name -> (gamma, beta, running mean, running variance) fp32 device tensors.

        Every parameter's FL search runs as one batch, every quantization as one launch reading the
        chosen formats on the device, and one read-back returns the formats and the L1 bounds."""
        shapes = {"input": (self.hw, self.hw, self.cp_in)}
        searches, owners = [], []
        dev = next(iter(weights_dev.values()))[0].device
        recips, alephs = {}, {}
        for i, L_ in enumerate(self.layers):
            nm = L_["name"]
            self.fmts.setdefault(nm, {})
            if L_["type"] == "conv":
                H, W, Cp = shapes[self._src(i, L_)]
                w, b = weights_dev[nm]
                K, R, _, C = w.shape
                assert C <= Cp
                searches.append((w, plan[nm]["w"]))
                owners.append((nm, "w"))
                if b is not None:
                    searches.append((b, plan[nm]["b"]))
                    owners.append((nm, "b"))
                if L_.get("bn"):
                    a1 = torch.empty(K, dtype=torch.float32, device=dev)
                    a2 = torch.empty(K, dtype=torch.float32, device=dev)
                    F.fxpq_bn_to_scale(*bn_dev[nm], BN_EPS, a1, a2, stream)
                    alephs[nm] = (a1, a2)
                    searches += [(a1, plan[nm]["s"]), (a2, plan[nm]["h"])]
                    owners += [(nm, "s"), (nm, "h")]
                P = (H + 2 * L_["pad"] - R) // L_["stride"] + 1
                shapes[nm] = (P, P, K)
            elif L_["type"] == "maxpool":
                H, W, Cp = shapes[self._src(i, L_)]
                P = (H + 2 * L_["pad"] - L_["k"]) // L_["stride"] + 1
                shapes[nm] = (P, P, Cp)
            elif L_["type"] == "eltwise":
                shapes[nm] = shapes[L_["a"]]
            elif L_["type"] == "avgpool":
                H, W, Cp = shapes[self._src(i, L_)]
                r = torch.tensor([1.0 / (H * W)], dtype=torch.float32, device=dev)
                recips[nm] = r
                searches.append((r, plan[nm]["r"]))
                owners.append((nm, "r"))
                shapes[nm] = (1, 1, Cp)
        # One buffer read back once: the search records, then the weight-code L1 bounds (int64 per
        # conv layer), then the avg-pool reciprocal codes (int32).  The quantization reads each
        # tensor's S and FL from the search records on the device (fxpq_quantize_batch).
        conv_names = [L_["name"] for L_ in self.layers if L_["type"] == "conv"]
        avg_names = [L_["name"] for L_ in self.layers if L_["type"] == "avgpool"]
        n_s = len(searches)
        off_l1 = n_s * REC
        off_rc = off_l1 + 8 * len(conv_names)
        buf = torch.zeros(off_rc + 4 * len(avg_names) + 8, dtype=torch.uint8, device=dev)
        launch_searches(searches, buf, stream)
        base = buf.data_ptr()
        rec = {key: base + REC * i for i, key in enumerate(owners)}
        items = []
        for i, L_ in enumerate(self.layers):
            nm = L_["name"]
            if L_["type"] == "conv":
                w, b = weights_dev[nm]
                K, R, _, C = w.shape
                Cp = shapes[self._src(i, L_)][2]
                kw, kb = plan[nm]["w"], plan[nm].get("b")
                wq = torch.empty(K * R * R * Cp * (2 if kw > 8 else 1), dtype=torch.float16, device=dev)
                l1p = base + off_l1 + 8 * conv_names.index(nm) if kw <= 8 else None
                items.append(L.QuantizeItem(w.data_ptr(), wq.data_ptr(), L.QB_ROWS_F16, kw, K * R * R, C, Cp, R * R, 0,
                                            rec[(nm, "w")], rec[(nm, "w")] + 8, l1p))
                bq = None
                if b is not None:
                    bq = torch.empty(K, dtype=torch.int32, device=dev)
                    items.append(L.QuantizeItem(b.data_ptr(), bq.data_ptr(), L.QB_FLAT_I32, kb, K, 0, 0, 1, 0,
                                                rec[(nm, "b")], rec[(nm, "b")] + 8, None))
                self.q[nm] = (wq, bq)
                if nm in alephs:
                    codes = []
                    for key, t in zip(("s", "h"), alephs[nm]):
                        c = torch.empty(K, dtype=torch.int32, device=dev)
                        items.append(L.QuantizeItem(t.data_ptr(), c.data_ptr(), L.QB_FLAT_I32, plan[nm][key], K, 0, 0,
                                                    1, 0, rec[(nm, key)], rec[(nm, key)] + 8, None))
                        codes.append(c)
                    self.qs[nm] = tuple(codes)
            elif L_["type"] == "avgpool":
                items.append(L.QuantizeItem(recips[nm].data_ptr(), base + off_rc + 4 * avg_names.index(nm),
                                            L.QB_FLAT_I32, plan[nm]["r"], 1, 0, 0, 1, 0,
                                            rec[(nm, "r")], rec[(nm, "r")] + 8, None))
        F.fxpq_quantize_batch(items, stream)
        host = bytes(buf.cpu().numpy().tobytes())
        for (nm, key), f in zip(owners, decode_fmts(host, [k for _, k in searches])):
            self.fmts[nm][key] = f
        self.w_l1 = {nm: int.from_bytes(host[off_l1 + 8 * j:off_l1 + 8 * j + 8], "little", signed=True)
                     for j, nm in enumerate(conv_names)}
        self.qp = {}
        for i, L_ in enumerate(self.layers):
            nm = L_["name"]
            if not self.pack_weights or L_["type"] != "conv" or plan[nm]["w"] > 8:
                continue
            H, _, Cp = shapes[self._src(i, L_)]
            R, st, pad = L_["R"], L_["stride"], L_["pad"]
            if pad == 0 and ((R == 1 and st == 1) or (R == H and shapes[nm][0] == 1)):
                self.qp[nm] = F.pack_weights(self.q[nm][0], self.fmts[nm]["w"], L_["K"], R * R * Cp, stream)
        for j, nm in enumerate(avg_names):
            self.q[nm] = (None, int.from_bytes(host[off_rc + 4 * j:off_rc + 4 * j + 4], "little", signed=True))
        self.shapes = shapes

    # ------------------------------------------------------------------ one C-Block on device tensors
    def run_layer(self, i, env, N, out_mode, stream=None):
        """Run layer i on env[name] = (tensor, fmt); returns (output tensor, scale exponent)."""
        L_ = self.layers[i]
        nm = L_["name"]
        H, W, Cp = self.shapes[nm]
        fy = self.fmts[nm].get("a")
        if out_mode == F.OUT_CODES:
            y = torch.empty(N * H * W * Cp * F.planes(fy), dtype=torch.float16, device=self._dev)
        elif out_mode == F.OUT_F32:
            y = torch.empty(N * H * W * Cp, dtype=torch.float32, device=self._dev)
        else:
            y = torch.empty(N * H * W * Cp, dtype=torch.int64, device=self._dev)
        if L_["type"] == "conv":
            src = self._src(i, L_)
            x, fx = env[src]
            sH, sW, sCp = self.shapes[src]
            wq, bq = self.q[nm]
            sq, hq = self.qs.get(nm, (None, None))
            d = F.conv_desc(N, sH, sW, sCp, sCp, L_["K"], L_["R"], L_["R"], L_["stride"], L_["pad"], L_["relu"],
                            out_mode, fx, self.fmts[nm]["w"], self.fmts[nm].get("b"), fy, self.w_l1.get(nm, 0),
                            scale=sq, fmt_scale=self.fmts[nm].get("s"), shift=hq, fmt_shift=self.fmts[nm].get("h"),
                            wpacked=self.qp.get(nm))
            nws = F.fxpq_conv_workspace(d)
            if nws and (getattr(self, "_cws", None) is None or self._cws.numel() < nws):
                self._cws = torch.empty(nws, dtype=torch.uint8, device=self._dev)
            s = F.fxpq_conv_fwd(d, x, wq, bq, y, stream, ws=self._cws if nws else None)
        elif L_["type"] == "maxpool":
            src = self._src(i, L_)
            x, fx = env[src]
            sH, sW, sCp = self.shapes[src]
            F.fxpq_maxpool(x, N, sH, sW, sCp, fx, L_["k"], L_["stride"], L_["pad"], y, stream)
            s = fx.fl
        elif L_["type"] == "eltwise":
            (a, fa), (b, fb) = env[L_["a"]], env[L_["b"]]
            s = F.fxpq_eltwise(a, fa, b, fb, N * H * W, Cp, L_["relu"], out_mode, fy, y, stream)
        elif L_["type"] == "avgpool":
            src = self._src(i, L_)
            x, fx = env[src]
            sH, sW, sCp = self.shapes[src]
            s = F.fxpq_avgpool(x, N, sH, sW, sCp, fx, self.q[nm][1], self.fmts[nm]["r"], out_mode, fy, y, stream)
        else:
            raise ValueError(L_["type"])
        return y, s

    # ------------------------------------------------------------------ calibration (Sec. IV-C order)
    def calibrate(self, calib_images, plan, stream=None):
        """Activation formats in the forward optimizer's order, by fxpq_net_calibrate on the op list (the
        planned wordlengths in, the searched S and FL out); then the final op list."""
        self._dev = calib_images.device
        N = calib_images.shape[0]
        last = len(self.layers) - 1
        self.fmts["input"] = {"a": F.fmt(plan["input"], 0, 0)}
        for i, L_ in enumerate(self.layers):
            if i < last and L_["type"] != "maxpool":
                self.fmts[L_["name"]]["a"] = F.fmt(plan[L_["name"]]["a"], 0, 0)
        self._build_ops()
        ws = F.workspace(F.fxpq_net_calibrate_workspace(self.net, N), self._dev)
        fin, fys = F.fxpq_net_calibrate(self.net, calib_images, N, FL_LO, FL_HI, ws, stream)
        self.fmts["input"]["a"] = fin
        for i, L_ in enumerate(self.layers):
            if i < last:
                self.fmts[L_["name"]]["a"] = fys[i]
        self._build_ops()
        return self.fmts

    # ------------------------------------------------------------------ forward through the C ABI
    def _build_ops(self):
        ops = (L.OpDesc * len(self.layers))()
        last = len(self.layers) - 1
        for i, L_ in enumerate(self.layers):
            o = ops[i]
            nm = L_["name"]
            o.dst = 0 if i == last else self.slot[nm]
            o.last = 1 if i == last else 0
            o.src1 = -1
            if L_["type"] == "conv":
                o.op = L.OP_CONV
                o.src0 = self.slot[self._src(i, L_)]
                o.K, o.R, o.S, o.stride, o.pad, o.relu = L_["K"], L_["R"], L_["R"], L_["stride"], L_["pad"], int(L_["relu"])
                o.fmt_w, o.fmt_b = self.fmts[nm]["w"], self.fmts[nm].get("b", L.Fmt(32, 1, 0))
                o.fmt_y = self.fmts[nm].get("a", L.Fmt(8, 1, 0))
                o.d_w = self.q[nm][0].data_ptr()
                o.d_bias = self.q[nm][1].data_ptr() if self.q[nm][1] is not None else None
                o.w_l1 = self.w_l1.get(nm, 0)
                o.d_wpacked = self.qp[nm].data_ptr() if nm in self.qp else None
                if nm in self.qs:
                    o.fmt_scale, o.fmt_shift = self.fmts[nm]["s"], self.fmts[nm]["h"]
                    o.d_scale, o.d_shift = self.qs[nm][0].data_ptr(), self.qs[nm][1].data_ptr()
            elif L_["type"] == "maxpool":
                o.op = L.OP_MAXPOOL
                o.src0 = self.slot[self._src(i, L_)]
                o.R = o.S = L_["k"]
                o.stride, o.pad = L_["stride"], L_["pad"]
            elif L_["type"] == "eltwise":
                o.op = L.OP_ELTWISE
                o.src0, o.src1 = self.slot[L_["a"]], self.slot[L_["b"]]
                o.relu = int(L_["relu"])
                o.fmt_y = self.fmts[nm]["a"]
            elif L_["type"] == "avgpool":
                o.op = L.OP_AVGPOOL
                o.src0 = self.slot[self._src(i, L_)]
                o.recip_code = self.q[nm][1]
                o.fmt_w = self.fmts[nm]["r"]
                o.fmt_y = self.fmts[nm]["a"]
        self._ops = ops
        self.net = L.Net(len(self.layers), len(self.names), self.cin, self.hw, self.hw, self.cp_in,
                         self.fmts["input"]["a"], ctypes.cast(ops, ctypes.POINTER(L.OpDesc)))
        self.n_classes = self.layers[-1]["K"]

    def memory(self):
        """Memory requirement of one inference (Sec. V-E.2): RW_R / RO_R in MB for the FxP network and
        its FP32 baseline, and the compression rates COMP_Act and COMP_Model."""
        rw_q, ro_q = F.fxpq_net_memory(self.net, False)
        rw_f, ro_f = F.fxpq_net_memory(self.net, True)
        return {"rw_mb": rw_q, "ro_mb": ro_q, "rw_fp32_mb": rw_f, "ro_fp32_mb": ro_f,
                "comp_act": rw_f / rw_q, "comp_model": ro_f / ro_q}

    def workspace_bytes(self, batch: int) -> int:
        return F.fxpq_net_workspace(self.net, batch)

    def forward(self, images, logits=None, ws=None, stream=None):
        """images: fp32 NCHW device tensor.  Returns (int64 logits [N, classes], scale exponent)."""
        N = images.shape[0]
        if logits is None:
            logits = torch.empty(N, self.n_classes, dtype=torch.int64, device=images.device)
        if ws is None:
            ws = F.workspace(self.workspace_bytes(N), images.device)
        s = F.fxpq_net_forward(self.net, images, N, logits, ws, stream)
        return logits, s

    def trace(self, images, stream=None):
        """Per-layer outputs (codes) of a forward with frozen formats, op by op (for parity tests)."""
        self._dev = images.device
        N = images.shape[0]
        fin = self.fmts["input"]["a"]
        x0 = torch.empty(N * self.hw * self.hw * self.cp_in * F.planes(fin), dtype=torch.float16, device=self._dev)
        F.fxpq_quantize_images(images, fin, self.cp_in, x0, stream)
        env = {"input": (x0, fin)}
        last = len(self.layers) - 1
        for i, L_ in enumerate(self.layers):
            nm = L_["name"]
            if i == last:
                y, s = self.run_layer(i, env, N, F.OUT_ACC64, stream)
                env[nm] = (y, s)
                break
            f = self.fmts[nm]["a"]
            y, _ = self.run_layer(i, env, N, F.OUT_CODES, stream)
            env[nm] = (y, f)
        return env


def build_qnet(layers, weights_np, calib_images, plan, device="cuda", stream=None, bn_np=None, pack_weights=False):
    """Quantize parameters and calibrate on `calib_images` (fp32 NCHW device tensor).  bn_np: BN conv
    name -> (gamma, beta, mean, var) fp32 arrays (layers with "bn").  pack_weights: FC layers with
    k <= 8 read packed k-bit weights."""
    wdev = {nm: (torch.from_numpy(w).to(device), None if b is None else torch.from_numpy(b).to(device))
            for nm, (w, b) in weights_np.items()}
    bn_dev = {nm: tuple(torch.from_numpy(t).to(device) for t in v) for nm, v in (bn_np or {}).items()}
    q = QNet(layers, hw=calib_images.shape[-1], cin=calib_images.shape[1], pack_weights=pack_weights)
    q._dev = torch.device(device)
    q.quantize_params(wdev, plan, stream, bn_dev)
    q.calibrate(calib_images, plan, stream)
    q.weights_dev = wdev
    return q
