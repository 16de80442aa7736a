"""Python binding of libfxpq.so: same names as include/fxpq.h, torch tensors in, argument
marshalling only.  PyTorch provides device memory and streams; every step runs in the library's
CUDA kernels.
"""
from __future__ import annotations

import ctypes

import torch

from . import _lib as L
from ._lib import DT_F16, DT_I8, DT_I16, DT_I32, DT_U8, DT_U16, OUT_ACC64, OUT_CODES, OUT_F32, Fmt, Stats  # noqa: F401


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _s(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def fmt(bits: int, is_signed: int, fl: int) -> Fmt:
    return Fmt(int(bits), int(is_signed), int(fl))


def planes(f: Fmt) -> int:
    return 2 if f.bits > 8 else 1


_WS = {}


def workspace(nbytes: int, device=None) -> torch.Tensor:
    """A cached uint8 device buffer of at least nbytes (256-byte aligned by the allocator)."""
    dev = torch.device(device) if device is not None else torch.device("cuda", torch.cuda.current_device())
    t = _WS.get(dev)
    if t is None or t.numel() < nbytes:
        t = torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=dev)
        _WS[dev] = t
    return t


# ------------------------------------------------------------------------------ quantizer
def fxpq_quantize(x, f: Fmt, dtype: int, out, stream=None):
    L.check("fxpq_quantize", L.lib().fxpq_quantize(_p(x), x.numel(), f, dtype, _p(out), _s(stream)))
    return out


def fxpq_quantize_rows(x, rows: int, C: int, f: Fmt, Cp: int, out, stream=None):
    L.check("fxpq_quantize_rows", L.lib().fxpq_quantize_rows(_p(x), rows, C, f, Cp, _p(out), _s(stream)))
    return out


def fxpq_code_l1max(codes, rows: int, L_: int, out, stream=None):
    """max_r sum_j |codes[r, j]| of a one-plane fp16 code tensor [rows, L_] into the int64 device
    tensor `out` (one element)."""
    L.check("fxpq_code_l1max", L.lib().fxpq_code_l1max(_p(codes), rows, L_, _p(out), _s(stream)))
    return out


def fxpq_quantize_images(x_nchw, f: Fmt, c_pad: int, out, stream=None):
    N, C, H, W = x_nchw.shape
    L.check("fxpq_quantize_images",
            L.lib().fxpq_quantize_images(_p(x_nchw), N, C, H, W, f, c_pad, _p(out), _s(stream)))
    return out


# ------------------------------------------------------------------------------ FL search
def fxpq_fl_search_workspace(n: int) -> int:
    return int(L.lib().fxpq_fl_search_workspace(n))


def fxpq_fl_search(x, is_signed: int, k_lo: int, k_hi: int, fl_lo: int, fl_hi: int, err, best, stats, ws, stream=None):
    L.check("fxpq_fl_search",
            L.lib().fxpq_fl_search(_p(x), x.numel(), is_signed, k_lo, k_hi, fl_lo, fl_hi, _p(err), _p(best),
                                   _p(stats), _p(ws), ws.numel(), _s(stream)))


def fl_search(x, is_signed: int, k_lo: int, k_hi: int, fl_lo: int, fl_hi: int, stream=None, score: str = "l2"):
    """Allocate the outputs and run fxpq_fl_search (score "l2"), or a one-item fxpq_fl_search_batch with
    the L1 score (score "l1").  Returns device (err[nk, nfl], best[nk], stats bytes)."""
    nk, nfl = k_hi - k_lo + 1, fl_hi - fl_lo + 1
    dev = x.device
    err = torch.empty(nk * nfl, dtype=torch.float64, device=dev)
    best = torch.empty(nk, dtype=torch.int32, device=dev)
    stats = torch.empty(ctypes.sizeof(Stats), dtype=torch.uint8, device=dev)
    if score == "l2":
        ws = workspace(fxpq_fl_search_workspace(x.numel()), dev)
        fxpq_fl_search(x, is_signed, k_lo, k_hi, fl_lo, fl_hi, err, best, stats, ws, stream)
    else:
        item = L.FlSearchItem(x.data_ptr(), x.numel(), is_signed, k_lo, k_hi, fl_lo, fl_hi, err.data_ptr(),
                              best.data_ptr(), stats.data_ptr(), {"l1": L.SCORE_L1}[score])
        fxpq_fl_search_batch([item], workspace(fxpq_fl_search_batch_workspace(1), dev), stream)
    return err.view(nk, nfl), best, stats


def fxpq_fl_search_batch_workspace(n_items: int) -> int:
    return L.lib().fxpq_fl_search_batch_workspace(n_items)


def fxpq_fl_search_batch(items, ws, stream=None):
    """items: list of L.FlSearchItem (device pointers filled in).  ws: a device workspace tensor."""
    arr = (L.FlSearchItem * len(items))(*items)
    L.check("fxpq_fl_search_batch", L.lib().fxpq_fl_search_batch(
        ctypes.cast(arr, ctypes.c_void_p), len(items), _p(ws), ws.numel() * ws.element_size(), _s(stream)))


def fxpq_quantize_batch(items, stream=None):
    """items: list of L.QuantizeItem (device pointers filled in)."""
    arr = (L.QuantizeItem * len(items))(*items)
    L.check("fxpq_quantize_batch", L.lib().fxpq_quantize_batch(ctypes.cast(arr, ctypes.c_void_p), len(items),
                                                                _s(stream)))


def fxpq_net_calibrate_workspace(net, n_calib: int) -> int:
    return L.lib().fxpq_net_calibrate_workspace(ctypes.byref(net), n_calib)


def fxpq_net_calibrate(net, calib_nchw, n_calib: int, fl_lo: int, fl_hi: int, ws, stream=None):
    """Returns (input format, [output format per op])."""
    fin = Fmt()
    fys = (Fmt * net.n_ops)()
    L.check("fxpq_net_calibrate", L.lib().fxpq_net_calibrate(
        ctypes.byref(net), _p(calib_nchw), n_calib, fl_lo, fl_hi, ctypes.byref(fin), ctypes.cast(fys, ctypes.c_void_p),
        _p(ws), ws.numel(), _s(stream)))
    return fin, list(fys)


def stats_from_device(stats_bytes) -> Stats:
    return Stats.from_buffer_copy(bytes(stats_bytes.cpu().numpy().tobytes()))


def fxpq_fl_init(stats: Stats, bits: int, strategy: int) -> Fmt:
    out = Fmt()
    L.check("fxpq_fl_init", L.lib().fxpq_fl_init(ctypes.byref(stats), bits, strategy, ctypes.byref(out)))
    return out


def fxpq_pack_codes(codes, n: int, f: Fmt, words, stream=None):
    """fp16 code tensor of n codes -> packed k-bit words (ceil(n / 32) * f.bits uint32)."""
    L.check("fxpq_pack_codes", L.lib().fxpq_pack_codes(_p(codes), n, f, _p(words), _s(stream)))
    return words


def fxpq_unpack_codes(words, n: int, f: Fmt, codes, stream=None):
    L.check("fxpq_unpack_codes", L.lib().fxpq_unpack_codes(_p(words), n, f, _p(codes), _s(stream)))
    return codes


def fxpq_packed_weights_bytes(fw: Fmt, K: int, Lw: int) -> int:
    return L.lib().fxpq_packed_weights_bytes(fw, K, Lw)


def fxpq_pack_weights(w, fw: Fmt, K: int, Lw: int, packed, stream=None):
    """One plane of fp16 weight codes [K][Lw] (fw.bits <= 8) -> the contraction's packed records."""
    L.check("fxpq_pack_weights", L.lib().fxpq_pack_weights(_p(w), fw, K, Lw, _p(packed), _s(stream)))
    return packed


def pack_weights(w, fw: Fmt, K: int, Lw: int, stream=None):
    """Allocates and fills the packed copy of the weights (a uint8 device tensor)."""
    import torch
    n = fxpq_packed_weights_bytes(fw, K, Lw)
    packed = torch.empty(n, dtype=torch.uint8, device=w.device)
    return fxpq_pack_weights(w, fw, K, Lw, packed, stream)


def packed_words(n: int, f: Fmt) -> int:
    return (n + 31) // 32 * f.bits


def fxpq_net_memory(net, fp32: bool):
    """(RW_R, RO_R) in MB of one inference of the op list (Sec. V-E.2); host-only."""
    rw, ro = ctypes.c_double(0), ctypes.c_double(0)
    L.check("fxpq_net_memory", L.lib().fxpq_net_memory(ctypes.byref(net), int(fp32), ctypes.byref(rw), ctypes.byref(ro)))
    return rw.value, ro.value


# ------------------------------------------------------------------------------ forward optimizer support
def fxpq_conv_f32(N, H, W, C, K, R, S, stride, pad, relu, x, w, bias, y, stream=None):
    d = L.ConvF32Desc(N, H, W, C, K, R, S, stride, pad, int(relu))
    L.check("fxpq_conv_f32", L.lib().fxpq_conv_f32(ctypes.byref(d), _p(x), _p(w), _p(bias), _p(y), _s(stream)))
    return y


def fxpq_maxpool_f32(x, N, H, W, C, k, stride, pad, y, stream=None):
    L.check("fxpq_maxpool_f32", L.lib().fxpq_maxpool_f32(_p(x), N, H, W, C, k, stride, pad, _p(y), _s(stream)))
    return y


def fxpq_eltwise_f32(a, b, n, relu, y, stream=None):
    L.check("fxpq_eltwise_f32", L.lib().fxpq_eltwise_f32(_p(a), _p(b), n, int(relu), _p(y), _s(stream)))
    return y


def fxpq_avgpool_f32(x, N, H, W, C, y, stream=None):
    L.check("fxpq_avgpool_f32", L.lib().fxpq_avgpool_f32(_p(x), N, H, W, C, _p(y), _s(stream)))
    return y


def fxpq_nchw_to_nhwc_f32(x, N, C, H, W, y, stream=None):
    L.check("fxpq_nchw_to_nhwc_f32", L.lib().fxpq_nchw_to_nhwc_f32(_p(x), N, C, H, W, _p(y), _s(stream)))
    return y


def fxpq_dequantize(codes, npix, Cp, C, f: Fmt, y, stream=None):
    L.check("fxpq_dequantize", L.lib().fxpq_dequantize(_p(codes), npix, Cp, C, f, _p(y), _s(stream)))
    return y


def fxpq_bias_relu_f32(y, npix, K, bias, relu, stream=None):
    L.check("fxpq_bias_relu_f32", L.lib().fxpq_bias_relu_f32(_p(y), npix, K, _p(bias), int(relu), _s(stream)))
    return y


def fxpq_ds_stats_batch(items, stream=None):
    """items: list of (fp32 device tensor, n_samples, nu, Fmt, record: device float64[3 + 2 n_samples])."""
    arr = (L.DsItem * len(items))(*[L.DsItem(x.data_ptr(), out.data_ptr(), nu, ns, f) for x, ns, nu, f, out in items])
    nbytes = L.lib().fxpq_ds_stats_batch_workspace(arr, len(items))
    if nbytes == 0:
        raise L.FxpqError("fxpq_ds_stats_batch_workspace", L.ERR_INVALID_ARG)
    dev = items[0][0].device
    L.check("fxpq_ds_stats_batch", L.lib().fxpq_ds_stats_batch(arr, len(items), _p(workspace(nbytes, dev)), nbytes,
                                                               _s(stream)))


def fxpq_fopt_cost(stats, cand_stride, terms, ties, N, n_classes, n_cand, cost, stream=None):
    """terms: list of (record offset in doubles, nu, n_samples, layer); cost: device float64[n_cand * 4]."""
    arr = (L.CostTerm * max(len(terms), 1))(*[L.CostTerm(o, nu, ns, ly) for o, nu, ns, ly in terms])
    L.check("fxpq_fopt_cost", L.lib().fxpq_fopt_cost(_p(stats), cand_stride, arr, len(terms), _p(ties), N, n_classes,
                                                     n_cand, _p(cost), _s(stream)))
    return cost


def fxpq_top1_ties(logits, N, C, counts, stream=None):
    is64 = 1 if logits.dtype == torch.int64 else 0
    L.check("fxpq_top1_ties", L.lib().fxpq_top1_ties(_p(logits), is64, N, C, _p(counts), _s(stream)))
    return counts


def fxpq_bn_to_scale(gamma, beta, mean, var, eps, aleph1, aleph2, stream=None):
    """BN -> Scale layer parameters (fp32 device tensors of one length)."""
    L.check("fxpq_bn_to_scale", L.lib().fxpq_bn_to_scale(_p(gamma), _p(beta), _p(mean), _p(var), gamma.numel(),
                                                          float(eps), _p(aleph1), _p(aleph2), _s(stream)))
    return aleph1, aleph2


# ------------------------------------------------------------------------------ C-Blocks
def conv_desc(N, H, W, C, Cp, K, R, S, stride, pad, relu, out_mode, fx, fw, fb, fy, w_l1=0,
              scale=None, fmt_scale=None, shift=None, fmt_shift=None, wpacked=None) -> L.ConvDesc:
    """C-Block descriptor.  scale / shift: int32 aleph1 / aleph2 code tensors [K] of a Scale layer (both
    or neither; the caller keeps them alive while the descriptor is used).  wpacked: optional packed
    copy of the weights (fxpq_pack_weights)."""
    return L.ConvDesc(N, H, W, C, Cp, K, R, S, stride, pad, int(relu), out_mode, fx, fw,
                      fb if fb is not None else Fmt(32, 1, 0), fy if fy is not None else Fmt(8, 1, 0), int(w_l1),
                      fmt_scale if fmt_scale is not None else Fmt(16, 1, 0),
                      fmt_shift if fmt_shift is not None else Fmt(16, 1, 0), _p(scale), _p(shift), _p(wpacked))


def fxpq_conv_workspace(desc: L.ConvDesc) -> int:
    return L.lib().fxpq_conv_workspace(ctypes.byref(desc))


def fxpq_conv_fwd(desc: L.ConvDesc, x, w, bias, y, stream=None, ws=None) -> int:
    """ws: optional device workspace (fxpq_conv_workspace bytes) for the split reduction of layers with
    too few tiles for the SMs."""
    scale = L.I32(0)
    L.check("fxpq_conv_fwd", L.lib().fxpq_conv_fwd(ctypes.byref(desc), _p(x), _p(w), _p(bias), _p(y),
                                                   ctypes.byref(scale), _p(ws),
                                                   0 if ws is None else ws.numel() * ws.element_size(), _s(stream)))
    return scale.value


def fxpq_gemm(x, fx, w, fw, bias, fb, M, N, Kdim, relu, out_mode, fy, y, stream=None, ws=None) -> int:
    scale = L.I32(0)
    L.check("fxpq_gemm", L.lib().fxpq_gemm(_p(x), fx, _p(w), fw, _p(bias), fb if fb is not None else Fmt(32, 1, 0),
                                           M, N, Kdim, int(relu), out_mode, fy if fy is not None else Fmt(8, 1, 0),
                                           _p(y), ctypes.byref(scale), _p(ws),
                                           0 if ws is None else ws.numel() * ws.element_size(), _s(stream)))
    return scale.value


def fxpq_maxpool(x, N, H, W, Cp, f: Fmt, k, stride, pad, y, stream=None):
    L.check("fxpq_maxpool", L.lib().fxpq_maxpool(_p(x), N, H, W, Cp, f, k, stride, pad, _p(y), _s(stream)))
    return y


def fxpq_eltwise(a, fa: Fmt, b, fb: Fmt, n_pix, Cp, relu, out_mode, fy, y, stream=None) -> int:
    scale = L.I32(0)
    L.check("fxpq_eltwise", L.lib().fxpq_eltwise(_p(a), fa, _p(b), fb, n_pix, Cp, int(relu), out_mode,
                                                 fy if fy is not None else Fmt(8, 1, 0), _p(y), ctypes.byref(scale),
                                                 _s(stream)))
    return scale.value


def fxpq_avgpool(x, N, H, W, Cp, fx: Fmt, recip_code: int, fr: Fmt, out_mode, fy, y, stream=None) -> int:
    scale = L.I32(0)
    L.check("fxpq_avgpool", L.lib().fxpq_avgpool(_p(x), N, H, W, Cp, fx, int(recip_code), fr, out_mode,
                                                 fy if fy is not None else Fmt(8, 1, 0), _p(y), ctypes.byref(scale),
                                                 _s(stream)))
    return scale.value


def fxpq_qlayer(v, s: int, out_mode: int, fy, y, stream=None):
    L.check("fxpq_qlayer", L.lib().fxpq_qlayer(_p(v), v.numel(), int(s), out_mode,
                                               fy if fy is not None else Fmt(8, 1, 0), _p(y), _s(stream)))
    return y


def fxpq_net_workspace(net: L.Net, batch: int) -> int:
    return int(L.lib().fxpq_net_workspace(ctypes.byref(net), batch))


def fxpq_net_forward(net: L.Net, images, batch, logits, ws, stream=None) -> int:
    scale = L.I32(0)
    L.check("fxpq_net_forward", L.lib().fxpq_net_forward(ctypes.byref(net), _p(images), batch, _p(logits),
                                                         ctypes.byref(scale), _p(ws), ws.numel(), _s(stream)))
    return scale.value


def fxpq_get_device_status(stream=None) -> int:
    return int(L.lib().fxpq_get_device_status(_s(stream)))


def fxpq_launch_count() -> int:
    return int(L.lib().fxpq_launch_count())


# ------------------------------------------------------------------------------ code tensors
def codes_to_int(t: torch.Tensor, f: Fmt, shape) -> torch.Tensor:
    """Decode an fp16 code tensor (plane-major, see include/fxpq.h) to int64 codes of `shape`."""
    t = t.reshape(-1).to(torch.int64)
    if planes(f) == 1:
        return t.view(*shape)
    t = t.view(2, -1)
    return (t[0] * 256 + t[1]).view(*shape)
