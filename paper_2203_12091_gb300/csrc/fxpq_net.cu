// fxpq_net.cu -- integer-only network forward (Sec. IV-A.2: FxP-QLayers as vertices, C-Blocks as
// edges).  Host-side driver: derives every slot's shape, carves the slots out of the caller's
// workspace, and launches the C-Block kernels in order on the caller's stream.
#include <vector>

#include "fxpq_common.cuh"

namespace {

struct Slot {
    int H = 0, W = 0, Cp = 0;
    fxpq_fmt fmt{0, 0, 0};
    bool defined = false;
    size_t offset = 0, bytes = 0;
};

size_t align256(size_t v) { return (v + 255) / 256 * 256; }

fxpq_status plan_net(const fxpq_net* net, int32_t batch, std::vector<Slot>& slots, size_t& total) {
    if (!net || !net->ops || net->n_ops < 1 || net->n_slots < 1 || net->n_slots > 4096 || batch < 0)
        return FXPQ_ERR_INVALID_ARG;
    if (net->C < 1 || net->H < 1 || net->W < 1 || net->Cp_in < net->C || (net->Cp_in % 8) || !fxpq::fmt_ok(net->fmt_in))
        return FXPQ_ERR_INVALID_ARG;
    slots.assign(net->n_slots, Slot());
    slots[0].H = net->H;
    slots[0].W = net->W;
    slots[0].Cp = net->Cp_in;
    slots[0].fmt = net->fmt_in;
    slots[0].defined = true;
    for (int i = 0; i < net->n_ops; ++i) {
        const fxpq_op_desc& o = net->ops[i];
        const bool last = (i == net->n_ops - 1);
        if ((o.last != 0) != last) return FXPQ_ERR_INVALID_ARG;
        if (o.src0 < 0 || o.src0 >= net->n_slots || !slots[o.src0].defined) return FXPQ_ERR_INVALID_ARG;
        if (!last && (o.dst <= 0 || o.dst >= net->n_slots || slots[o.dst].defined)) return FXPQ_ERR_INVALID_ARG;
        const Slot& s0 = slots[o.src0];
        Slot out;
        switch (o.op) {
            case FXPQ_OP_CONV: {
                if (o.K < 1 || o.R < 1 || o.S < 1 || o.stride < 1 || o.pad < 0 || !o.d_w) return FXPQ_ERR_INVALID_ARG;
                out.H = (s0.H + 2 * o.pad - o.R) / o.stride + 1;
                out.W = (s0.W + 2 * o.pad - o.S) / o.stride + 1;
                out.Cp = o.K;
                out.fmt = o.fmt_y;
                if (last) break;
                if (!fxpq::fmt_ok(o.fmt_y) || (o.K % 8)) return FXPQ_ERR_INVALID_ARG;
                break;
            }
            case FXPQ_OP_MAXPOOL:
                if (o.R < 1 || o.stride < 1 || o.pad < 0 || o.pad >= o.R) return FXPQ_ERR_INVALID_ARG;
                out.H = (s0.H + 2 * o.pad - o.R) / o.stride + 1;
                out.W = (s0.W + 2 * o.pad - o.R) / o.stride + 1;
                out.Cp = s0.Cp;
                out.fmt = s0.fmt;
                break;
            case FXPQ_OP_ELTWISE: {
                if (o.src1 < 0 || o.src1 >= net->n_slots || !slots[o.src1].defined) return FXPQ_ERR_INVALID_ARG;
                const Slot& s1 = slots[o.src1];
                if (s1.H != s0.H || s1.W != s0.W || s1.Cp != s0.Cp) return FXPQ_ERR_INVALID_ARG;
                out = s0;
                out.fmt = o.fmt_y;
                break;
            }
            case FXPQ_OP_AVGPOOL:
                out.H = out.W = 1;
                out.Cp = s0.Cp;
                out.fmt = o.fmt_y;
                break;
            default:
                return FXPQ_ERR_INVALID_ARG;
        }
        if (out.H < 1 || out.W < 1) return FXPQ_ERR_INVALID_ARG;
        if (last) {
            if (o.op != FXPQ_OP_CONV) return FXPQ_ERR_INVALID_ARG;
            continue;
        }
        out.defined = true;
        slots[o.dst] = out;
    }
    total = 0;
    for (auto& s : slots) {
        if (!s.defined) continue;
        s.bytes = align256((size_t)batch * s.H * s.W * s.Cp * fxpq::planes_of(s.fmt) * sizeof(__half));
        s.offset = total;
        total += s.bytes;
    }
    return FXPQ_OK;
}

}  // namespace

extern "C" size_t fxpq_net_workspace(const fxpq_net* h_net, int32_t batch) {
    std::vector<Slot> slots;
    size_t total = 0;
    if (plan_net(h_net, batch, slots, total) != FXPQ_OK) return 0;
    return total + 256;
}

extern "C" fxpq_status fxpq_net_forward(const fxpq_net* h_net, const float* d_images_nchw, int32_t batch,
                                        int64_t* d_logits, int32_t* h_logits_scale, void* d_ws, size_t ws_bytes,
                                        void* stream) {
    std::vector<Slot> slots;
    size_t total = 0;
    fxpq_status st = plan_net(h_net, batch, slots, total);
    if (st != FXPQ_OK) return st;
    if (batch > 0 && (!d_images_nchw || !d_logits)) return FXPQ_ERR_INVALID_ARG;
    if (!d_ws || ws_bytes < total || !fxpq::aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    char* base = static_cast<char*>(d_ws);
    auto ptr = [&](int slot) { return static_cast<void*>(base + slots[slot].offset); };
    if (batch == 0) return FXPQ_OK;

    st = fxpq_quantize_images(d_images_nchw, batch, h_net->C, h_net->H, h_net->W, h_net->fmt_in, h_net->Cp_in, ptr(0),
                              stream);
    if (st != FXPQ_OK) return st;
    for (int i = 0; i < h_net->n_ops; ++i) {
        const fxpq_op_desc& o = h_net->ops[i];
        const Slot& s0 = slots[o.src0];
        const bool last = o.last != 0;
        switch (o.op) {
            case FXPQ_OP_CONV: {
                fxpq_conv_desc d;
                d.N = batch;
                d.H = s0.H;
                d.W = s0.W;
                d.C = s0.Cp;
                d.Cp = s0.Cp;
                d.K = o.K;
                d.R = o.R;
                d.S = o.S;
                d.stride = o.stride;
                d.pad = o.pad;
                d.relu = o.relu;
                d.out_mode = last ? FXPQ_OUT_ACC64 : FXPQ_OUT_CODES;
                d.fmt_x = s0.fmt;
                d.fmt_w = o.fmt_w;
                d.fmt_b = o.fmt_b;
                d.fmt_y = o.fmt_y;
                d.w_l1 = o.w_l1;
                int32_t scale = 0;
                st = fxpq_conv_fwd(&d, ptr(o.src0), o.d_w, o.d_bias, last ? (void*)d_logits : ptr(o.dst), &scale,
                                   nullptr, 0, stream);
                if (last && h_logits_scale) *h_logits_scale = scale;
                break;
            }
            case FXPQ_OP_MAXPOOL:
                st = fxpq_maxpool(ptr(o.src0), batch, s0.H, s0.W, s0.Cp, s0.fmt, o.R, o.stride, o.pad, ptr(o.dst),
                                  stream);
                break;
            case FXPQ_OP_ELTWISE:
                st = fxpq_eltwise(ptr(o.src0), s0.fmt, ptr(o.src1), slots[o.src1].fmt, (int64_t)batch * s0.H * s0.W,
                                  s0.Cp, o.relu, FXPQ_OUT_CODES, o.fmt_y, ptr(o.dst), nullptr, stream);
                break;
            case FXPQ_OP_AVGPOOL:
                st = fxpq_avgpool(ptr(o.src0), batch, s0.H, s0.W, s0.Cp, s0.fmt, o.recip_code, o.fmt_w, FXPQ_OUT_CODES,
                                  o.fmt_y, ptr(o.dst), nullptr, stream);
                break;
            default:
                st = FXPQ_ERR_INVALID_ARG;
        }
        if (st != FXPQ_OK) return st;
    }
    return FXPQ_OK;
}
