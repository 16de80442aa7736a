// fxpq_net.cu -- integer-only network forward (Sec. IV-A.2: FxP-QLayers as vertices, C-Blocks as
// edges).  Host-side driver: derives every slot's shape, carves the slots out of the caller's
// workspace, and launches the C-Block kernels in order on the caller's stream.
#include <algorithm>
#include <cstring>
#include <mutex>
#include <vector>

#include "fxpq_common.cuh"
#include "fxpq_conv.cuh"

namespace {

struct Slot {
    int H = 0, W = 0, Cp = 0;
    int C = 0;  // true channel count (Cp without the padding)
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
    slots[0].C = net->C;
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
                out.C = o.K;
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
                out.C = s0.C;
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
                out.C = s0.C;
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

// Largest split-reduction scratch any conv op of the list may use at this batch.
size_t net_conv_ws(const fxpq_net* net, const std::vector<Slot>& slots, int32_t batch) {
    size_t m = 0;
    for (int i = 0; i < net->n_ops; ++i) {
        const fxpq_op_desc& o = net->ops[i];
        if (o.op != FXPQ_OP_CONV) continue;
        const Slot& s0 = slots[o.src0];
        const int P = (s0.H + 2 * o.pad - o.R) / o.stride + 1, Q = (s0.W + 2 * o.pad - o.S) / o.stride + 1;
        const size_t b = fxpq::conv_split_ws_bytes((long long)batch * P * Q, o.K);
        if (b > m) m = b;
    }
    return align256(m);
}

}  // namespace

extern "C" fxpq_status fxpq_net_memory(const fxpq_net* h_net, int32_t fp32, double* h_rw_mb, double* h_ro_mb) {
    std::vector<Slot> slots;
    size_t total = 0;
    fxpq_status st = plan_net(h_net, 0, slots, total);
    if (st != FXPQ_OK) return st;
    if (!h_rw_mb || !h_ro_mb) return FXPQ_ERR_INVALID_ARG;
    // MFP(d) = nu * k / 2^23 MB, k = 32 for FP32
    auto mfp = [fp32](double nu, int bits) { return nu * (fp32 ? 32 : bits) / 8388608.0; };
    auto act = [&](const Slot& s) { return mfp((double)s.H * s.W * s.C, s.fmt.bits); };
    double rw = 0.0, ro = 0.0;
    for (int i = 0; i < h_net->n_ops; ++i) {
        const fxpq_op_desc& o = h_net->ops[i];
        const Slot& s0 = slots[o.src0];
        double in = act(s0);
        if (o.op == FXPQ_OP_ELTWISE) in += act(slots[o.src1]);
        double out;
        if (o.last) {
            const int P = (s0.H + 2 * o.pad - o.R) / o.stride + 1, Q = (s0.W + 2 * o.pad - o.S) / o.stride + 1;
            out = (double)P * Q * o.K * 32 / 8388608.0;  // the last layer has no FxP-QLayer
        } else {
            out = act(slots[o.dst]);
        }
        if (in + out > rw) rw = in + out;
        if (o.op == FXPQ_OP_CONV) {
            ro += mfp((double)o.K * o.R * o.S * s0.C, o.fmt_w.bits);
            if (o.d_bias) ro += mfp(o.K, o.fmt_b.bits);
            if (o.d_scale) ro += mfp(o.K, o.fmt_scale.bits) + mfp(o.K, o.fmt_shift.bits);
        }
    }
    *h_rw_mb = rw;
    *h_ro_mb = ro;
    return FXPQ_OK;
}

extern "C" size_t fxpq_net_workspace(const fxpq_net* h_net, int32_t batch) {
    std::vector<Slot> slots;
    size_t total = 0;
    if (plan_net(h_net, batch, slots, total) != FXPQ_OK) return 0;
    return total + net_conv_ws(h_net, slots, batch) + 256;
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
    // the convs' split-reduction scratch follows the slots when the caller provided it
    const size_t cws = net_conv_ws(h_net, slots, batch);
    void* conv_ws = (cws && ws_bytes >= total + cws) ? static_cast<void*>(base + total) : nullptr;

    st = fxpq_quantize_images(d_images_nchw, batch, h_net->C, h_net->H, h_net->W, h_net->fmt_in, h_net->Cp_in, ptr(0),
                              stream);
    if (st != FXPQ_OK) return st;
    for (int i = 0; i < h_net->n_ops; ++i) {
        const fxpq_op_desc& o = h_net->ops[i];
        const Slot& s0 = slots[o.src0];
        const bool last = o.last != 0;
        switch (o.op) {
            case FXPQ_OP_CONV: {
                fxpq_conv_desc d = {};
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
                d.fmt_scale = o.fmt_scale;
                d.fmt_shift = o.fmt_shift;
                d.d_scale = o.d_scale;
                d.d_shift = o.d_shift;
                d.d_wpacked = o.d_wpacked;
                int32_t scale = 0;
                st = fxpq_conv_fwd(&d, ptr(o.src0), o.d_w, o.d_bias, last ? (void*)d_logits : ptr(o.dst), &scale,
                                   conv_ws, conv_ws ? cws : 0, stream);
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

// ------------------------------------------------------------------------------------------
// Calibration of the activation formats (Sec. IV-C: the forward optimizer visits the layers in
// order; every earlier layer is already quantized when a layer's output FL is searched).
// ------------------------------------------------------------------------------------------
namespace {

struct CalibLayout {
    std::vector<Slot> slots;
    size_t slots_bytes = 0, acc_off = 0, f32_off = 0, fls_off = 0, err_off = 0, cws_off = 0, cws = 0, total = 0;
};

// The calibration of a contraction's output format needs its exact values twice: as the fp32 image
// for the FL search and as codes once the format is known.  Either the contraction runs once to int64
// values and the FxP-QLayer twice from them, or the contraction runs twice (to the fp32 image, then to
// codes).  The first costs about 30 bytes of traffic per output value and two small launches, the
// second one more pass over the input codes and weights and the contraction's work: a rough time
// model (5 TB/s, 1 PFLOP/s, 10 / 8 us of fixed cost) picks the cheaper, so FC layers and the late
// 3x3 layers at calibration batch sizes take int64 values, and the large early layers the second pass.
bool calib_acc64(const fxpq_op_desc& o, const Slot& s0, const Slot& d, int32_t n) {
    if (o.op != FXPQ_OP_CONV) return false;
    const double n_out = (double)n * d.H * d.W * d.Cp;
    const double n_in = (double)n * s0.H * s0.W * s0.Cp;
    const double w_bytes = (double)o.K * o.R * o.S * s0.Cp * 2.0 * (o.fmt_w.bits > 8 ? 2.0 : 1.0);
    const double flops = 2.0 * (double)n * d.H * d.W * o.K * o.R * o.S * s0.Cp;
    const double t_pass = std::max(flops / 1e15, (2.0 * n_in + w_bytes + 2.0 * n_out) / 5e12) + 10e-6;
    const double t_acc = 30.0 * n_out / 5e12 + 8e-6;
    return t_acc < t_pass;
}

fxpq_status plan_calib(const fxpq_net* net, int32_t n, CalibLayout& L) {
    fxpq_status st = plan_net(net, n, L.slots, L.slots_bytes);
    if (st != FXPQ_OK) return st;
    // largest per-op output (elements): the fp32 image of a C-Block output searched by the calibration,
    // and of the contractions that go through int64 values
    size_t max_out = 1, max_acc = 0;
    for (int i = 0; i < net->n_ops - 1; ++i) {
        const fxpq_op_desc& o = net->ops[i];
        const Slot& d = L.slots[o.dst];
        const size_t e = (size_t)n * d.H * d.W * d.Cp;
        if (e > max_out) max_out = e;
        if (calib_acc64(o, L.slots[o.src0], d, n) && e > max_acc) max_acc = e;
    }
    const size_t img = (size_t)n * net->C * net->H * net->W;
    L.acc_off = L.slots_bytes;
    L.f32_off = L.acc_off + align256(max_acc * sizeof(int64_t));
    L.fls_off = L.f32_off + align256((max_out > img ? max_out : img) * sizeof(float));
    L.err_off = L.fls_off + align256(fxpq_fl_search_workspace(0));
    L.cws_off = L.err_off + align256(32 * sizeof(double));
    L.cws = net_conv_ws(net, L.slots, n);
    L.total = L.cws_off + L.cws;
    return FXPQ_OK;
}

// Mapped pinned host records: the FL search's final kernel writes the chosen FL and the stats
// straight into host memory, so that the calibration reads them after a stream synchronisation
// with no copy in between.  A small pool, one record per running calibration, kept for the
// process's lifetime.
struct HostRec {
    unsigned char* h = nullptr;  // host address
    unsigned char* d = nullptr;  // its device address
};
constexpr size_t kHostRecBytes = 256;
static_assert(64 + sizeof(fxpq_stats) <= kHostRecBytes, "the record holds the FL and the stats");
std::mutex g_rec_mu;
std::vector<HostRec> g_rec_free;

struct HostRecLease {
    HostRec r;
    bool ok = false;
    HostRecLease() {
        {
            std::lock_guard<std::mutex> lk(g_rec_mu);
            if (!g_rec_free.empty()) {
                r = g_rec_free.back();
                g_rec_free.pop_back();
                ok = true;
                return;
            }
        }
        void* h = nullptr;
        void* d = nullptr;
        if (cudaHostAlloc(&h, kHostRecBytes, cudaHostAllocMapped | cudaHostAllocPortable) != cudaSuccess) return;
        if (cudaHostGetDevicePointer(&d, h, 0) != cudaSuccess) {
            cudaFreeHost(h);
            return;
        }
        r.h = static_cast<unsigned char*>(h);
        r.d = static_cast<unsigned char*>(d);
        ok = true;
    }
    ~HostRecLease() {
        if (!ok) return;
        std::lock_guard<std::mutex> lk(g_rec_mu);
        g_rec_free.push_back(r);
    }
    HostRecLease(const HostRecLease&) = delete;
    HostRecLease& operator=(const HostRecLease&) = delete;
};

// FL search of one fp32 tensor at wordlength k, S picked from the data; waits for the result.
fxpq_status calib_search(const float* d_x, int64_t n, int k, int fl_lo, int fl_hi, char* base, const CalibLayout& L,
                         const HostRec& rec, cudaStream_t s, fxpq_fmt& out) {
    int32_t* d_best = reinterpret_cast<int32_t*>(rec.d);
    fxpq_stats* d_stats = reinterpret_cast<fxpq_stats*>(rec.d + 64);
    fxpq_status st = fxpq_fl_search(d_x, n, -1, k, k, fl_lo, fl_hi, reinterpret_cast<double*>(base + L.err_off),
                                    d_best, d_stats, base + L.fls_off, fxpq_fl_search_workspace(n), s);
    if (st != FXPQ_OK) return st;
    if (cudaStreamSynchronize(s) != cudaSuccess) return FXPQ_ERR_CUDA;
    int32_t best;
    fxpq_stats stats;
    memcpy(&best, rec.h, sizeof(best));
    memcpy(&stats, rec.h + 64, sizeof(stats));
    out.bits = k;
    out.is_signed = stats.is_signed;
    out.fl = best;
    return FXPQ_OK;
}

}  // namespace

extern "C" size_t fxpq_net_calibrate_workspace(const fxpq_net* h_net, int32_t n_calib) {
    CalibLayout L;
    if (plan_calib(h_net, n_calib, L) != FXPQ_OK) return 0;
    return L.total + 256;
}

extern "C" fxpq_status fxpq_net_calibrate(const fxpq_net* h_net, const float* d_calib_nchw, int32_t n_calib,
                                          int32_t fl_lo, int32_t fl_hi, fxpq_fmt* h_fmt_in, fxpq_fmt* h_fmt_y,
                                          void* d_ws, size_t ws_bytes, void* stream) {
    CalibLayout L;
    fxpq_status st = plan_calib(h_net, n_calib, L);
    if (st != FXPQ_OK) return st;
    if (n_calib < 1 || !d_calib_nchw || !h_fmt_in || !h_fmt_y) return FXPQ_ERR_INVALID_ARG;
    if (fl_lo < -32 || fl_hi > 40 || fl_lo > fl_hi || fl_hi - fl_lo > 31) return FXPQ_ERR_INVALID_ARG;
    if (!d_ws || ws_bytes < L.total || !fxpq::aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    cudaStream_t s = fxpq::as_stream(stream);
    char* base = static_cast<char*>(d_ws);
    auto ptr = [&](int slot) { return static_cast<void*>(base + L.slots[slot].offset); };
    float* f32 = reinterpret_cast<float*>(base + L.f32_off);
    HostRecLease lease;
    if (!lease.ok) return FXPQ_ERR_CUDA;
    std::vector<fxpq_fmt> fmt(h_net->n_slots, fxpq_fmt{0, 0, 0});

    // input FxP-QLayer: FL search on the fp32 images, then the codes
    const int64_t n_img = (int64_t)n_calib * h_net->C * h_net->H * h_net->W;
    st = calib_search(d_calib_nchw, n_img, h_net->fmt_in.bits, fl_lo, fl_hi, base, L, lease.r, s, fmt[0]);
    if (st != FXPQ_OK) return st;
    *h_fmt_in = fmt[0];
    st = fxpq_quantize_images(d_calib_nchw, n_calib, h_net->C, h_net->H, h_net->W, fmt[0], h_net->Cp_in, ptr(0), s);
    if (st != FXPQ_OK) return st;

    for (int i = 0; i < h_net->n_ops; ++i) {
        const fxpq_op_desc& o = h_net->ops[i];
        h_fmt_y[i] = o.fmt_y;
        if (o.last) break;  // the logits layer has no QLayer to calibrate
        const Slot& s0 = L.slots[o.src0];
        const Slot& d = L.slots[o.dst];
        const int64_t n_out = (int64_t)n_calib * d.H * d.W * d.Cp;
        fxpq_fmt fy{o.fmt_y.bits, 0, 0};
        switch (o.op) {
            case FXPQ_OP_MAXPOOL:
                fy = fmt[o.src0];  // no QLayer follows a max-pool
                st = fxpq_maxpool(ptr(o.src0), n_calib, s0.H, s0.W, s0.Cp, fmt[o.src0], o.R, o.stride, o.pad,
                                  ptr(o.dst), s);
                break;
            case FXPQ_OP_CONV: {
                // either the contraction writes the fp32 nearest-even image of its exact C-Block output
                // for the search, then runs again with the searched format to codes (the same exact
                // values both times), or it writes the int64 values once and the FxP-QLayer makes the
                // image and then the codes from them (calib_acc64 picks)
                const bool acc64 = calib_acc64(o, s0, d, n_calib);
                fxpq_conv_desc cd = {};
                cd.N = n_calib;
                cd.H = s0.H;
                cd.W = s0.W;
                cd.C = s0.Cp;
                cd.Cp = s0.Cp;
                cd.K = o.K;
                cd.R = o.R;
                cd.S = o.S;
                cd.stride = o.stride;
                cd.pad = o.pad;
                cd.relu = o.relu;
                cd.out_mode = FXPQ_OUT_F32;
                cd.fmt_x = fmt[o.src0];
                cd.fmt_w = o.fmt_w;
                cd.fmt_b = o.fmt_b;
                cd.fmt_y = fy;
                cd.w_l1 = o.w_l1;
                cd.fmt_scale = o.fmt_scale;
                cd.fmt_shift = o.fmt_shift;
                cd.d_scale = o.d_scale;
                cd.d_shift = o.d_shift;
                cd.d_wpacked = o.d_wpacked;
                int32_t sc = 0;
                void* cws = L.cws ? base + L.cws_off : nullptr;
                if (acc64) {
                    int64_t* acc = reinterpret_cast<int64_t*>(base + L.acc_off);
                    cd.out_mode = FXPQ_OUT_ACC64;
                    st = fxpq_conv_fwd(&cd, ptr(o.src0), o.d_w, o.d_bias, acc, &sc, cws, L.cws, s);
                    if (st == FXPQ_OK) st = fxpq_qlayer(acc, n_out, sc, FXPQ_OUT_F32, fy, f32, s);
                    if (st == FXPQ_OK)
                        st = calib_search(f32, n_out, o.fmt_y.bits, fl_lo, fl_hi, base, L, lease.r, s, fy);
                    if (st == FXPQ_OK) st = fxpq_qlayer(acc, n_out, sc, FXPQ_OUT_CODES, fy, ptr(o.dst), s);
                    break;
                }
                st = fxpq_conv_fwd(&cd, ptr(o.src0), o.d_w, o.d_bias, f32, &sc, cws, L.cws, s);
                if (st == FXPQ_OK) st = calib_search(f32, n_out, o.fmt_y.bits, fl_lo, fl_hi, base, L, lease.r, s, fy);
                if (st == FXPQ_OK) {
                    cd.out_mode = FXPQ_OUT_CODES;
                    cd.fmt_y = fy;
                    st = fxpq_conv_fwd(&cd, ptr(o.src0), o.d_w, o.d_bias, ptr(o.dst), &sc, cws, L.cws, s);
                }
                break;
            }
            case FXPQ_OP_ELTWISE: {
                const int64_t npix = (int64_t)n_calib * s0.H * s0.W;
                st = fxpq_eltwise(ptr(o.src0), fmt[o.src0], ptr(o.src1), fmt[o.src1], npix, s0.Cp, o.relu, FXPQ_OUT_F32,
                                  fy, f32, nullptr, s);
                if (st == FXPQ_OK) st = calib_search(f32, n_out, o.fmt_y.bits, fl_lo, fl_hi, base, L, lease.r, s, fy);
                if (st == FXPQ_OK)
                    st = fxpq_eltwise(ptr(o.src0), fmt[o.src0], ptr(o.src1), fmt[o.src1], npix, s0.Cp, o.relu,
                                      FXPQ_OUT_CODES, fy, ptr(o.dst), nullptr, s);
                break;
            }
            case FXPQ_OP_AVGPOOL:
                st = fxpq_avgpool(ptr(o.src0), n_calib, s0.H, s0.W, s0.Cp, fmt[o.src0], o.recip_code, o.fmt_w,
                                  FXPQ_OUT_F32, fy, f32, nullptr, s);
                if (st == FXPQ_OK) st = calib_search(f32, n_out, o.fmt_y.bits, fl_lo, fl_hi, base, L, lease.r, s, fy);
                if (st == FXPQ_OK)
                    st = fxpq_avgpool(ptr(o.src0), n_calib, s0.H, s0.W, s0.Cp, fmt[o.src0], o.recip_code, o.fmt_w,
                                      FXPQ_OUT_CODES, fy, ptr(o.dst), nullptr, s);
                break;
            default:
                st = FXPQ_ERR_INVALID_ARG;
        }
        if (st != FXPQ_OK) return st;
        fmt[o.dst] = fy;
        h_fmt_y[i] = fy;
    }
    return FXPQ_OK;
}
