// fxpq_conv.cu -- C-Block on integer codes (Sec. IV-B): convolution / FC with exact integer
// accumulation and the fused epilogue (bias alignment, ReLU, FxP-QLayer shift-requantize).
//
// This translation unit holds the CUDA-core implicit-GEMM kernel (exact int32 / int64 MACs),
// used for every shape, and the host entry points.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include "fxpq_common.cuh"
#include "fxpq_conv.cuh"

namespace fxpq {
namespace {

__device__ __forceinline__ int load_code(const __half* __restrict__ t, long long row, int Cp, int planes, int c,
                                         long long plane_stride) {
    return code_get(t, row * Cp + c, planes, plane_stride);
}

constexpr int TM = 64, TN = 64, TK = 16, NT = 256;

template <typename ACC>
__global__ void __launch_bounds__(NT) conv_simt_kernel(ConvArgs a) {
    __shared__ int As[TK][TM + 1];
    __shared__ int Bs[TK][TN + 1];
    const int tid = threadIdx.x;
    const int tx = tid % 16, ty = tid / 16;
    const long long M = (long long)a.N * a.P * a.Q;
    const long long m0 = (long long)blockIdx.x * TM;
    const int n0 = blockIdx.y * TN;

    // per-thread loader coordinates: 4 (row, channel) entries of the A and B tiles
    long long pix_n[4];
    int pix_p[4], pix_q[4];
    bool pix_ok[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        int e = tid + NT * i;
        long long m = m0 + (e >> 4);
        pix_ok[i] = m < M;
        long long mm = pix_ok[i] ? m : 0;
        pix_n[i] = mm / ((long long)a.P * a.Q);
        int pq = (int)(mm - pix_n[i] * a.P * a.Q);
        pix_p[i] = pq / a.Q;
        pix_q[i] = pq - pix_p[i] * a.Q;
    }

    ACC acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0;

    for (int r = 0; r < a.R; ++r)
        for (int s = 0; s < a.S; ++s)
            for (int c0 = 0; c0 < a.Cp; c0 += TK) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    int e = tid + NT * i;
                    int cc = e & (TK - 1);
                    int row = e >> 4;
                    int c = c0 + cc;
                    int code = 0;
                    int h = pix_p[i] * a.stride + r - a.pad;
                    int w = pix_q[i] * a.stride + s - a.pad;
                    if (pix_ok[i] && c < a.Cp && h >= 0 && h < a.H && w >= 0 && w < a.W)
                        code = load_code(a.x, (pix_n[i] * a.H + h) * a.W + w, a.Cp, a.px, c, a.x_ps);
                    As[cc][row] = code;
                    int k = n0 + row;
                    int wc = 0;
                    if (k < a.K && c < a.Cp)
                        wc = load_code(a.w, ((long long)k * a.R + r) * a.S + s, a.Cp, a.pw, c, a.w_ps);
                    Bs[cc][row] = wc;
                }
                __syncthreads();
#pragma unroll
                for (int cc = 0; cc < TK; ++cc) {
                    int av[4], bv[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) av[i] = As[cc][ty * 4 + i];
#pragma unroll
                    for (int j = 0; j < 4; ++j) bv[j] = Bs[cc][tx * 4 + j];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int j = 0; j < 4; ++j) acc[i][j] += (ACC)av[i] * (ACC)bv[j];
                }
                __syncthreads();
            }

#pragma unroll
    for (int i = 0; i < 4; ++i) {
        long long m = m0 + ty * 4 + i;
        if (m >= M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            int k = n0 + tx * 4 + j;
            if (k < a.K) cblock_epilogue_store(a, m, k, (long long)acc[i][j]);
        }
    }
}

template <typename ACC>
__global__ void splitk_reduce_kernel(const ConvArgs a, const ACC* __restrict__ part, int ks) {
    const long long total = a.M * a.K;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        long long v = 0;
        for (int s = 0; s < ks; ++s) v += (long long)part[s * total + i];
        cblock_epilogue_store(a, i / a.K, (int)(i % a.K), v);
    }
}

}  // namespace

fxpq_status launch_splitk_reduce(const ConvArgs& a, const void* part, int ks, bool acc64, cudaStream_t st) {
    const long long total = a.M * a.K;
    long long blocks = (total + 255) / 256;
    if (blocks > 152LL * 8) blocks = 152LL * 8;
    if (blocks < 1) blocks = 1;
    if (acc64)
        splitk_reduce_kernel<long long><<<(unsigned)blocks, 256, 0, st>>>(a, static_cast<const long long*>(part), ks);
    else
        splitk_reduce_kernel<int><<<(unsigned)blocks, 256, 0, st>>>(a, static_cast<const int*>(part), ks);
    return after_launch("splitk_reduce");
}

// At most 16 shares of int64 sums, for layers whose M x K outputs are small enough for the split to pay
// (it is taken only when the tiles cannot occupy the SMs); capped at 64 MiB.
size_t conv_split_ws_bytes(long long M, int K) {
    const size_t one = (size_t)M * (size_t)K * sizeof(long long);
    const size_t cap = (size_t)64 << 20;
    if (M <= 0 || K <= 0 || 2 * one > cap) return 0;
    return 16 * one < cap ? 16 * one : cap;
}

// Host-side planning shared by conv and gemm: fills ConvArgs, checks the integer bounds.
fxpq_status plan_conv(const fxpq_conv_desc& d, const void* x, const void* w, const int32_t* bias, void* y,
                      ConvArgs& a, int32_t* out_scale, bool& need64) {
    if (d.N < 0 || d.H < 1 || d.W < 1 || d.C < 1 || d.Cp < d.C || (d.Cp % 8) || d.K < 1 || d.R < 1 || d.S < 1 ||
        d.stride < 1 || d.pad < 0)
        return FXPQ_ERR_INVALID_ARG;
    if (!fmt_ok(d.fmt_x) || !fmt_ok(d.fmt_w)) return FXPQ_ERR_INVALID_ARG;
    if (bias && !fmt_ok(d.fmt_b, 32)) return FXPQ_ERR_INVALID_ARG;
    if (d.out_mode < FXPQ_OUT_CODES || d.out_mode > FXPQ_OUT_F32) return FXPQ_ERR_INVALID_ARG;
    if (d.out_mode == FXPQ_OUT_CODES && (!fmt_ok(d.fmt_y) || (d.K % 8))) return FXPQ_ERR_INVALID_ARG;
    const int P = (d.H + 2 * d.pad - d.R) / d.stride + 1, Q = (d.W + 2 * d.pad - d.S) / d.stride + 1;
    if (P < 1 || Q < 1) return FXPQ_ERR_INVALID_ARG;
    if (d.N > 0 && (!x || !w || !y)) return FXPQ_ERR_INVALID_ARG;
    if (!aligned(x, 16) || !aligned(w, 16) || !aligned(y, 16)) return FXPQ_ERR_INVALID_ARG;
    // |acc| <= max|x code| * max|w code| * R*S*C
    const double ax = ldexp(1.0, d.fmt_x.bits - d.fmt_x.is_signed), aw = ldexp(1.0, d.fmt_w.bits - d.fmt_w.is_signed);
    double bound = ax * aw * (double)d.R * d.S * d.C;
    // with a weight-code L1 bound: |acc| <= max|x code| * max_o sum |w code|
    if (d.w_l1 > 0 && d.fmt_w.bits <= 8 && ax * (double)d.w_l1 < bound) bound = ax * (double)d.w_l1;
    if (d.w_l1 < 0) return FXPQ_ERR_INVALID_ARG;
    if (bound >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
    need64 = bound >= ldexp(1.0, 31) - 1.0;
    a.x = static_cast<const __half*>(x);
    a.w = static_cast<const __half*>(w);
    a.bias = bias;
    a.y = y;
    a.N = d.N, a.H = d.H, a.W = d.W, a.Cp = d.Cp, a.K = d.K, a.R = d.R, a.S = d.S;
    a.stride = d.stride, a.pad = d.pad, a.P = P, a.Q = Q;
    a.M = (long long)d.N * P * Q;
    a.x_ps = (long long)d.N * d.H * d.W * d.Cp;
    a.w_ps = (long long)d.K * d.R * d.S * d.Cp;
    a.px = planes_of(d.fmt_x);
    a.pw = planes_of(d.fmt_w);
    a.relu = d.relu;
    a.out_mode = d.out_mode;
    int s = d.fmt_x.fl + d.fmt_w.fl;
    a.delta = 0;
    double vbound = bound;
    if (bias) {
        a.delta = s - d.fmt_b.fl;
        const double bb = ldexp(1.0, d.fmt_b.bits - d.fmt_b.is_signed);
        if (a.delta >= 0) {
            if (a.delta > 40 || bb * ldexp(1.0, a.delta) + bound >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
            vbound = bound + bb * ldexp(1.0, a.delta);
        } else {
            if (-a.delta > 40 || bound * ldexp(1.0, -a.delta) + bb >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
            vbound = bound * ldexp(1.0, -a.delta) + bb;
            s = d.fmt_b.fl;
        }
    }
    a.has_scale = d.d_scale != nullptr;
    a.scale = d.d_scale;
    a.shift = d.d_shift;
    a.delta2 = 0;
    if (a.has_scale) {
        // v * aleph1 at scale s + fl_aleph1, then aleph2 aligned like the bias
        if (!d.d_shift || !fmt_ok(d.fmt_scale, 32) || !fmt_ok(d.fmt_shift, 32)) return FXPQ_ERR_INVALID_ARG;
        const double mb = ldexp(1.0, d.fmt_scale.bits - d.fmt_scale.is_signed);
        const double hb = ldexp(1.0, d.fmt_shift.bits - d.fmt_shift.is_signed);
        const double pbound = vbound * mb;
        if (pbound >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
        s += d.fmt_scale.fl;
        a.delta2 = s - d.fmt_shift.fl;
        if (a.delta2 >= 0) {
            if (a.delta2 > 40 || hb * ldexp(1.0, a.delta2) + pbound >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
            vbound = pbound + hb * ldexp(1.0, a.delta2);
        } else {
            if (-a.delta2 > 40 || pbound * ldexp(1.0, -a.delta2) + hb >= ldexp(1.0, 62)) return FXPQ_ERR_RANGE;
            vbound = pbound * ldexp(1.0, -a.delta2) + hb;
            s = d.fmt_shift.fl;
        }
    } else if (d.d_shift) {
        return FXPQ_ERR_INVALID_ARG;
    }
    (void)vbound;
    a.s_out = s;
    a.has_bias = bias != nullptr;
    a.v32 = 0;
    if (d.out_mode == FXPQ_OUT_CODES) {
        a.sh = s - d.fmt_y.fl;
        if (a.sh > 62) return FXPQ_ERR_RANGE;
        a.lo = qmin_of(d.fmt_y);
        a.hi = qmax_of(d.fmt_y);
        a.py = planes_of(d.fmt_y);
        // 32-bit path: N = acc + aligned integer part of the bias, plus the rounding increment
        // 2^(sh32 - 1), stays below 2^31 in magnitude and the FxP-QLayer is a right shift by 1..30 bits
        // of N (see qlayer_code32)
        const double two31 = ldexp(1.0, 31) - 1.0;
        const double bb = bias ? ldexp(1.0, d.fmt_b.bits - d.fmt_b.is_signed) : 0.0;
        const int s_acc = d.fmt_x.fl + d.fmt_w.fl;
        a.bsh = a.delta;
        a.sh32 = s_acc - d.fmt_y.fl;
        const double nbound = bound + (a.delta >= 0 ? bb * ldexp(1.0, a.delta) : bb * ldexp(1.0, a.delta) + 1.0);
        a.v32 = (!a.has_scale && a.sh32 >= 1 && a.sh32 <= 30 && nbound + ldexp(1.0, a.sh32 - 1) < two31 && a.delta >= -30 &&
                 a.delta <= 30)
                    ? 1
                    : 0;
    } else {
        a.sh = 0;
        a.lo = a.hi = 0;
        a.py = 1;
    }
    a.f32_scale = ldexpf(1.0f, -s);
    if (out_scale) *out_scale = s;
    return FXPQ_OK;
}

// FXPQ_CONV_PATH=simt selects the CUDA-core kernel for every shape (tests use it to cover both).
static bool tc_path_enabled() {
    const char* e = getenv("FXPQ_CONV_PATH");
    return !(e && strcmp(e, "simt") == 0);
}

fxpq_status launch_conv(const ConvArgs& a, const fxpq_conv_desc& d, bool need64, cudaStream_t st, void* ws,
                        size_t ws_bytes) {
    const long long M = (long long)a.N * a.P * a.Q;
    if (M == 0) return FXPQ_OK;
    if (tc_path_enabled()) {
        bool launched = false;
        fxpq_status s = launch_conv_tc(a, d, st, launched, ws, ws_bytes);
        if (s != FXPQ_OK || launched) return s;
    }
    dim3 grid((unsigned)((M + TM - 1) / TM), (unsigned)((a.K + TN - 1) / TN));
    if (need64)
        conv_simt_kernel<long long><<<grid, NT, 0, st>>>(a);
    else
        conv_simt_kernel<int><<<grid, NT, 0, st>>>(a);
    return after_launch("conv_simt");
}

}  // namespace fxpq

using namespace fxpq;

extern "C" size_t fxpq_conv_workspace(const fxpq_conv_desc* h_desc) {
    if (!h_desc || h_desc->N < 1 || h_desc->stride < 1 || h_desc->R < 1 || h_desc->S < 1) return 0;
    const int P = (h_desc->H + 2 * h_desc->pad - h_desc->R) / h_desc->stride + 1;
    const int Q = (h_desc->W + 2 * h_desc->pad - h_desc->S) / h_desc->stride + 1;
    if (P < 1 || Q < 1) return 0;
    return conv_split_ws_bytes((long long)h_desc->N * P * Q, h_desc->K);
}

extern "C" fxpq_status fxpq_conv_fwd(const fxpq_conv_desc* h_desc, const void* d_x, const void* d_w,
                                     const int32_t* d_bias, void* d_y, int32_t* h_out_scale, void* d_ws,
                                     size_t ws_bytes, void* stream) {
    if (!h_desc) return FXPQ_ERR_INVALID_ARG;
    if (d_ws && !aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    ConvArgs a;
    bool need64 = false;
    fxpq_status st = plan_conv(*h_desc, d_x, d_w, d_bias, d_y, a, h_out_scale, need64);
    if (st != FXPQ_OK) return st;
    return launch_conv(a, *h_desc, need64, as_stream(stream), d_ws, d_ws ? ws_bytes : 0);
}

extern "C" fxpq_status fxpq_gemm(const void* d_x, fxpq_fmt fmt_x, const void* d_w, fxpq_fmt fmt_w,
                                 const int32_t* d_bias, fxpq_fmt fmt_b, int32_t M, int32_t N, int32_t Kdim,
                                 int32_t relu, int32_t out_mode, fxpq_fmt fmt_y, void* d_y, int32_t* h_out_scale,
                                 void* d_ws, size_t ws_bytes, void* stream) {
    fxpq_conv_desc d = {};
    d.N = M;
    d.H = d.W = 1;
    d.C = Kdim;
    d.Cp = Kdim;
    d.K = N;
    d.R = d.S = 1;
    d.stride = 1;
    d.pad = 0;
    d.relu = relu;
    d.out_mode = out_mode;
    d.fmt_x = fmt_x;
    d.fmt_w = fmt_w;
    d.fmt_b = fmt_b;
    d.fmt_y = fmt_y;
    d.w_l1 = 0;
    return fxpq_conv_fwd(&d, d_x, d_w, d_bias, d_y, h_out_scale, d_ws, ws_bytes, stream);
}
