// fxpq_ops.cu -- the non-contraction C-Blocks of the integer-only graph (Sec. IV-A.2):
// MAX-POOL (no FxP-QLayer), Eltwise residual add with FL alignment, global AVG-POOL with the
// reciprocal of the patch size quantized like a parameter.  All HBM-bound, one thread per output.
#include "fxpq_common.cuh"

namespace fxpq {
namespace {

struct OutArgs {
    int mode;         // FXPQ_OUT_*
    int sh;           // requant shift (CODES)
    long long lo, hi;
    int py;
    float f32_scale;  // 2^-s
};

// y plane stride for CODES output: y_ps elements
__device__ __forceinline__ void store_out(const OutArgs& o, void* y, long long pix, int Cp, int c, long long v,
                                          long long y_ps) {
    if (o.mode == FXPQ_OUT_CODES) {
        long long q;
        if (o.sh > 0) {
            q = rne_shift(v, o.sh);
        } else {
            const int l = -o.sh;
            const long long lim = 1LL << 20;
            if (l >= 32 || v > lim || v < -lim)
                q = v > 0 ? o.hi : (v < 0 ? o.lo : 0);
            else
                q = v << l;
        }
        q = q < o.lo ? o.lo : (q > o.hi ? o.hi : q);
        code_put(static_cast<__half*>(y), pix * Cp + c, o.py, y_ps, (int)q);
    } else if (o.mode == FXPQ_OUT_ACC64) {
        static_cast<long long*>(y)[pix * Cp + c] = v;
    } else {
        static_cast<float*>(y)[pix * Cp + c] = __ll2float_rn(v) * o.f32_scale;
    }
}

__global__ void maxpool_kernel(const __half* __restrict__ x, int N, int H, int W, int Cp, int planes, int k,
                               int stride, int pad, int P, int Q, __half* __restrict__ y) {
    const long long total = (long long)N * P * Q * Cp;
    const long long step = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += step) {
        const int c = (int)(i % Cp);
        const long long pix = i / Cp;
        const int q = (int)(pix % Q);
        const int p = (int)((pix / Q) % P);
        const long long n = pix / ((long long)P * Q);
        int best = INT_MIN;
        for (int r = 0; r < k; ++r) {
            const int h = p * stride + r - pad;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < k; ++s) {
                const int w = q * stride + s - pad;
                if (w < 0 || w >= W) continue;
                best = max(best, code_get(x, ((n * H + h) * W + w) * Cp + c, planes, (long long)N * H * W * Cp));
            }
        }
        code_put(y, pix * Cp + c, planes, total, best);
    }
}

// One-plane codes: 8 channels per thread with 16-byte loads and stores.  The codes are exact
// integers in fp16, so the half-precision max is exact.
__global__ void maxpool_vec8_kernel(const uint4* __restrict__ x, int N, int H, int W, int C8, int k, int stride,
                                    int pad, int P, int Q, uint4* __restrict__ y) {
    const long long total = (long long)N * P * Q * C8;
    const long long step = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += step) {
        const int c8 = (int)(i % C8);
        const long long pix = i / C8;
        const int q = (int)(pix % Q);
        const int p = (int)((pix / Q) % P);
        const long long n = pix / ((long long)P * Q);
        const __half2 ninf = __halves2half2(__ushort_as_half(0xFC00u), __ushort_as_half(0xFC00u));
        __half2 m0 = ninf, m1 = ninf, m2 = ninf, m3 = ninf;
        for (int r = 0; r < k; ++r) {
            const int h = p * stride + r - pad;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < k; ++s) {
                const int w = q * stride + s - pad;
                if (w < 0 || w >= W) continue;
                const uint4 v = __ldg(x + ((n * H + h) * W + w) * C8 + c8);
                m0 = __hmax2(m0, *reinterpret_cast<const __half2*>(&v.x));
                m1 = __hmax2(m1, *reinterpret_cast<const __half2*>(&v.y));
                m2 = __hmax2(m2, *reinterpret_cast<const __half2*>(&v.z));
                m3 = __hmax2(m3, *reinterpret_cast<const __half2*>(&v.w));
            }
        }
        uint4 o;
        o.x = *reinterpret_cast<uint32_t*>(&m0);
        o.y = *reinterpret_cast<uint32_t*>(&m1);
        o.z = *reinterpret_cast<uint32_t*>(&m2);
        o.w = *reinterpret_cast<uint32_t*>(&m3);
        y[i] = o;
    }
}

__global__ void eltwise_kernel(const __half* __restrict__ a, int pa, int sa, const __half* __restrict__ b, int pb,
                               int sb, long long npix, int Cp, int relu, OutArgs o, void* y) {
    const long long total = npix * Cp;
    const long long step = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += step) {
        const int c = (int)(i % Cp);
        const long long pix = i / Cp;
        long long v = ((long long)code_get(a, i, pa, total) << sa) + ((long long)code_get(b, i, pb, total) << sb);
        if (relu && v < 0) v = 0;
        store_out(o, y, pix, Cp, c, v, total);
    }
}

// FxP-QLayer on int64 C-Block values (scale 2^-s): codes (fp16 code tensor), int64 copy, or fp32 image.
__global__ void qlayer_kernel(const long long* __restrict__ v, long long n, OutArgs o, void* y) {
    const long long step = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += step)
        store_out(o, y, i, 1, 0, v[i], n);
}

__global__ void avgpool_kernel(const __half* __restrict__ x, int N, int HW, int Cp, int planes, long long recip,
                               OutArgs o, void* y) {
    const long long total = (long long)N * Cp;
    const long long step = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += step) {
        const int c = (int)(i % Cp);
        const long long n = i / Cp;
        long long s = 0;
        for (int t = 0; t < HW; ++t) s += code_get(x, (n * HW + t) * Cp + c, planes, (long long)N * HW * Cp);
        store_out(o, y, n, Cp, c, s * recip, total);
    }
}

int grid_for(long long work) {
    long long b = (work + 255) / 256;
    if (b < 1) b = 1;
    if (b > 152LL * 32) b = 152LL * 32;
    return (int)b;
}

fxpq_status make_out(int mode, const fxpq_fmt& fy, int s, OutArgs& o, int32_t* h_out_scale) {
    if (mode < FXPQ_OUT_CODES || mode > FXPQ_OUT_F32) return FXPQ_ERR_INVALID_ARG;
    o.mode = mode;
    if (mode == FXPQ_OUT_CODES) {
        if (!fmt_ok(fy)) return FXPQ_ERR_INVALID_ARG;
        o.sh = s - fy.fl;
        if (o.sh > 62) return FXPQ_ERR_RANGE;
        o.lo = qmin_of(fy);
        o.hi = qmax_of(fy);
        o.py = planes_of(fy);
    } else {
        o.sh = 0;
        o.lo = o.hi = 0;
        o.py = 1;
    }
    o.f32_scale = ldexpf(1.0f, -s);
    if (h_out_scale) *h_out_scale = s;
    return FXPQ_OK;
}

}  // namespace
}  // namespace fxpq

using namespace fxpq;

extern "C" fxpq_status fxpq_maxpool(const void* d_x, int32_t N, int32_t H, int32_t W, int32_t Cp, fxpq_fmt fmt,
                                    int32_t k, int32_t stride, int32_t pad, void* d_y, void* stream) {
    if (N < 0 || H < 1 || W < 1 || Cp < 1 || (Cp % 8) || k < 1 || stride < 1 || pad < 0 || pad >= k || !fmt_ok(fmt))
        return FXPQ_ERR_INVALID_ARG;
    const int P = (H + 2 * pad - k) / stride + 1, Q = (W + 2 * pad - k) / stride + 1;
    if (P < 1 || Q < 1) return FXPQ_ERR_INVALID_ARG;
    if (N == 0) return FXPQ_OK;
    if (!d_x || !d_y) return FXPQ_ERR_INVALID_ARG;
    const long long total = (long long)N * P * Q * Cp;
    if (planes_of(fmt) == 1 && aligned(d_x, 16) && aligned(d_y, 16)) {
        maxpool_vec8_kernel<<<grid_for(total / 8), 256, 0, as_stream(stream)>>>(
            static_cast<const uint4*>(d_x), N, H, W, Cp / 8, k, stride, pad, P, Q, static_cast<uint4*>(d_y));
        return after_launch("maxpool_vec8");
    }
    maxpool_kernel<<<grid_for(total), 256, 0, as_stream(stream)>>>(static_cast<const __half*>(d_x), N, H, W, Cp,
                                                                   planes_of(fmt), k, stride, pad, P, Q,
                                                                   static_cast<__half*>(d_y));
    return after_launch("maxpool");
}

extern "C" fxpq_status fxpq_eltwise(const void* d_a, fxpq_fmt fmt_a, const void* d_b, fxpq_fmt fmt_b, int64_t n_pix,
                                    int32_t Cp, int32_t relu, int32_t out_mode, fxpq_fmt fmt_y, void* d_y,
                                    int32_t* h_out_scale, void* stream) {
    if (n_pix < 0 || Cp < 1 || (Cp % 8) || !fmt_ok(fmt_a) || !fmt_ok(fmt_b)) return FXPQ_ERR_INVALID_ARG;
    const int fl = fmt_a.fl > fmt_b.fl ? fmt_a.fl : fmt_b.fl;
    const int sa = fl - fmt_a.fl, sb = fl - fmt_b.fl;
    if (sa > 40 || sb > 40) return FXPQ_ERR_RANGE;
    OutArgs o;
    fxpq_status st = make_out(out_mode, fmt_y, fl, o, h_out_scale);
    if (st != FXPQ_OK) return st;
    if (n_pix == 0) return FXPQ_OK;
    if (!d_a || !d_b || !d_y) return FXPQ_ERR_INVALID_ARG;
    eltwise_kernel<<<grid_for(n_pix * Cp), 256, 0, as_stream(stream)>>>(
        static_cast<const __half*>(d_a), planes_of(fmt_a), sa, static_cast<const __half*>(d_b), planes_of(fmt_b), sb,
        n_pix, Cp, relu, o, d_y);
    return after_launch("eltwise");
}

extern "C" fxpq_status fxpq_avgpool(const void* d_x, int32_t N, int32_t H, int32_t W, int32_t Cp, fxpq_fmt fmt_x,
                                    int32_t recip_code, fxpq_fmt fmt_recip, int32_t out_mode, fxpq_fmt fmt_y,
                                    void* d_y, int32_t* h_out_scale, void* stream) {
    if (N < 0 || H < 1 || W < 1 || Cp < 1 || (Cp % 8) || !fmt_ok(fmt_x) || !fmt_ok(fmt_recip))
        return FXPQ_ERR_INVALID_ARG;
    if (recip_code < qmin_of(fmt_recip) || recip_code > qmax_of(fmt_recip)) return FXPQ_ERR_INVALID_ARG;
    OutArgs o;
    fxpq_status st = make_out(out_mode, fmt_y, fmt_x.fl + fmt_recip.fl, o, h_out_scale);
    if (st != FXPQ_OK) return st;
    if (N == 0) return FXPQ_OK;
    if (!d_x || !d_y) return FXPQ_ERR_INVALID_ARG;
    avgpool_kernel<<<grid_for((long long)N * Cp), 256, 0, as_stream(stream)>>>(
        static_cast<const __half*>(d_x), N, H * W, Cp, planes_of(fmt_x), (long long)recip_code, o, d_y);
    return after_launch("avgpool");
}

extern "C" fxpq_status fxpq_qlayer(const int64_t* d_v, int64_t n, int32_t s, int32_t out_mode, fxpq_fmt fmt_y,
                                   void* d_y, void* stream) {
    if (n < 0 || s < -64 || s > 80) return FXPQ_ERR_INVALID_ARG;
    OutArgs o;
    const fxpq_status st = make_out(out_mode, fmt_y, s, o, nullptr);
    if (st != FXPQ_OK) return st;
    if (n == 0) return FXPQ_OK;
    if (!d_v || !d_y) return FXPQ_ERR_INVALID_ARG;
    qlayer_kernel<<<grid_for(n), 256, 0, as_stream(stream)>>>(reinterpret_cast<const long long*>(d_v), n, o, d_y);
    return after_launch("qlayer");
}

// ---------------------------------------------------------------- BN -> Scale (Sec. IV-A.1)
namespace fxpq {
namespace {

// aleph1 = gamma / r and aleph2 = beta - (gamma * mean) / r with r = sqrt(var + eps), every step one
// correctly rounded fp32 operation (the _rn intrinsics are IEEE round-to-nearest-even, so the
// result does not depend on contraction into fused multiply-adds).
__global__ void bn_to_scale_kernel(const float* __restrict__ g, const float* __restrict__ b,
                                   const float* __restrict__ mu, const float* __restrict__ var, long long n, float eps,
                                   float* __restrict__ a1, float* __restrict__ a2) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const float r = __fsqrt_rn(__fadd_rn(var[i], eps));
    a1[i] = __fdiv_rn(g[i], r);
    a2[i] = __fsub_rn(b[i], __fdiv_rn(__fmul_rn(g[i], mu[i]), r));
}

}  // namespace
}  // namespace fxpq

extern "C" fxpq_status fxpq_bn_to_scale(const float* d_gamma, const float* d_beta, const float* d_mean,
                                        const float* d_var, int64_t n, float eps, float* d_aleph1, float* d_aleph2,
                                        void* stream) {
    using namespace fxpq;
    if (n < 0 || !(eps >= 0.0f)) return FXPQ_ERR_INVALID_ARG;
    if (n == 0) return FXPQ_OK;
    if (!d_gamma || !d_beta || !d_mean || !d_var || !d_aleph1 || !d_aleph2) return FXPQ_ERR_INVALID_ARG;
    const int T = 256;
    bn_to_scale_kernel<<<(unsigned)((n + T - 1) / T), T, 0, as_stream(stream)>>>(d_gamma, d_beta, d_mean, d_var, n,
                                                                                 eps, d_aleph1, d_aleph2);
    return after_launch("bn_to_scale");
}
