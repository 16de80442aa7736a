// fxpq_conv.cuh -- arguments and fused epilogue of the C-Block kernels (Sec. IV-B).
#pragma once

#include "fxpq_common.cuh"

namespace fxpq {

struct ConvArgs {
    const __half* x;   // NHWC fp16 code tensor, px planes of [N, H, W, Cp]
    const __half* w;   // KRSC fp16 code tensor, pw planes of [K, R, S, Cp]
    const int32_t* bias;
    void* y;           // CODES: fp16, py planes of [M, K]; ACC64: int64 [M, K]; F32: float [M, K]
    int N, H, W, Cp, K, R, S, stride, pad, P, Q;
    long long M;       // N * P * Q output rows
    long long x_ps, w_ps;  // plane strides (elements) of x and w
    int px, pw, py;
    int relu, out_mode, has_bias;
    int delta;         // bias alignment: s_acc - fl_b
    int s_out;         // scale exponent after alignment
    int sh;            // FxP-QLayer right shift s_out - fl_y
    long long lo, hi;  // clip levels of fmt_y
    float f32_scale;   // 2^-s_out
    int v32;           // 1: qlayer_code32 applies (the host checked its 32-bit bounds)
    int bsh;           // bias shift of the 32-bit path (= delta)
    int sh32;          // right shift of the 32-bit path, relative to the accumulator's scale
    const int32_t* scale;  // Scale layer aleph1 codes [K] (has_scale)
    const int32_t* shift;  // Scale layer aleph2 codes [K]
    int has_scale;
    int delta2;        // aleph2 alignment: (scale after the bias) + fl_aleph1 - fl_aleph2
};

// Bias alignment (B << delta, or the accumulator shifted left when delta < 0), the Scale layer
// (v * aleph1, then aleph2 aligned the same way) and ReLU: the C-Block output before its FxP-QLayer,
// in units of 2^-s_out.  SC = false compiles the Scale layer out (for kernels the host launches only
// for layers without one).
template <bool SC = true>
__host__ __device__ __forceinline__ long long cblock_value(const ConvArgs& a, int k, long long v, int32_t bias) {
    if (a.has_bias) {
        const long long b = bias;
        if (a.delta >= 0)
            v += b << a.delta;
        else
            v = (v << (-a.delta)) + b;
    }
    if constexpr (SC) {
        if (a.has_scale) {
            v *= (long long)__ldg(a.scale + k);
            const long long h = __ldg(a.shift + k);
            if (a.delta2 >= 0)
                v += h << a.delta2;
            else
                v = (v << (-a.delta2)) + h;
        }
    }
    if (a.relu && v < 0) v = 0;
    return v;
}

// FxP-QLayer: v * 2^(fl_y - s_out) rounded half to even on the dropped bits, clipped to fmt_y.
__host__ __device__ __forceinline__ int qlayer_code(const ConvArgs& a, long long v) {
    long long q;
    if (a.sh > 0) {
        q = rne_shift(v, a.sh);
    } else {
        const int l = -a.sh;  // left shift; saturate before it could overflow
        const long long lim = 1LL << 20;
        if (l >= 32 || v > lim || v < -lim)
            q = v > 0 ? a.hi : (v < 0 ? a.lo : 0);
        else
            q = v << l;
    }
    q = q < a.lo ? a.lo : (q > a.hi ? a.hi : q);
    return (int)q;
}

// Bias alignment, ReLU and the FxP-QLayer in 32-bit arithmetic (valid when a.v32; the host checked
// the bounds).  The value, in units of 2^-s (s = fl_x + fl_w), is acc + B 2^-delta:
//   delta >= 0 (bsh = delta):   N = acc + (B << delta), phi = 0;
//   delta <  0 (bsh = delta):   N = acc + floor(B / 2^d), phi = (B mod 2^d) / 2^d in [0, 1), d = -delta;
// and the code is round_half_even((N + phi) / 2^sh32) with sh32 = s - fl_y >= 1.  Because
// 0 <= phi < 1, floor((N + phi) / 2^sh32) = N >> sh32, and against half = 2^(sh32-1) the remainder
// (N mod 2^sh32) + phi is above half iff rem > half or (rem == half and phi > 0), a tie iff
// rem == half and phi == 0.  ReLU: N + phi < 0 iff N < 0.
__host__ __device__ __forceinline__ int qlayer_code32(const ConvArgs& a, int acc, int32_t bias) {
    int N = acc;
    bool phi = false;
    if (a.has_bias) {
        if (a.bsh >= 0) {
            N += bias << a.bsh;
        } else {
            const int d = -a.bsh;
            N += bias >> d;
            phi = (bias & ((1 << d) - 1)) != 0;
        }
    }
    if (a.relu && N < 0) {
        N = 0;
        phi = false;
    }
    const int q = N >> a.sh32;
    const int rem = N & ((1 << a.sh32) - 1);
    const int half = 1 << (a.sh32 - 1);
    const bool up = rem > half || (rem == half && (phi || (q & 1)));
    const int c = max(q + (up ? 1 : 0), (int)a.lo);
    return min(c, (int)a.hi);
}

// Bias alignment, ReLU and the FxP-QLayer for one output value of row m, channel k.
__device__ __forceinline__ void cblock_epilogue_store(const ConvArgs& a, long long m, int k, long long v) {
    v = cblock_value(a, k, v, a.has_bias ? a.bias[k] : 0);
    if (a.out_mode == FXPQ_OUT_CODES) {
        code_put(static_cast<__half*>(a.y), m * a.K + k, a.py, a.M * a.K, qlayer_code(a, v));
    } else if (a.out_mode == FXPQ_OUT_ACC64) {
        static_cast<long long*>(a.y)[m * a.K + k] = v;
    } else {
        static_cast<float*>(a.y)[m * a.K + k] = __ll2float_rn(v) * a.f32_scale;
    }
}

fxpq_status plan_conv(const fxpq_conv_desc& d, const void* x, const void* w, const int32_t* bias, void* y,
                      ConvArgs& a, int32_t* out_scale, bool& need64);
fxpq_status launch_conv(const ConvArgs& a, const fxpq_conv_desc& d, bool need64, cudaStream_t st, void* ws,
                        size_t ws_bytes);
// Tensor-core path; sets launched = false when the shape needs the CUDA-core kernel instead.  ws (may be
// null): scratch for the split reduction of layers with too few tiles for the SMs.
fxpq_status launch_conv_tc(const ConvArgs& a, const fxpq_conv_desc& d, cudaStream_t st, bool& launched, void* ws,
                           size_t ws_bytes);
// Adds the ks integer shares part[s][M][K] (int32, or int64 when acc64) of a split reduction and applies
// the C-Block epilogue (cblock_epilogue_store) to every output.
fxpq_status launch_splitk_reduce(const ConvArgs& a, const void* part, int ks, bool acc64, cudaStream_t st);
// Scratch bytes a conv may use for its split reduction (0: never split).
size_t conv_split_ws_bytes(long long M, int K);

}  // namespace fxpq
