// fxpq_fopt.cu -- the forward optimizer's FP32 side (Sec. IV-C, Alg. 1 and its cost F): while one
// data-structure's QPs are searched, every later layer runs in FP32, and the cost needs each
// data-structure's quantization error, range and dispersion and the logits' top-1 ties.
//   conv / max-pool / eltwise / global avg-pool in fp32 (NHWC, true channel counts);
//   code tensors -> fp32 values; fp32 bias + ReLU after an integer contraction;
//   per-data-structure statistics (L of Eq. DSB_QE at one format, min, max, per-sample moments);
//   top-1 tie counts of logits (fp32 or exact int64).
#include <math.h>

#include "fxpq_common.cuh"

namespace fxpq {
namespace {

// ------------------------------------------------------------------ fp32 implicit-GEMM convolution
// Tile 128 output pixels x BN output channels (BN = 128 for wide layers, 64 otherwise), 8 reduction
// steps per stage (double-buffered shared memory), 256 threads with 8 x BN/16 outputs each (64 or 32
// FMAs per 16 or 12 shared-memory words).  x: [N, H, W, C]; w: [K, R*S*C] (KRSC); y: [N, P, Q, K].
// When C % 8 == 0 a stage's 8 reduction steps are 8 channels of one tap, loaded as float4.
constexpr int CF_BM = 128, CF_BK = 8;

struct ConvF32Args {
    const float* x;
    const float* w;
    const float* bias;
    float* y;
    int N, H, W, C, K, R, S, stride, pad, P, Q, relu;
    long long M;
};

template <int CF_BN>
__global__ void __launch_bounds__(256) conv_f32_kernel(const ConvF32Args a) {
    constexpr int TN = CF_BN / 16;  // output channels per thread
    __shared__ __align__(16) float sa[2][CF_BK][CF_BM];
    __shared__ __align__(16) float sb[2][CF_BK][CF_BN];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const long long m0 = (long long)blockIdx.x * CF_BM;
    const int n0 = blockIdx.y * CF_BN;
    const int RSC = a.R * a.S * a.C;
    // staging: thread t loads row t / 2 of the A tile (and of the B tile when BN = 128; rows t / 4 with
    // two columns each when BN = 64), reduction columns 4 (t % 2) .. + 3
    const int lr = threadIdx.x >> 1, lk = (threadIdx.x & 1) * 4;
    const int br = CF_BN == 128 ? lr : (threadIdx.x >> 2), bk = CF_BN == 128 ? lk : (threadIdx.x & 3) * 2;
    const long long m = m0 + lr;
    const bool mok = m < a.M;
    int pn = 0, pp = 0, pq = 0;
    if (mok) {
        pn = (int)(m / ((long long)a.P * a.Q));
        const int rem = (int)(m - (long long)pn * a.P * a.Q);
        pp = rem / a.Q;
        pq = rem - pp * a.Q;
    }
    const int o = n0 + br;
    const bool ook = o < a.K;
    const bool vecA = (a.C % 8) == 0, vecB = (RSC % 4) == 0;
    float ra[4], rb[4];
    auto load = [&](int k0) {
        if (vecA) {
            const int rs = k0 / a.C, c = k0 - rs * a.C + lk;
            const int s = rs % a.S, r = rs / a.S;
            const int h = pp * a.stride + r - a.pad, ww = pq * a.stride + s - a.pad;
            if (mok && k0 < RSC && h >= 0 && h < a.H && ww >= 0 && ww < a.W) {
                const float4 v =
                    *reinterpret_cast<const float4*>(a.x + (((long long)pn * a.H + h) * a.W + ww) * a.C + c);
                ra[0] = v.x, ra[1] = v.y, ra[2] = v.z, ra[3] = v.w;
            } else {
                ra[0] = ra[1] = ra[2] = ra[3] = 0.0f;
            }
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int kk = k0 + lk + e;
                float v = 0.0f;
                if (mok && kk < RSC) {
                    const int c = kk % a.C, rs = kk / a.C;
                    const int s = rs % a.S, r = rs / a.S;
                    const int h = pp * a.stride + r - a.pad, ww = pq * a.stride + s - a.pad;
                    if (h >= 0 && h < a.H && ww >= 0 && ww < a.W)
                        v = a.x[(((long long)pn * a.H + h) * a.W + ww) * a.C + c];
                }
                ra[e] = v;
            }
        }
        const int kb = k0 + bk;
        constexpr int NB = CF_BN == 128 ? 4 : 2;
        if (CF_BN == 128 && vecB && ook && kb + 3 < RSC) {
            const float4 v = *reinterpret_cast<const float4*>(a.w + (long long)o * RSC + kb);
            rb[0] = v.x, rb[1] = v.y, rb[2] = v.z, rb[3] = v.w;
        } else {
#pragma unroll
            for (int e = 0; e < NB; ++e) rb[e] = (ook && kb + e < RSC) ? a.w[(long long)o * RSC + kb + e] : 0.0f;
        }
    };
    auto store = [&](int buf) {
#pragma unroll
        for (int e = 0; e < 4; ++e) sa[buf][lk + e][lr] = ra[e];
#pragma unroll
        for (int e = 0; e < (CF_BN == 128 ? 4 : 2); ++e) sb[buf][bk + e][br] = rb[e];
    };
    float acc[8][TN];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = 0.0f;
    load(0);
    store(0);
    __syncthreads();
    int buf = 0;
    for (int k0 = 0; k0 < RSC; k0 += CF_BK) {
        const bool more = k0 + CF_BK < RSC;
        if (more) load(k0 + CF_BK);  // next stage's global loads in flight during this stage's FMAs
#pragma unroll
        for (int kk = 0; kk < CF_BK; ++kk) {
            const float4 a0 = *reinterpret_cast<const float4*>(&sa[buf][kk][ty * 8]);
            const float4 a1 = *reinterpret_cast<const float4*>(&sa[buf][kk][ty * 8 + 4]);
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            float bv[TN];
#pragma unroll
            for (int q = 0; q < TN / 4; ++q) {
                const float4 b = *reinterpret_cast<const float4*>(&sb[buf][kk][tx * TN + 4 * q]);
                bv[4 * q] = b.x, bv[4 * q + 1] = b.y, bv[4 * q + 2] = b.z, bv[4 * q + 3] = b.w;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        if (more) {
            store(buf ^ 1);
            __syncthreads();
            buf ^= 1;
        }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const long long mm = m0 + ty * 8 + i;
        if (mm >= a.M) continue;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int oo = n0 + tx * TN + j;
            if (oo >= a.K) continue;
            float v = acc[i][j];
            if (a.bias) v += a.bias[oo];
            if (a.relu) v = fmaxf(v, 0.0f);
            a.y[mm * a.K + oo] = v;
        }
    }
}

// Small layers (too few 128-row tiles to occupy the SMs): 64 x 64 tiles, 4 x 4 outputs per thread.
constexpr int SF_BM = 64, SF_BN = 64, SF_BK = 16;

__global__ void __launch_bounds__(256) conv_f32_small_kernel(const ConvF32Args a) {
    __shared__ float sa[SF_BK][SF_BM + 4];
    __shared__ float sb[SF_BK][SF_BN + 4];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const long long m0 = (long long)blockIdx.x * SF_BM;
    const int n0 = blockIdx.y * SF_BN;
    const int RSC = a.R * a.S * a.C;
    // the A element this thread stages: pixel row (threadIdx.x / 4) and reduction columns 4 * (tid % 4) ..
    const int lr = threadIdx.x >> 2, lk = (threadIdx.x & 3) * 4;
    const long long m = m0 + lr;
    int pn = 0, pp = 0, pq = 0;
    if (m < a.M) {
        pn = (int)(m / ((long long)a.P * a.Q));
        const int rem = (int)(m - (long long)pn * a.P * a.Q);
        pp = rem / a.Q;
        pq = rem - pp * a.Q;
    }
    float acc[4][4] = {};
    for (int k0 = 0; k0 < RSC; k0 += SF_BK) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int kk = k0 + lk + e;
            float v = 0.0f;
            if (m < a.M && kk < RSC) {
                const int c = kk % a.C, rs = kk / a.C;
                const int s = rs % a.S, r = rs / a.S;
                const int h = pp * a.stride + r - a.pad, ww = pq * a.stride + s - a.pad;
                if (h >= 0 && h < a.H && ww >= 0 && ww < a.W) v = a.x[(((long long)pn * a.H + h) * a.W + ww) * a.C + c];
            }
            sa[lk + e][lr] = v;
            const int o = n0 + lr;
            sb[lk + e][lr] = (o < a.K && kk < RSC) ? a.w[(long long)o * RSC + kk] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < SF_BK; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = sa[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bv[j] = sb[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const long long mm = m0 + ty * 4 + i;
        if (mm >= a.M) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int o = n0 + tx * 4 + j;
            if (o >= a.K) continue;
            float v = acc[i][j];
            if (a.bias) v += a.bias[o];
            if (a.relu) v = fmaxf(v, 0.0f);
            a.y[mm * a.K + o] = v;
        }
    }
}

__global__ void maxpool_f32_kernel(const float* __restrict__ x, int N, int H, int W, int C, int k, int stride, int pad,
                                   int P, int Q, float* __restrict__ y) {
    const long long total = (long long)N * P * Q * C;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        const long long pix = i / C;
        const int q = (int)(pix % Q), p = (int)((pix / Q) % P);
        const long long n = pix / ((long long)P * Q);
        float best = -INFINITY;
        for (int r = 0; r < k; ++r) {
            const int h = p * stride + r - pad;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < k; ++s) {
                const int w = q * stride + s - pad;
                if (w >= 0 && w < W) best = fmaxf(best, x[((n * H + h) * W + w) * C + c]);
            }
        }
        y[i] = best;
    }
}

__global__ void eltwise_f32_kernel(const float* __restrict__ a, const float* __restrict__ b, long long n, int relu,
                                   float* __restrict__ y) {
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
        const float v = a[i] + b[i];
        y[i] = relu ? fmaxf(v, 0.0f) : v;
    }
}

// one thread per (n, c): the mean over H x W (sum in fp32, then divided by H W)
__global__ void avgpool_f32_kernel(const float* __restrict__ x, int N, int HW, int C, float* __restrict__ y) {
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (long long)N * C) return;
    const long long n = i / C;
    const int c = (int)(i % C);
    float s = 0.0f;
    for (int p = 0; p < HW; ++p) s += x[(n * HW + p) * C + c];
    y[i] = s / (float)HW;
}

// fp16 code tensor [npix, Cp] (planes) -> fp32 values [npix, C]; the binary quantizer's codes decode
// 0 -> +1, -1 -> -1
__global__ void dequantize_kernel(const __half* __restrict__ codes, long long npix, int Cp, int C, int planes, float scale,
                                  int binary, float* __restrict__ y) {
    const long long total = npix * C;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
        const long long pix = i / C;
        const int c = (int)(i - pix * C);
        int code = code_get(codes, pix * Cp + c, planes, npix * Cp);
        if (binary) code = 2 * code + 1;
        y[i] = (float)code * scale;  // exact: |code| < 2^17 and scale a power of two
    }
}

__global__ void bias_relu_f32_kernel(float* __restrict__ y, long long npix, int K, const float* __restrict__ bias,
                                     int relu) {
    const long long total = npix * K;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
        float v = y[i];
        if (bias) v += bias[i % K];
        y[i] = relu ? fmaxf(v, 0.0f) : v;
    }
}

__device__ __forceinline__ unsigned ord_key(float x) {
    const unsigned u = __float_as_uint(x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// ---------------------------------------------------------------- data-structure statistics (batched)
// Items of fxpq_ds_stats_batch, split into work units of DS_CHUNK values of one sample each; the unit
// prefix of each item sits in the kernel parameters.  Three passes: per-unit sums; per-unit sums of
// squared deviations from the sample mean (the mean from the first pass's sums, in unit order), the
// quantization error and the extremes; per-item records from the units in order.  No floating-point
// atomics: every total is formed in a fixed order.
constexpr int DS_MAX_ITEMS = 128;  // items per launch group
constexpr long long DS_CHUNK = 1 << 16;
constexpr int DS_T = 256;

struct DsItemDev {
    const float* x;
    double* out;
    long long nu;
    int n_samples, k, S, fl;
    int chunks;  // units per sample
    int unit0;   // first unit of the item (within its launch group)
};
struct DsBatchDev {
    int n;
    DsItemDev it[DS_MAX_ITEMS];
    int unit_end;  // units of the launch group
};

// Per-unit scratch of one launch group.
struct DsUnit {
    double sum, m2, l2;
    unsigned mn, mx;
};

__device__ __forceinline__ int ds_item_of(const DsBatchDev& B, int u) {
    int lo = 0, hi = B.n - 1;  // last item whose unit0 <= u
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (B.it[mid].unit0 <= u) lo = mid; else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ double ds_block_sum(double v, double* red) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) red[w] = v;
    __syncthreads();
    double t = 0.0;
    if (threadIdx.x == 0)
        for (int i = 0; i < DS_T / 32; ++i) t += red[i];  // fixed order
    return t;  // valid in thread 0
}

__global__ void __launch_bounds__(DS_T) ds_sum_kernel(const __grid_constant__ DsBatchDev B, DsUnit* units) {
    __shared__ double red[DS_T / 32];
    const int u = blockIdx.x;
    const DsItemDev& it = B.it[ds_item_of(B, u)];
    const int rel = u - it.unit0, s = rel / it.chunks, c = rel % it.chunks;
    const float* xs = it.x + (long long)s * it.nu;
    const long long i0 = (long long)c * DS_CHUNK, i1 = min(i0 + DS_CHUNK, it.nu);
    double acc = 0.0;
    for (long long i = i0 + threadIdx.x; i < i1; i += DS_T) acc += (double)xs[i];
    const double t = ds_block_sum(acc, red);
    if (threadIdx.x == 0) units[u].sum = t;
}

__global__ void __launch_bounds__(DS_T) ds_dev_kernel(const __grid_constant__ DsBatchDev B, DsUnit* units) {
    __shared__ double red[DS_T / 32];
    __shared__ unsigned kmn, kmx;
    const int u = blockIdx.x;
    const DsItemDev& it = B.it[ds_item_of(B, u)];
    const int rel = u - it.unit0, s = rel / it.chunks, c = rel % it.chunks;
    const float* xs = it.x + (long long)s * it.nu;
    const long long i0 = (long long)c * DS_CHUNK, i1 = min(i0 + DS_CHUNK, it.nu);
    // the sample mean from the first pass's unit sums, in unit order
    const int first = it.unit0 + s * it.chunks;
    double sum = 0.0;
    for (int v = 0; v < it.chunks; ++v) sum += units[first + v].sum;
    const double mean = sum / (double)it.nu;
    const double scale = ldexp(1.0, it.fl), inv = ldexp(1.0, -it.fl);
    const double lo = it.S ? -ldexp(1.0, it.k - 1) : 0.0, hi = ldexp(1.0, it.k - it.S) - 1.0;
    const bool binary = it.k == 1 && it.S == 1;
    double m2 = 0.0, l2 = 0.0;
    unsigned mn = 0xFFFFFFFFu, mx = 0u;
    for (long long i = i0 + threadIdx.x; i < i1; i += DS_T) {
        const float v = xs[i];
        const double d = (double)v;
        const double q = binary ? (v < 0.0f ? -inv : inv) : fmin(fmax(nearbyint(d * scale), lo), hi) * inv;
        const double e = d - q, dv = d - mean;
        l2 += e * e;
        m2 += dv * dv;
        const unsigned key = ord_key(v);
        mn = min(mn, key);
        mx = max(mx, key);
    }
    if (threadIdx.x == 0) {
        kmn = 0xFFFFFFFFu;
        kmx = 0u;
    }
    const double tm2 = ds_block_sum(m2, red);
    const double tl2 = ds_block_sum(l2, red);
    mn = __reduce_min_sync(0xFFFFFFFFu, mn);
    mx = __reduce_max_sync(0xFFFFFFFFu, mx);
    if ((threadIdx.x & 31) == 0) {
        atomicMin(&kmn, mn);
        atomicMax(&kmx, mx);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        units[u].m2 = tm2;
        units[u].l2 = tl2;
        units[u].mn = kmn;
        units[u].mx = kmx;
    }
}

__device__ __forceinline__ float ds_key_value(unsigned k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// One thread per item: its record from its units, in unit order.
__global__ void ds_finish_kernel(const __grid_constant__ DsBatchDev B, const DsUnit* units) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= B.n) return;
    const DsItemDev& it = B.it[i];
    double l2 = 0.0;
    unsigned mn = 0xFFFFFFFFu, mx = 0u;
    for (int s = 0; s < it.n_samples; ++s) {
        double sum = 0.0, m2 = 0.0;
        for (int c = 0; c < it.chunks; ++c) {
            const DsUnit& q = units[it.unit0 + s * it.chunks + c];
            sum += q.sum;
            m2 += q.m2;
            l2 += q.l2;
            mn = min(mn, q.mn);
            mx = max(mx, q.mx);
        }
        it.out[3 + 2 * s] = sum / (double)it.nu;
        it.out[4 + 2 * s] = m2;
    }
    it.out[0] = l2;
    it.out[1] = (double)ds_key_value(mn);
    it.out[2] = (double)ds_key_value(mx);
}

// ---------------------------------------------------------------- the cost F of Alg. 1
constexpr int COST_MAX_TERMS = 512;
struct CostTermDev {
    long long offset, nu;
    int n_samples, layer;
};
struct CostTerms {
    int n;
    CostTermDev t[COST_MAX_TERMS];
};

// One block per candidate; thread 0 adds the terms in order (a few dozen per network).
__global__ void fopt_cost_kernel(const double* __restrict__ stats, long long cand_stride,
                                 const __grid_constant__ CostTerms T, const int* __restrict__ ties, int N,
                                 int n_classes, double* __restrict__ cost) {
    const int c = blockIdx.x;
    const double* base = stats + (long long)c * cand_stride;
    __shared__ unsigned n_tied, extra;
    if (threadIdx.x == 0) n_tied = extra = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        const int k = ties[(long long)c * N + i];
        if (k > 1) atomicAdd(&n_tied, 1u);
        atomicAdd(&extra, (unsigned)(k - 1));
    }
    __syncthreads();
    if (threadIdx.x != 0) return;
    double E = 0.0;
    int t0 = 0;
    while (t0 < T.n) {
        int t1 = t0;
        double den = 0.0;
        while (t1 < T.n && T.t[t1].layer == T.t[t0].layer) {  // one layer: sum of sigma nu
            const CostTermDev& q = T.t[t1];
            const double* r = base + q.offset;
            double sig = 0.0;
            for (int s = 0; s < q.n_samples; ++s) sig += sqrt(r[4 + 2 * s] / (double)q.nu);
            den += sig / q.n_samples * (double)q.nu;
            ++t1;
        }
        if (den > 0.0) {
            for (int t = t0; t < t1; ++t) {
                const CostTermDev& q = T.t[t];
                const double* r = base + q.offset;
                const double R = r[2] - r[1];
                if (R == 0.0) continue;
                double sig = 0.0;
                for (int s = 0; s < q.n_samples; ++s) sig += sqrt(r[4 + 2 * s] / (double)q.nu);
                E += (sig / q.n_samples * (double)q.nu / den) * r[0] / R;
            }
        }
        t0 = t1;
    }
    const double uc = (double)n_tied / N, mp = (double)extra / ((double)N * n_classes);
    cost[4 * c + 0] = E + uc + mp;
    cost[4 * c + 1] = E;
    cost[4 * c + 2] = uc;
    cost[4 * c + 3] = mp;
}

// one warp per sample: the number of classes whose logit equals the sample's largest
template <typename T>
__global__ void top1_ties_kernel(const T* __restrict__ logits, int N, int C, int32_t* __restrict__ counts) {
    const int n = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (n >= N) return;
    const T* row = logits + (long long)n * C;
    T best = row[0];
    for (int c = lane; c < C; c += 32) best = row[c] > best ? row[c] : best;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const T o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        best = o > best ? o : best;
    }
    int cnt = 0;
    for (int c = lane; c < C; c += 32) cnt += row[c] == best ? 1 : 0;
    cnt = __reduce_add_sync(0xFFFFFFFFu, (unsigned)cnt);
    if (lane == 0) counts[n] = cnt;
}

__global__ void nchw_to_nhwc_kernel(const float* __restrict__ x, int N, int C, int HW, float* __restrict__ y) {
    const long long total = (long long)N * C * HW;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        const long long pix = i / C;  // n * HW + p
        const long long n = pix / HW;
        y[i] = x[(n * C + c) * HW + (pix - n * HW)];
    }
}

int grid_of(long long work) {
    long long b = (work + 255) / 256;
    if (b < 1) b = 1;
    if (b > 152LL * 16) b = 152LL * 16;
    return (int)b;
}

}  // namespace
}  // namespace fxpq

using namespace fxpq;

extern "C" fxpq_status fxpq_conv_f32(const fxpq_conv_f32_desc* h_desc, const float* d_x, const float* d_w,
                                     const float* d_bias, float* d_y, void* stream) {
    if (!h_desc) return FXPQ_ERR_INVALID_ARG;
    const fxpq_conv_f32_desc& d = *h_desc;
    if (d.N < 0 || d.H < 1 || d.W < 1 || d.C < 1 || d.K < 1 || d.R < 1 || d.S < 1 || d.stride < 1 || d.pad < 0)
        return FXPQ_ERR_INVALID_ARG;
    const int P = (d.H + 2 * d.pad - d.R) / d.stride + 1, Q = (d.W + 2 * d.pad - d.S) / d.stride + 1;
    if (P < 1 || Q < 1) return FXPQ_ERR_INVALID_ARG;
    if (d.N > 0 && (!d_x || !d_w || !d_y)) return FXPQ_ERR_INVALID_ARG;
    ConvF32Args a{d_x, d_w, d_bias, d_y, d.N, d.H, d.W, d.C, d.K, d.R, d.S, d.stride, d.pad, P, Q, d.relu ? 1 : 0,
                  (long long)d.N * P * Q};
    if (a.M == 0) return FXPQ_OK;
    const long long big = ((a.M + CF_BM - 1) / CF_BM) * ((d.K + (d.K >= 128 ? 127 : 63)) / (d.K >= 128 ? 128 : 64));
    if (big < 152) {
        dim3 grid((unsigned)((a.M + SF_BM - 1) / SF_BM), (unsigned)((d.K + SF_BN - 1) / SF_BN));
        conv_f32_small_kernel<<<grid, 256, 0, as_stream(stream)>>>(a);
    } else if (d.K >= 128) {
        dim3 grid((unsigned)((a.M + CF_BM - 1) / CF_BM), (unsigned)((d.K + 127) / 128));
        conv_f32_kernel<128><<<grid, 256, 0, as_stream(stream)>>>(a);
    } else {
        dim3 grid((unsigned)((a.M + CF_BM - 1) / CF_BM), (unsigned)((d.K + 63) / 64));
        conv_f32_kernel<64><<<grid, 256, 0, as_stream(stream)>>>(a);
    }
    return after_launch("conv_f32");
}

extern "C" fxpq_status fxpq_maxpool_f32(const float* d_x, int32_t N, int32_t H, int32_t W, int32_t C, int32_t k,
                                        int32_t stride, int32_t pad, float* d_y, void* stream) {
    if (N < 0 || H < 1 || W < 1 || C < 1 || k < 1 || stride < 1 || pad < 0 || pad >= k) return FXPQ_ERR_INVALID_ARG;
    const int P = (H + 2 * pad - k) / stride + 1, Q = (W + 2 * pad - k) / stride + 1;
    if (P < 1 || Q < 1 || (N > 0 && (!d_x || !d_y))) return FXPQ_ERR_INVALID_ARG;
    const long long total = (long long)N * P * Q * C;
    if (total == 0) return FXPQ_OK;
    maxpool_f32_kernel<<<grid_of(total), 256, 0, as_stream(stream)>>>(d_x, N, H, W, C, k, stride, pad, P, Q, d_y);
    return after_launch("maxpool_f32");
}

extern "C" fxpq_status fxpq_eltwise_f32(const float* d_a, const float* d_b, int64_t n, int32_t relu, float* d_y,
                                        void* stream) {
    if (n < 0 || (n > 0 && (!d_a || !d_b || !d_y))) return FXPQ_ERR_INVALID_ARG;
    if (n == 0) return FXPQ_OK;
    eltwise_f32_kernel<<<grid_of(n), 256, 0, as_stream(stream)>>>(d_a, d_b, n, relu, d_y);
    return after_launch("eltwise_f32");
}

extern "C" fxpq_status fxpq_avgpool_f32(const float* d_x, int32_t N, int32_t H, int32_t W, int32_t C, float* d_y,
                                        void* stream) {
    if (N < 0 || H < 1 || W < 1 || C < 1 || (N > 0 && (!d_x || !d_y))) return FXPQ_ERR_INVALID_ARG;
    const long long total = (long long)N * C;
    if (total == 0) return FXPQ_OK;
    avgpool_f32_kernel<<<(unsigned)((total + 255) / 256), 256, 0, as_stream(stream)>>>(d_x, N, H * W, C, d_y);
    return after_launch("avgpool_f32");
}

extern "C" fxpq_status fxpq_dequantize(const void* d_codes, int64_t npix, int32_t Cp, int32_t C, fxpq_fmt fmt,
                                       float* d_y, void* stream) {
    if (npix < 0 || C < 1 || Cp < C || !fmt_ok1(fmt) || (npix > 0 && (!d_codes || !d_y))) return FXPQ_ERR_INVALID_ARG;
    if (npix == 0) return FXPQ_OK;
    dequantize_kernel<<<grid_of(npix * C), 256, 0, as_stream(stream)>>>(
        static_cast<const __half*>(d_codes), npix, Cp, C, planes_of(fmt), ldexpf(1.0f, -fmt.fl),
        fmt.bits == 1 && fmt.is_signed == 1, d_y);
    return after_launch("dequantize");
}

extern "C" fxpq_status fxpq_bias_relu_f32(float* d_y, int64_t npix, int32_t K, const float* d_bias, int32_t relu,
                                          void* stream) {
    if (npix < 0 || K < 1 || (npix > 0 && !d_y)) return FXPQ_ERR_INVALID_ARG;
    if (npix == 0) return FXPQ_OK;
    bias_relu_f32_kernel<<<grid_of(npix * K), 256, 0, as_stream(stream)>>>(d_y, npix, K, d_bias, relu);
    return after_launch("bias_relu_f32");
}

namespace {
// Units of one item (DS_CHUNK values of one sample each), or -1 for an invalid item.
long long ds_units(const fxpq_ds_item& it) {
    if (it.n_samples < 1 || it.n_samples > 65535 || it.nu < 1 || !fxpq::fmt_ok1(it.fmt, 32) || !it.d_x || !it.d_out)
        return -1;
    return (long long)it.n_samples * ((it.nu + DS_CHUNK - 1) / DS_CHUNK);
}
}  // namespace

extern "C" size_t fxpq_ds_stats_batch_workspace(const fxpq_ds_item* h_items, int32_t n_items) {
    if (n_items < 1 || n_items > 4096 || !h_items) return 0;
    long long most = 0;  // the largest launch group's units
    for (int i0 = 0; i0 < n_items; i0 += DS_MAX_ITEMS) {
        long long u = 0;
        for (int i = i0; i < n_items && i < i0 + DS_MAX_ITEMS; ++i) {
            const long long v = ds_units(h_items[i]);
            if (v < 0) return 0;
            u += v;
        }
        most = u > most ? u : most;
    }
    return ((size_t)most * sizeof(DsUnit) + 255) / 256 * 256;
}

extern "C" fxpq_status fxpq_ds_stats_batch(const fxpq_ds_item* h_items, int32_t n_items, void* d_ws, size_t ws_bytes,
                                           void* stream) {
    if (n_items < 1 || n_items > 4096 || !h_items) return FXPQ_ERR_INVALID_ARG;
    for (int i = 0; i < n_items; ++i)
        if (ds_units(h_items[i]) < 0) return FXPQ_ERR_INVALID_ARG;
    const size_t need = fxpq_ds_stats_batch_workspace(h_items, n_items);
    if (!d_ws || ws_bytes < need || !aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    cudaStream_t s = as_stream(stream);
    DsUnit* units = static_cast<DsUnit*>(d_ws);
    for (int i0 = 0; i0 < n_items; i0 += DS_MAX_ITEMS) {
        DsBatchDev B;
        B.n = 0;
        long long u = 0;
        for (int i = i0; i < n_items && i < i0 + DS_MAX_ITEMS; ++i) {
            const fxpq_ds_item& h = h_items[i];
            DsItemDev& d = B.it[B.n++];
            d.x = h.d_x;
            d.out = h.d_out;
            d.nu = h.nu;
            d.n_samples = h.n_samples;
            d.k = h.fmt.bits;
            d.S = h.fmt.is_signed;
            d.fl = h.fmt.fl;
            d.chunks = (int)((h.nu + DS_CHUNK - 1) / DS_CHUNK);
            d.unit0 = (int)u;
            u += ds_units(h);
        }
        if (u > 0x7FFFFFFFLL) return FXPQ_ERR_INVALID_ARG;
        B.unit_end = (int)u;
        ds_sum_kernel<<<(unsigned)u, DS_T, 0, s>>>(B, units);
        fxpq_status st = after_launch("ds_sum");
        if (st != FXPQ_OK) return st;
        ds_dev_kernel<<<(unsigned)u, DS_T, 0, s>>>(B, units);
        st = after_launch("ds_dev");
        if (st != FXPQ_OK) return st;
        ds_finish_kernel<<<(B.n + 127) / 128, 128, 0, s>>>(B, units);
        st = after_launch("ds_finish");
        if (st != FXPQ_OK) return st;
    }
    return FXPQ_OK;
}

extern "C" fxpq_status fxpq_fopt_cost(const double* d_stats, int64_t cand_stride, const fxpq_cost_term* h_terms,
                                      int32_t n_terms, const int32_t* d_ties, int32_t N, int32_t n_classes,
                                      int32_t n_cand, double* d_cost, void* stream) {
    if (n_terms < 0 || n_terms > COST_MAX_TERMS || (n_terms > 0 && !h_terms) || N < 1 || n_classes < 1 || n_cand < 1 ||
        cand_stride < 0 || !d_stats || !d_ties || !d_cost)
        return FXPQ_ERR_INVALID_ARG;
    CostTerms T;
    T.n = n_terms;
    for (int i = 0; i < n_terms; ++i) {
        const fxpq_cost_term& h = h_terms[i];
        if (h.offset < 0 || h.nu < 1 || h.n_samples < 1) return FXPQ_ERR_INVALID_ARG;
        T.t[i] = CostTermDev{h.offset, h.nu, h.n_samples, h.layer};
    }
    fopt_cost_kernel<<<n_cand, 128, 0, as_stream(stream)>>>(d_stats, cand_stride, T, d_ties, N, n_classes, d_cost);
    return after_launch("fopt_cost");
}

extern "C" fxpq_status fxpq_top1_ties(const void* d_logits, int32_t is_int64, int32_t N, int32_t C, int32_t* d_counts,
                                      void* stream) {
    if (N < 0 || C < 1 || (N > 0 && (!d_logits || !d_counts))) return FXPQ_ERR_INVALID_ARG;
    if (N == 0) return FXPQ_OK;
    const unsigned blocks = (unsigned)((N + 7) / 8);
    if (is_int64)
        top1_ties_kernel<long long><<<blocks, 256, 0, as_stream(stream)>>>(static_cast<const long long*>(d_logits), N, C,
                                                                           d_counts);
    else
        top1_ties_kernel<float><<<blocks, 256, 0, as_stream(stream)>>>(static_cast<const float*>(d_logits), N, C,
                                                                       d_counts);
    return after_launch("top1_ties");
}

extern "C" fxpq_status fxpq_nchw_to_nhwc_f32(const float* d_x, int32_t N, int32_t C, int32_t H, int32_t W, float* d_y,
                                             void* stream) {
    if (N < 0 || C < 1 || H < 1 || W < 1 || (N > 0 && (!d_x || !d_y))) return FXPQ_ERR_INVALID_ARG;
    const long long total = (long long)N * C * H * W;
    if (total == 0) return FXPQ_OK;
    nchw_to_nhwc_kernel<<<grid_of(total), 256, 0, as_stream(stream)>>>(d_x, N, C, H * W, d_y);
    return after_launch("nchw_to_nhwc");
}
