// fxpq_quant.cu -- quantizer Q (Sec. IV-B, Eq. fp_k_bit_quantization, Eq. clip, Eq. quantization_levels):
// fp32 tensors to integer codes, and to the fp16 code tensors of the network path.
#include <math.h>

#include "fxpq_common.cuh"

namespace fxpq {
namespace {

// ------------------------------------------------------------------------------------------
// Quantize kernels
// ------------------------------------------------------------------------------------------
struct QParams {
    float scale;  // 2^fl (exact power of two; fl in [-32, 40])
    float lo, hi; // Qmin, Qmax as floats (exact, |.| <= 2^16)
    int binary;   // signed 1-bit: the binary quantizer (Eq. fp_1_bit_quantization)
    int* status;
};

__device__ __forceinline__ int quant1(float x, const QParams& p, bool& bad) {
    if (!isfinite(x)) {
        bad = true;
        return 0;
    }
    if (p.binary) return x < 0.0f ? -1 : 0;  // -0.0 is not below zero
    // x * 2^fl is exact unless it overflows (then it saturates) or falls below 2^-126 (then it
    // rounds to 0 either way); rintf rounds half to even.
    float y = rintf(x * p.scale);
    y = fminf(fmaxf(y, p.lo), p.hi);
    return __float2int_rn(y);
}

template <typename T>
__global__ void quantize_kernel(const float* __restrict__ x, long long n, QParams p, T* __restrict__ out) {
    bool bad = false;
    long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        out[i] = (T)quant1(x[i], p, bad);
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// 4 elements per thread with 128-bit loads (x 16-byte aligned, n % 4 == 0 handled by caller)
template <typename T>
__global__ void quantize_vec4_kernel(const float4* __restrict__ x, long long n4, QParams p, T* __restrict__ out) {
    bool bad = false;
    long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float4 v = __ldg(x + i);
        T* o = out + 4 * i;
        o[0] = (T)quant1(v.x, p, bad);
        o[1] = (T)quant1(v.y, p, bad);
        o[2] = (T)quant1(v.z, p, bad);
        o[3] = (T)quant1(v.w, p, bad);
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// Storage bits of one code: the integer itself, or (F16) the bit pattern of its fp16 value.
template <typename S, bool F16>
__device__ __forceinline__ S code_bits(int c) {
    if (F16) return (S)__half_as_ushort(__int2half_rn(c));
    return (S)c;
}

// Flat quantization, 16 codes per thread and iteration: four 16-byte loads issued together, the
// codes packed into sizeof(S) 16-byte stores.  x and out 16-byte aligned; the n % 16 tail is done
// element by element by the first threads of the grid.
template <typename S, bool F16>
__global__ void quantize_vec16_kernel(const float* __restrict__ x, long long n, QParams p, S* __restrict__ out) {
    bool bad = false;
    const long long n16 = n / 16;
    const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long stride = (long long)gridDim.x * blockDim.x;
    const float4* x4 = reinterpret_cast<const float4*>(x);
    uint4* o4 = reinterpret_cast<uint4*>(out);
    for (long long i = tid; i < n16; i += stride) {
        float4 v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] = __ldg(x4 + 4 * i + j);
        union {
            S s[16];
            uint4 u[sizeof(S)];
        } pk;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            pk.s[4 * j + 0] = code_bits<S, F16>(quant1(v[j].x, p, bad));
            pk.s[4 * j + 1] = code_bits<S, F16>(quant1(v[j].y, p, bad));
            pk.s[4 * j + 2] = code_bits<S, F16>(quant1(v[j].z, p, bad));
            pk.s[4 * j + 3] = code_bits<S, F16>(quant1(v[j].w, p, bad));
        }
#pragma unroll
        for (int q = 0; q < (int)sizeof(S); ++q) o4[sizeof(S) * i + q] = pk.u[q];
    }
    for (long long i = 16 * n16 + tid; i < n; i += stride) out[i] = code_bits<S, F16>(quant1(__ldg(x + i), p, bad));
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// rows x C fp32 -> fp16 code tensor: planes of [rows, Cp] (hi plane, then lo plane when k > 8)
__global__ void quantize_rows_f16_kernel(const float* __restrict__ x, long long rows, int C, int Cp, int planes,
                                         QParams p, __half* __restrict__ out) {
    bool bad = false;
    long long total = rows * (long long)Cp;
    long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
        long long r = i / Cp;
        int c = (int)(i - r * Cp);
        int code = c < C ? quant1(x[r * C + c], p, bad) : 0;
        code_put(out, i, planes, total, code);
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// Unpadded rows (C == Cp): the tensor is n = rows * C contiguous codes, n % 8 == 0; 8 codes per
// thread from two 16-byte loads, one 16-byte store per plane.
__global__ void quantize_rows_vec8_kernel(const float4* __restrict__ x, long long n8, int planes, QParams p,
                                          uint4* __restrict__ out) {
    bool bad = false;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n8; i += stride) {
        const float4 a = __ldg(x + 2 * i), b = __ldg(x + 2 * i + 1);
        const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int c0 = quant1(v[2 * e], p, bad), c1 = quant1(v[2 * e + 1], p, bad);
            if (planes == 1) {
                hi[e] = (uint32_t)__half_as_ushort(__int2half_rn(c0)) |
                        ((uint32_t)__half_as_ushort(__int2half_rn(c1)) << 16);
            } else {
                __half h0, l0, h1, l1;
                split_limbs(c0, h0, l0);
                split_limbs(c1, h1, l1);
                hi[e] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                lo[e] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
            }
        }
        out[i] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        if (planes == 2) out[n8 + i] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// NCHW fp32 -> NHWC fp16 codes, channels padded to Cp (a multiple of 8); one thread per pixel, each
// group of 8 channels written as one 16-byte store per plane
__global__ void quantize_images_kernel(const float* __restrict__ x, int N, int C, int H, int W, int Cp, int planes,
                                       QParams p, __half* __restrict__ out) {
    bool bad = false;
    const long long hw = (long long)H * W;
    const long long npix = (long long)N * hw;
    const long long stride = (long long)gridDim.x * blockDim.x;
    uint4* o = reinterpret_cast<uint4*>(out);
    const long long plane8 = npix * Cp / 8;  // plane stride in 16-byte units
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < npix; i += stride) {
        const long long n = i / hw;
        const long long pix = i - n * hw;
        for (int c0 = 0; c0 < Cp; c0 += 8) {
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                int code[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int c = c0 + 2 * e + h;
                    code[h] = c < C ? quant1(__ldg(x + (n * C + c) * hw + pix), p, bad) : 0;
                }
                if (planes == 1) {
                    hi[e] = (uint32_t)__half_as_ushort(__int2half_rn(code[0])) |
                            ((uint32_t)__half_as_ushort(__int2half_rn(code[1])) << 16);
                } else {
                    __half h0, l0, h1, l1;
                    split_limbs(code[0], h0, l0);
                    split_limbs(code[1], h1, l1);
                    hi[e] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                    lo[e] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
                }
            }
            const long long q = (i * Cp + c0) / 8;
            o[q] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            if (planes == 2) o[plane8 + q] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// max over rows of sum |code|: one block per row (grid-stride over rows), 8 codes per 16-byte load
__global__ void code_l1max_kernel(const uint4* __restrict__ codes, long long rows, long long L8,
                                  unsigned long long* __restrict__ out) {
    __shared__ long long red[32];
    for (long long r = blockIdx.x; r < rows; r += gridDim.x) {
        const uint4* row = codes + r * L8;
        long long sum = 0;
        for (long long i = threadIdx.x; i < L8; i += blockDim.x) {
            const uint4 v = __ldg(row + i);
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
            int part = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const __half2 h = *reinterpret_cast<const __half2*>(&w[j]);
                part += abs(__half2int_rn(__low2half(h))) + abs(__half2int_rn(__high2half(h)));
            }
            sum += part;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sum;
        __syncthreads();
        if (threadIdx.x < 32) {
            long long t = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
            if (threadIdx.x == 0) atomicMax(out, (unsigned long long)t);
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------------------------------------
// Batched parameter quantization with device-resident formats
// ------------------------------------------------------------------------------------------
constexpr int QB_MAX = 32;
constexpr int QB_FLAT_UNIT = 4096;  // elements per block of a flat item

struct QbItem {
    const float* x;
    void* out;
    long long* l1;
    const int* fl;
    const fxpq_stats* st;
    long long rows;
    int C, Cp, rpg, bits, kind;
};

struct QbBatch {
    int n;
    int unit0[QB_MAX + 1];  // first block of each item
    QbItem it[QB_MAX];
    int* status;
};

// One block per work unit: an output-channel group (rpg rows) of a row item, or QB_FLAT_UNIT elements of
// a flat item.  The format (k from the item, S and FL from the device) is read once per block.
__global__ void __launch_bounds__(256) quantize_batch_kernel(const __grid_constant__ QbBatch B) {
    int item = 0;
    while (item + 1 < B.n && (int)blockIdx.x >= B.unit0[item + 1]) ++item;
    const QbItem& I = B.it[item];
    const long long u = (long long)blockIdx.x - B.unit0[item];
    const int fl = *I.fl;
    const int S = I.st->is_signed;
    QParams p;
    p.scale = __int_as_float((127 + fl) << 23);  // 2^fl, fl in [-32, 40]
    p.lo = S ? -(float)(1 << (I.bits - 1)) : 0.0f;
    p.hi = (float)((1 << (I.bits - S)) - 1);
    p.binary = 0;  // batch items have k >= 2
    p.status = B.status;
    bool bad = false;
    if (I.kind == FXPQ_QB_FLAT_I32) {
        const long long e0 = u * QB_FLAT_UNIT;
        const long long e1 = min(e0 + QB_FLAT_UNIT, I.rows);
        int32_t* out = static_cast<int32_t*>(I.out);
        for (long long e = e0 + threadIdx.x; e < e1; e += blockDim.x) out[e] = quant1(__ldg(I.x + e), p, bad);
    } else {
        const int planes = I.bits > 8 ? 2 : 1;
        const long long r0 = u * I.rpg;
        const long long total = I.rows * (long long)I.Cp;  // plane stride
        long long l1 = 0;
        if (I.C == I.Cp) {
            // unpadded rows: 8 codes per step, one 16-byte store per plane
            const long long n8 = (long long)I.rpg * I.Cp / 8, b8 = r0 * I.Cp / 8;
            const float4* x4 = reinterpret_cast<const float4*>(I.x);
            uint4* o = static_cast<uint4*>(I.out);
            for (long long i = threadIdx.x; i < n8; i += blockDim.x) {
                const float4 a = __ldg(x4 + 2 * (b8 + i)), b = __ldg(x4 + 2 * (b8 + i) + 1);
                const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int c0 = quant1(v[2 * e], p, bad), c1 = quant1(v[2 * e + 1], p, bad);
                    l1 += abs(c0) + abs(c1);
                    if (planes == 1) {
                        hi[e] = (uint32_t)__half_as_ushort(__int2half_rn(c0)) |
                                ((uint32_t)__half_as_ushort(__int2half_rn(c1)) << 16);
                    } else {
                        __half h0, l0, h1, l1h;
                        split_limbs(c0, h0, l0);
                        split_limbs(c1, h1, l1h);
                        hi[e] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                        lo[e] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1h) << 16);
                    }
                }
                o[b8 + i] = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                if (planes == 2) o[total / 8 + b8 + i] = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
        } else {
            __half* out = static_cast<__half*>(I.out);
            const long long n = (long long)I.rpg * I.Cp;
            for (long long i = threadIdx.x; i < n; i += blockDim.x) {
                const long long r = r0 + i / I.Cp;
                const int c = (int)(i % I.Cp);
                const int code = c < I.C ? quant1(__ldg(I.x + r * I.C + c), p, bad) : 0;
                l1 += abs(code);
                code_put(out, r * I.Cp + c, planes, total, code);
            }
        }
        if (I.l1 && planes == 1) {
            __shared__ long long red[8];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) l1 += __shfl_xor_sync(0xffffffffu, l1, o);
            if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = l1;
            __syncthreads();
            if (threadIdx.x == 0) {
                long long t = 0;
                for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
                atomicMax(reinterpret_cast<unsigned long long*>(I.l1), (unsigned long long)t);
            }
        }
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// ------------------------------------------------------------------------------------------
// Packed k-bit code storage: bit-plane words per group of 32 codes (see fxpq_pack_codes)
// ------------------------------------------------------------------------------------------
constexpr int PACK_G = 4;  // groups per warp and iteration (their code loads are issued together)

__global__ void pack_codes_kernel(const __half* __restrict__ codes, long long n, int k, int planes,
                                  uint32_t* __restrict__ words) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    const long long ng = (n + 31) / 32;
    const uint32_t mask = (1u << k) - 1;
    for (long long g0 = warp * PACK_G; g0 < ng; g0 += nwarps * PACK_G) {
        uint32_t f[PACK_G];
#pragma unroll
        for (int j = 0; j < PACK_G; ++j) {
            const long long e = (g0 + j) * 32 + lane;
            f[j] = e < n ? (uint32_t)code_get(codes, e, planes, n) & mask : 0u;
        }
#pragma unroll
        for (int j = 0; j < PACK_G; ++j) {
            if (g0 + j >= ng) break;
            uint32_t mine = 0;
#pragma unroll
            for (int b = 0; b < 16; ++b) {
                if (b >= k) break;
                const uint32_t w = __ballot_sync(0xffffffffu, (f[j] >> b) & 1u);
                if (lane == b) mine = w;
            }
            if (lane < k) words[(g0 + j) * k + lane] = mine;
        }
    }
}

__global__ void unpack_codes_kernel(const uint32_t* __restrict__ words, long long n, int k, int is_signed,
                                    int planes, __half* __restrict__ codes) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    const long long ng = (n + 31) / 32;
    for (long long g0 = warp * PACK_G; g0 < ng; g0 += nwarps * PACK_G) {
        uint32_t w[PACK_G];
#pragma unroll
        for (int j = 0; j < PACK_G; ++j) w[j] = (g0 + j < ng && lane < k) ? __ldg(words + (g0 + j) * k + lane) : 0u;
#pragma unroll
        for (int j = 0; j < PACK_G; ++j) {
            if (g0 + j >= ng) break;
            int field = 0;
#pragma unroll
            for (int b = 0; b < 16; ++b) {
                if (b >= k) break;
                field |= (int)((__shfl_sync(0xffffffffu, w[j], b) >> lane) & 1u) << b;
            }
            if (is_signed && (field >> (k - 1))) field -= 1 << k;  // sign extension of the k-bit field
            const long long e = (g0 + j) * 32 + lane;
            if (e < n) code_put(codes, e, planes, n, field);
        }
    }
}

// Packed weights for the contraction: one warp per 32 codes (kb, o, h), codes W[o][64 kb + 32 h + i]
// (zero past L and past K); lane i reads code i, lane b < k writes bit plane b to word
// (((kb * n_ct + o / 256) * k + b) * 256 + o % 256) * 2 + h.
__global__ void pack_weights_kernel(const __half* __restrict__ w, int K, int L, int K_pad, int k,
                                    uint32_t* __restrict__ words) {
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    const long long n_kb = (L + 63) / 64;
    const long long n_rec = n_kb * K_pad * 2;
    const long long n_ct = K_pad / 256;
    const uint32_t mask = (1u << k) - 1;
    for (long long r = warp; r < n_rec; r += nwarps) {
        const int h = (int)(r & 1);
        const long long ko = r >> 1;
        const int o = (int)(ko % K_pad);
        const long long kb = ko / K_pad;
        const long long col = kb * 64 + h * 32 + lane;
        const uint32_t f = (o < K && col < L) ? (uint32_t)__half2int_rn(w[(long long)o * L + col]) & mask : 0u;
        uint32_t mine = 0;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            if (b >= k) break;
            const uint32_t v = __ballot_sync(0xffffffffu, (f >> b) & 1u);
            if (lane == b) mine = v;
        }
        if (lane < k) words[(((kb * n_ct + o / 256) * k + lane) * 256 + o % 256) * 2 + h] = mine;
    }
}

}  // namespace


static QParams make_qparams(const fxpq_fmt& f) {
    QParams p;
    p.scale = ldexpf(1.0f, f.fl);
    p.lo = (float)qmin_of(f);
    p.hi = (float)qmax_of(f);
    p.binary = f.bits == 1 && f.is_signed == 1;
    p.status = status_ptr();
    return p;
}

static int grid_for(long long work, int threads) {
    long long b = (work + threads - 1) / threads;
    if (b < 1) b = 1;
    if (b > 152LL * 16) b = 152LL * 16;
    return (int)b;
}

}  // namespace fxpq

using namespace fxpq;

extern "C" fxpq_status fxpq_quantize(const float* d_x, int64_t n, fxpq_fmt f, int32_t dtype, void* d_codes,
                                     void* stream) {
    if (n < 0 || (n > 0 && (!d_x || !d_codes)) || !fmt_ok1(f, 32)) return FXPQ_ERR_INVALID_ARG;
    if (f.bits > 16 && dtype != FXPQ_DT_I32) return FXPQ_ERR_INVALID_ARG;
    switch (dtype) {
        case FXPQ_DT_I8: if (!(f.is_signed && f.bits <= 8)) return FXPQ_ERR_INVALID_ARG; break;
        case FXPQ_DT_U8: if (!(!f.is_signed && f.bits <= 8)) return FXPQ_ERR_INVALID_ARG; break;
        case FXPQ_DT_I16: if (!(f.is_signed && f.bits <= 16)) return FXPQ_ERR_INVALID_ARG; break;
        case FXPQ_DT_U16: if (!(!f.is_signed && f.bits <= 16)) return FXPQ_ERR_INVALID_ARG; break;
        case FXPQ_DT_I32: if (f.bits > 31) return FXPQ_ERR_INVALID_ARG; break;
        case FXPQ_DT_F16: break;
        default: return FXPQ_ERR_INVALID_ARG;
    }
    if (n == 0) return FXPQ_OK;
    cudaStream_t s = as_stream(stream);
    QParams p = make_qparams(f);
    const int T = 256;
    const bool al16 = aligned(d_x, 16) && aligned(d_codes, 16);
    if (dtype == FXPQ_DT_F16) {
        if (planes_of(f) == 1 && al16) {
            quantize_vec16_kernel<uint16_t, true><<<grid_for((n + 15) / 16, T), T, 0, s>>>(
                d_x, n, p, static_cast<uint16_t*>(d_codes));
            return after_launch("quantize_f16");
        }
        if (al16 && n % 8 == 0) {
            quantize_rows_vec8_kernel<<<grid_for(n / 8, T), T, 0, s>>>(reinterpret_cast<const float4*>(d_x), n / 8,
                                                                      planes_of(f), p, static_cast<uint4*>(d_codes));
            return after_launch("quantize_rows_vec8");
        }
        // unaligned: one code per row of one channel
        quantize_rows_f16_kernel<<<grid_for(n, T), T, 0, s>>>(d_x, n, 1, 1, planes_of(f), p,
                                                              static_cast<__half*>(d_codes));
        return after_launch("quantize_rows_f16");
    }
    if (al16) {
        const int g = grid_for((n + 15) / 16, T);
        switch (dtype) {
            case FXPQ_DT_I8:
            case FXPQ_DT_U8:
                quantize_vec16_kernel<uint8_t, false><<<g, T, 0, s>>>(d_x, n, p, static_cast<uint8_t*>(d_codes));
                break;
            case FXPQ_DT_I16:
            case FXPQ_DT_U16:
                quantize_vec16_kernel<uint16_t, false><<<g, T, 0, s>>>(d_x, n, p, static_cast<uint16_t*>(d_codes));
                break;
            default:
                quantize_vec16_kernel<uint32_t, false><<<g, T, 0, s>>>(d_x, n, p, static_cast<uint32_t*>(d_codes));
                break;
        }
        return after_launch("quantize_vec16");
    }
    bool vec = aligned(d_x, 16) && (n % 4 == 0);
#define FXPQ_Q_LAUNCH(TYPE)                                                                                       \
    if (vec)                                                                                                      \
        quantize_vec4_kernel<TYPE><<<grid_for(n / 4, T), T, 0, s>>>(reinterpret_cast<const float4*>(d_x), n / 4, \
                                                                    p, static_cast<TYPE*>(d_codes));              \
    else                                                                                                          \
        quantize_kernel<TYPE><<<grid_for(n, T), T, 0, s>>>(d_x, n, p, static_cast<TYPE*>(d_codes));
    switch (dtype) {
        case FXPQ_DT_I8: FXPQ_Q_LAUNCH(int8_t) break;
        case FXPQ_DT_U8: FXPQ_Q_LAUNCH(uint8_t) break;
        case FXPQ_DT_I16: FXPQ_Q_LAUNCH(int16_t) break;
        case FXPQ_DT_U16: FXPQ_Q_LAUNCH(uint16_t) break;
        default: FXPQ_Q_LAUNCH(int32_t) break;
    }
#undef FXPQ_Q_LAUNCH
    return after_launch("quantize");
}

extern "C" fxpq_status fxpq_quantize_rows(const float* d_x, int64_t rows, int32_t C, fxpq_fmt f, int32_t Cp,
                                          void* d_y, void* stream) {
    if (rows < 0 || C < 1 || Cp < C || (Cp % 8) || !fmt_ok(f)) return FXPQ_ERR_INVALID_ARG;
    if (rows == 0) return FXPQ_OK;
    if (!d_x || !d_y) return FXPQ_ERR_INVALID_ARG;
    QParams p = make_qparams(f);
    if (C == Cp && aligned(d_x, 16) && aligned(d_y, 16)) {
        const long long n8 = rows * (long long)C / 8;
        quantize_rows_vec8_kernel<<<grid_for(n8, 256), 256, 0, as_stream(stream)>>>(
            reinterpret_cast<const float4*>(d_x), n8, planes_of(f), p, static_cast<uint4*>(d_y));
        return after_launch("quantize_rows_vec8");
    }
    quantize_rows_f16_kernel<<<grid_for(rows * Cp, 256), 256, 0, as_stream(stream)>>>(
        d_x, rows, C, Cp, planes_of(f), p, static_cast<__half*>(d_y));
    return after_launch("quantize_rows_f16");
}

extern "C" fxpq_status fxpq_quantize_images(const float* d_x_nchw, int32_t N, int32_t C, int32_t H, int32_t W,
                                            fxpq_fmt f, int32_t c_pad, void* d_y, void* stream) {
    if (N < 0 || C < 1 || H < 1 || W < 1 || c_pad < C || (c_pad % 8) || !fmt_ok(f)) return FXPQ_ERR_INVALID_ARG;
    if (N == 0) return FXPQ_OK;
    if (!d_x_nchw || !d_y || !aligned(d_y, 16)) return FXPQ_ERR_INVALID_ARG;
    QParams p = make_qparams(f);
    long long npix = (long long)N * H * W;
    quantize_images_kernel<<<grid_for(npix, 256), 256, 0, as_stream(stream)>>>(d_x_nchw, N, C, H, W, c_pad,
                                                                                planes_of(f), p,
                                                                                static_cast<__half*>(d_y));
    return after_launch("quantize_images");
}

extern "C" fxpq_status fxpq_code_l1max(const void* d_codes, int64_t rows, int64_t L, int64_t* d_out, void* stream) {
    if (rows < 0 || L < 0 || (L % 8) || !d_out || !aligned(d_out, 8)) return FXPQ_ERR_INVALID_ARG;
    if (rows > 0 && L > 0 && (!d_codes || !aligned(d_codes, 16))) return FXPQ_ERR_INVALID_ARG;
    cudaStream_t s = as_stream(stream);
    if (cudaMemsetAsync(d_out, 0, sizeof(int64_t), s) != cudaSuccess) return FXPQ_ERR_CUDA;
    if (rows == 0 || L == 0) return FXPQ_OK;
    const int grid = rows < 4096 ? (int)rows : 4096;
    code_l1max_kernel<<<grid, 256, 0, s>>>(static_cast<const uint4*>(d_codes), rows, L / 8,
                                           reinterpret_cast<unsigned long long*>(d_out));
    return after_launch("code_l1max");
}

extern "C" fxpq_status fxpq_quantize_batch(const fxpq_quantize_item* h_items, int32_t n_items, void* stream) {
    if (n_items < 0 || (n_items > 0 && !h_items)) return FXPQ_ERR_INVALID_ARG;
    for (int i = 0; i < n_items; ++i) {
        const fxpq_quantize_item& it = h_items[i];
        if (it.bits < 2 || it.bits > 16 || it.rows < 0 || !it.d_fl || !it.d_stats) return FXPQ_ERR_INVALID_ARG;
        if (it.rows > 0 && (!it.d_x || !it.d_out)) return FXPQ_ERR_INVALID_ARG;
        if (it.kind == FXPQ_QB_FLAT_I32) {
            if (it.d_l1) return FXPQ_ERR_INVALID_ARG;
        } else if (it.kind == FXPQ_QB_ROWS_F16) {
            if (it.C < 1 || it.Cp < it.C || (it.Cp % 8) || it.rows_per_group < 1 || it.rows % it.rows_per_group)
                return FXPQ_ERR_INVALID_ARG;
            if (it.C == it.Cp && (!aligned(it.d_x, 16) || !aligned(it.d_out, 16))) return FXPQ_ERR_INVALID_ARG;
            if (it.d_l1 && (it.bits > 8 || !aligned(it.d_l1, 8))) return FXPQ_ERR_INVALID_ARG;
        } else {
            return FXPQ_ERR_INVALID_ARG;
        }
    }
    cudaStream_t s = as_stream(stream);
    for (int i0 = 0; i0 < n_items; i0 += QB_MAX) {
        const int m = n_items - i0 < QB_MAX ? n_items - i0 : QB_MAX;
        QbBatch B;
        B.n = m;
        B.status = status_ptr();
        long long units = 0;
        for (int i = 0; i < m; ++i) {
            const fxpq_quantize_item& it = h_items[i0 + i];
            QbItem& q = B.it[i];
            q.x = it.d_x;
            q.out = it.d_out;
            q.l1 = reinterpret_cast<long long*>(it.d_l1);
            q.fl = it.d_fl;
            q.st = it.d_stats;
            q.rows = it.rows;
            q.C = it.C;
            q.Cp = it.Cp;
            q.rpg = it.rows_per_group;
            q.bits = it.bits;
            q.kind = it.kind;
            B.unit0[i] = (int)units;
            units += it.kind == FXPQ_QB_FLAT_I32 ? (it.rows + QB_FLAT_UNIT - 1) / QB_FLAT_UNIT
                                                 : it.rows / it.rows_per_group;
            if (units > (1LL << 30)) return FXPQ_ERR_INVALID_ARG;
        }
        B.unit0[m] = (int)units;
        if (units == 0) continue;
        quantize_batch_kernel<<<(unsigned)units, 256, 0, s>>>(B);
        const fxpq_status st = after_launch("quantize_batch");
        if (st != FXPQ_OK) return st;
    }
    return FXPQ_OK;
}

extern "C" fxpq_status fxpq_pack_codes(const void* d_codes, int64_t n, fxpq_fmt fmt, uint32_t* d_words,
                                       void* stream) {
    if (n < 0 || !fmt_ok1(fmt) || (n > 0 && (!d_codes || !d_words)) || !aligned(d_words, 4))
        return FXPQ_ERR_INVALID_ARG;
    if (n == 0) return FXPQ_OK;
    const long long ng = (n + 31) / 32;
    const int T = 256;
    pack_codes_kernel<<<grid_for((ng + PACK_G - 1) / PACK_G * 32, T), T, 0, as_stream(stream)>>>(
        static_cast<const __half*>(d_codes), n, fmt.bits, planes_of(fmt), d_words);
    return after_launch("pack_codes");
}

extern "C" size_t fxpq_packed_weights_bytes(fxpq_fmt fmt_w, int32_t K, int32_t L) {
    if (fmt_w.bits < 1 || fmt_w.bits > 8 || K < 1 || L < 1) return 0;
    const size_t n_kb = ((size_t)L + 63) / 64, K_pad = ((size_t)K + 255) / 256 * 256;
    return n_kb * K_pad * 2 * (size_t)fmt_w.bits * 4;
}

extern "C" fxpq_status fxpq_pack_weights(const void* d_w, fxpq_fmt fmt_w, int32_t K, int32_t L, void* d_packed,
                                         void* stream) {
    if (!fmt_ok1(fmt_w) || fmt_w.bits > 8 || K < 1 || L < 1 || !d_w || !d_packed || !aligned(d_packed, 16) ||
        !aligned(d_w, 2))
        return FXPQ_ERR_INVALID_ARG;
    const int K_pad = (K + 255) / 256 * 256;
    const long long n_rec = ((long long)L + 63) / 64 * K_pad * 2;
    const int T = 256;
    pack_weights_kernel<<<grid_for(n_rec * 32, T), T, 0, as_stream(stream)>>>(
        static_cast<const __half*>(d_w), K, L, K_pad, fmt_w.bits, static_cast<uint32_t*>(d_packed));
    return after_launch("pack_weights");
}

extern "C" fxpq_status fxpq_unpack_codes(const uint32_t* d_words, int64_t n, fxpq_fmt fmt, void* d_codes,
                                         void* stream) {
    if (n < 0 || !fmt_ok1(fmt) || (n > 0 && (!d_codes || !d_words)) || !aligned(d_words, 4))
        return FXPQ_ERR_INVALID_ARG;
    if (n == 0) return FXPQ_OK;
    const long long ng = (n + 31) / 32;
    const int T = 256;
    unpack_codes_kernel<<<grid_for((ng + PACK_G - 1) / PACK_G * 32, T), T, 0, as_stream(stream)>>>(
        d_words, n, fmt.bits, fmt.is_signed, planes_of(fmt), static_cast<__half*>(d_codes));
    return after_launch("unpack_codes");
}
