// fxpq_quant.cu -- quantizer Q (Sec. IV-B) and the batched FL search (Sec. IV-C, Eq. DSB_QE).
//
// FL search design (one HBM pass, exact result).
//   For fp32 x = (-1)^sg * M * 2^(E-23) (M the 24-bit significand) and a candidate (k, FL):
//   y = |x| * 2^FL has integer exponent q = E + FL.  With T the clip level in y units
//   (S=1: 2^(k-1)-1 for x >= 0, 2^(k-1) for x < 0; S=0: 2^k - 1 for x >= 0, 0 for x < 0), the
//   per-element error is (|x| - T 2^-FL)^2 if |y| >= T (saturated) and r^2 otherwise, r the
//   round-half-even remainder.  For T = 2^t - 1 the test |y| >= T is "q >= t, or q = t-1 and the
//   significand's leading-ones count LO >= t"; for T = 2^t it is q >= t.  Hence
//     * saturated terms are polynomials in T whose coefficients are the moments
//       (count, sum M, sum M^2) of elements grouped by (sign, E [, LO class]);
//     * unsaturated terms need sum r^2 grouped by (sign, j = q, FL), split by whether
//       LO >= j+1 (the boundary class), for j in [-1, 15]; q <= -2 rounds to 0 (error x^2,
//       a moment) and q >= 23 is exact.
//   All bins are integers (r^2 in units of 2^(2(E-23))), so each candidate's sum is exact.  The
//   finalize kernel adds the terms of one candidate in a 768-bit fixed-point accumulator and
//   rounds once to nearest-even double -- the same value as the exact definition.
#include <math.h>

#include <mutex>

#include "fxpq_common.cuh"

namespace fxpq {
namespace {

// ------------------------------------------------------------------------------------------
// Quantize kernels
// ------------------------------------------------------------------------------------------
struct QParams {
    float scale;  // 2^fl (exact power of two; fl in [-32, 40])
    float lo, hi; // Qmin, Qmax as floats (exact, |.| <= 2^16)
    int* status;
};

__device__ __forceinline__ int quant1(float x, const QParams& p, bool& bad) {
    if (!isfinite(x)) {
        bad = true;
        return 0;
    }
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

// NCHW fp32 -> NHWC fp16 codes, channels padded to Cp; one thread per pixel
__global__ void quantize_images_kernel(const float* __restrict__ x, int N, int C, int H, int W, int Cp, int planes,
                                       QParams p, __half* __restrict__ out) {
    bool bad = false;
    long long npix = (long long)N * H * W;
    long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < npix; i += stride) {
        long long n = i / ((long long)H * W);
        long long hw = i - n * H * W;
        for (int c = 0; c < Cp; ++c) {
            int code = c < C ? quant1(x[(n * C + c) * (long long)H * W + hw], p, bad) : 0;
            code_put(out, i * Cp + c, planes, npix * Cp, code);
        }
    }
    if (bad) latch_status(p.status, FXPQ_ERR_NONFINITE);
}

// ------------------------------------------------------------------------------------------
// FL search
// ------------------------------------------------------------------------------------------
constexpr int NE = 254;    // E in [-126, 127]
constexpr int EOFF = 126;  // bin index = E + EOFF
constexpr int WE = 48;     // width of the E window that keeps leading-ones classes
constexpr int NLO = 17;    // leading-ones classes 0..15 and >= 16
constexpr int NJ = 17;     // j in [-1, 15]
constexpr int MAXFL = 32;  // candidates per k
constexpr int MAXK = 15;   // k in [2, 16]
constexpr int FS_THREADS = 256;

typedef unsigned long long u64;

struct FsSmem {
    unsigned pn[2][NE];
    u64 ps1[2][NE];
    u64 ps2[2][NE];
    unsigned wn[WE][NLO];
    u64 ws1[WE][NLO];
    u64 ws2[WE][NLO];
    u64 r0[2][NJ][MAXFL];
    u64 r1[NJ][MAXFL];
    unsigned mn, mx, nonfinite, pad;
};

// 128-bit quantities are stored as {lo, hi}
struct FsGlobal {
    u64 pn[2][NE];
    u64 ps1[2][NE][2];
    u64 ps2[2][NE][2];
    u64 wn[WE][NLO];
    u64 ws1[WE][NLO][2];
    u64 ws2[WE][NLO][2];
    u64 r0[2][NJ][MAXFL][2];
    u64 r1[NJ][MAXFL][2];
    unsigned mn, mx, nonfinite, pad;
    // derived by the totals kernel
    u64 tn[2][NE];           // per (sign, E): count
    u64 ts1[2][NE][2];       // sum M
    u64 ts2[2][NE][2];       // sum M^2
    u64 wsn[WE][NLO];        // suffix over LO classes (positives in the window): count with LO >= l
    u64 wss1[WE][NLO][2];
    u64 wss2[WE][NLO][2];
    double cells[2][MAXK][MAXFL];
    double stat_sum, stat_sumsq;
    u64 n;
};

struct FsParams {
    const float* x;
    long long n;
    int chunk;
    int fl_lo, nfl;
    int ew0;       // first E of the leading-ones window
    int jmax_pos;  // largest j whose r^2 is needed for x >= 0 (-2: none)
    int jmax_neg;  // same for x < 0
    FsGlobal* g;
};

__device__ __forceinline__ void atomic_add_u128(u64* p, u64 v) {
    if (v == 0) return;
    u64 old = atomicAdd(p, v);
    if (old + v < old) atomicAdd(p + 1, 1ull);
}

__device__ __forceinline__ unsigned order_key(float x) {
    unsigned u = __float_as_uint(x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float order_key_inv(unsigned k) {
    unsigned u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
    return __uint_as_float(u);
}

// All 32 lanes call this together (warp-collective), ok = this lane holds an element.
__device__ __forceinline__ void fs_element(FsSmem& sm, const FsParams& P, float x, bool ok, unsigned& tmn,
                                           unsigned& tmx, bool& tnf) {
    const unsigned u = __float_as_uint(x);
    const unsigned eb = (u >> 23) & 0xFFu;
    if (ok && eb == 0xFFu) tnf = true;
    ok = ok && (eb != 0xFFu);
    if (ok) {
        unsigned key = order_key(x);
        tmn = min(tmn, key);
        tmx = max(tmx, key);
    }
    const unsigned sgn = u >> 31;
    const unsigned frac = u & 0x7FFFFFu;
    const int E = eb ? (int)eb - 127 : -126;
    const unsigned M = eb ? (frac | 0x800000u) : frac;
    const bool live = ok && (M != 0u);
    const int LO = __clz(~(M << 8));  // leading ones of the 24-bit significand
    const unsigned lane = threadIdx.x & 31u;

    // ---- moments: (sign, E) bins, leading-ones classes for x >= 0 inside the window
    const int wi = E - P.ew0;
    const bool inwin = (sgn == 0u) && wi >= 0 && wi < WE;
    const int loc = min(LO, NLO - 1);
    const unsigned mkey =
        !live ? 0xFFFFFFFFu
              : (inwin ? (unsigned)(wi * NLO + loc) : (unsigned)(WE * NLO + sgn * NE + (unsigned)(E + EOFF)));
    const unsigned grp = __match_any_sync(0xFFFFFFFFu, mkey);
    const u64 m2 = (u64)M * M;  // < 2^48
    const unsigned s1 = __reduce_add_sync(grp, live ? M : 0u);
    const unsigned s2h = __reduce_add_sync(grp, live ? (unsigned)(m2 >> 24) : 0u);
    const unsigned s2l = __reduce_add_sync(grp, live ? (unsigned)(m2 & 0xFFFFFFu) : 0u);
    if (live && lane == (unsigned)(__ffs(grp) - 1)) {
        const unsigned cnt = __popc(grp);
        const u64 S2 = ((u64)s2h << 24) + (u64)s2l;
        if (inwin) {
            atomicAdd(&sm.wn[wi][loc], cnt);
            atomicAdd(&sm.ws1[wi][loc], (u64)s1);
            atomicAdd(&sm.ws2[wi][loc], S2);
        } else {
            atomicAdd(&sm.pn[sgn][E + EOFF], cnt);
            atomicAdd(&sm.ps1[sgn][E + EOFF], (u64)s1);
            atomicAdd(&sm.ps2[sgn][E + EOFF], S2);
        }
    }

    // ---- remainders: r^2 of round-half-even at j = q = E + FL, j in [-1, 15]
    const unsigned rkey = live ? (sgn * 256u + (unsigned)(E + EOFF)) : 0xFFFFFFFFu;
    const unsigned rgrp = __match_any_sync(0xFFFFFFFFu, rkey);
    const bool rlead = live && lane == (unsigned)(__ffs(rgrp) - 1);
    const int jmax = sgn ? P.jmax_neg : P.jmax_pos;
#pragma unroll
    for (int jj = 0; jj < NJ; ++jj) {
        const int j = jj - 1;
        const int p = 23 - j;  // fractional bits of y in units of M: 24 .. 8
        const int fi = j - E - P.fl_lo;
        const bool valid = live && j <= jmax && fi >= 0 && fi < P.nfl;
        const unsigned t = M & ((1u << p) - 1u);
        const unsigned odd = (M >> p) & 1u;
        const bool up = (t + odd) > (1u << (p - 1));
        const unsigned r = up ? (1u << p) - t : t;
        const u64 r2 = (u64)r * r;  // <= 2^46
        const bool beta = (sgn == 0u) && (j >= 0) && (LO >= j + 1);
        const u64 v0 = (valid && !beta) ? r2 : 0ull;
        const unsigned h = __reduce_add_sync(rgrp, (unsigned)(v0 >> 23));
        const unsigned l = __reduce_add_sync(rgrp, (unsigned)(v0 & 0x7FFFFFu));
        if (rlead && valid) {
            const u64 s = ((u64)h << 23) + (u64)l;
            if (s) atomicAdd(&sm.r0[sgn][jj][fi], s);
        }
        if (valid && beta && r2) atomicAdd(&sm.r1[jj][fi], r2);
    }
}

template <bool VEC>
__global__ void __launch_bounds__(FS_THREADS) fl_search_bins_kernel(FsParams P) {
    __shared__ FsSmem sm;
    for (int i = threadIdx.x; i < (int)(sizeof(FsSmem) / 4); i += FS_THREADS) reinterpret_cast<unsigned*>(&sm)[i] = 0u;
    __syncthreads();
    if (threadIdx.x == 0) sm.mn = 0xFFFFFFFFu;
    __syncthreads();

    const long long start = (long long)blockIdx.x * P.chunk;
    const long long end = min(start + (long long)P.chunk, P.n);
    unsigned tmn = 0xFFFFFFFFu, tmx = 0u;
    bool tnf = false;
    for (long long base = start; base < end; base += 4 * FS_THREADS) {
        const long long i0 = base + 4 * (long long)threadIdx.x;
        float v[4];
        bool ok[4];
        if (VEC && i0 + 3 < end) {
            float4 f = __ldg(reinterpret_cast<const float4*>(P.x + i0));
            v[0] = f.x, v[1] = f.y, v[2] = f.z, v[3] = f.w;
            ok[0] = ok[1] = ok[2] = ok[3] = true;
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                ok[k] = i0 + k < end;
                v[k] = ok[k] ? P.x[i0 + k] : 0.0f;
            }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) fs_element(sm, P, v[k], ok[k], tmn, tmx, tnf);
    }
    atomicMin(&sm.mn, tmn);
    atomicMax(&sm.mx, tmx);
    if (tnf) sm.nonfinite = 1u;
    __syncthreads();

    // flush the block's bins into the exact 128-bit global bins
    FsGlobal* g = P.g;
    for (int i = threadIdx.x; i < 2 * NE; i += FS_THREADS) {
        int s = i / NE, e = i % NE;
        if (sm.pn[s][e]) {
            atomicAdd(&g->pn[s][e], (u64)sm.pn[s][e]);
            atomic_add_u128(g->ps1[s][e], sm.ps1[s][e]);
            atomic_add_u128(g->ps2[s][e], sm.ps2[s][e]);
        }
    }
    for (int i = threadIdx.x; i < WE * NLO; i += FS_THREADS) {
        int w = i / NLO, l = i % NLO;
        if (sm.wn[w][l]) {
            atomicAdd(&g->wn[w][l], (u64)sm.wn[w][l]);
            atomic_add_u128(g->ws1[w][l], sm.ws1[w][l]);
            atomic_add_u128(g->ws2[w][l], sm.ws2[w][l]);
        }
    }
    for (int i = threadIdx.x; i < 2 * NJ * MAXFL; i += FS_THREADS) {
        int s = i / (NJ * MAXFL), r = i % (NJ * MAXFL);
        atomic_add_u128(g->r0[s][r / MAXFL][r % MAXFL], sm.r0[s][r / MAXFL][r % MAXFL]);
    }
    for (int i = threadIdx.x; i < NJ * MAXFL; i += FS_THREADS)
        atomic_add_u128(g->r1[i / MAXFL][i % MAXFL], sm.r1[i / MAXFL][i % MAXFL]);
    if (threadIdx.x == 0) {
        atomicMin(&g->mn, sm.mn);
        atomicMax(&g->mx, sm.mx);
        if (sm.nonfinite) atomicOr(&g->nonfinite, 1u);
    }
}

// 128-bit helpers for the (small) derived-bin and finalize kernels
struct U128 {
    u64 lo, hi;
};
__device__ __forceinline__ U128 ld128(const u64* p) { return U128{p[0], p[1]}; }
__device__ __forceinline__ U128 add128(U128 a, U128 b) {
    U128 r;
    r.lo = a.lo + b.lo;
    r.hi = a.hi + b.hi + (r.lo < a.lo ? 1ull : 0ull);
    return r;
}
__device__ __forceinline__ void st128(u64* p, U128 v) {
    p[0] = v.lo;
    p[1] = v.hi;
}
// (a * m) for a 128-bit a and 64-bit m: result fits 128 bits by the callers' bounds
__device__ __forceinline__ U128 mul128_64(U128 a, u64 m) {
    U128 r;
    r.lo = a.lo * m;
    r.hi = __umul64hi(a.lo, m) + a.hi * m;
    return r;
}

// per (sign, E) totals and per-window leading-ones suffix sums
__global__ void fl_search_totals_kernel(FsParams P) {
    FsGlobal* g = P.g;
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < 2 * NE) {
        int s = i / NE, e = i % NE;
        u64 n = g->pn[s][e];
        U128 s1 = ld128(g->ps1[s][e]), s2 = ld128(g->ps2[s][e]);
        int wi = (e - EOFF) - P.ew0;
        if (s == 0 && wi >= 0 && wi < WE) {
            for (int l = 0; l < NLO; ++l) {
                n += g->wn[wi][l];
                s1 = add128(s1, ld128(g->ws1[wi][l]));
                s2 = add128(s2, ld128(g->ws2[wi][l]));
            }
        }
        g->tn[s][e] = n;
        st128(g->ts1[s][e], s1);
        st128(g->ts2[s][e], s2);
    } else if (i < 2 * NE + WE) {
        int wi = i - 2 * NE;
        u64 n = 0;
        U128 s1{0, 0}, s2{0, 0};
        for (int l = NLO - 1; l >= 0; --l) {
            n += g->wn[wi][l];
            s1 = add128(s1, ld128(g->ws1[wi][l]));
            s2 = add128(s2, ld128(g->ws2[wi][l]));
            g->wsn[wi][l] = n;
            st128(g->wss1[wi][l], s1);
            st128(g->wss2[wi][l], s2);
        }
    }
}

// ---- exact fixed-point accumulator: 12 x 64-bit two's complement words, word i weighs 2^(64 i - 320)
constexpr int BW = 12;
constexpr int BBASE = -320;

struct Big {
    u64 w[BW];
};

__device__ void big_zero(Big& a) {
#pragma unroll
    for (int i = 0; i < BW; ++i) a.w[i] = 0;
}

// a += (neg ? -1 : 1) * v * 2^e for a 128-bit magnitude v
__device__ void big_add(Big& a, U128 v, int e, bool neg) {
    if ((v.lo | v.hi) == 0) return;
    int pos = e - BBASE;
    int wi = pos >> 6, b = pos & 63;
    u64 s[3];
    s[0] = v.lo << b;
    s[1] = b ? ((v.hi << b) | (v.lo >> (64 - b))) : v.hi;
    s[2] = b ? (v.hi >> (64 - b)) : 0ull;
    if (!neg) {
        u64 carry = 0;
        for (int i = wi; i < BW; ++i) {
            u64 add = (i - wi < 3) ? s[i - wi] : 0ull;
            u64 t = a.w[i] + add;
            u64 c1 = t < add;
            u64 t2 = t + carry;
            u64 c2 = t2 < t;
            a.w[i] = t2;
            carry = c1 | c2;
            if (i - wi >= 2 && carry == 0) break;
        }
    } else {
        u64 borrow = 0;
        for (int i = wi; i < BW; ++i) {
            u64 sub = (i - wi < 3) ? s[i - wi] : 0ull;
            u64 t = a.w[i] - sub;
            u64 b1 = a.w[i] < sub;
            u64 t2 = t - borrow;
            u64 b2 = t < borrow;
            a.w[i] = t2;
            borrow = b1 | b2;
            if (i - wi >= 2 && borrow == 0) break;
        }
    }
}

// bits [pos, pos+64) of a (pos may be negative: zero below bit 0)
__device__ u64 big_bits64(const Big& a, int pos) {
    u64 r;
    // assemble from up to two words
    int wi = pos >= 0 ? (pos >> 6) : -((-pos + 63) >> 6);
    int b = pos - wi * 64;  // 0..63
    u64 lo = (wi >= 0 && wi < BW) ? a.w[wi] : 0ull;
    u64 hi = (wi + 1 >= 0 && wi + 1 < BW) ? a.w[wi + 1] : 0ull;
    r = b ? ((lo >> b) | (hi << (64 - b))) : lo;
    return r;
}

__device__ bool big_any_below(const Big& a, int pos) {  // any set bit strictly below pos
    if (pos <= 0) return false;
    int wi = pos >> 6, b = pos & 63;
    for (int i = 0; i < wi && i < BW; ++i)
        if (a.w[i]) return true;
    if (wi < BW && b && (a.w[wi] & ((1ull << b) - 1ull))) return true;
    return false;
}

// round the (non-negative) accumulator to nearest-even double; a negative value returns -1
__device__ double big_to_double(const Big& a) {
    if ((long long)a.w[BW - 1] < 0) return -1.0;
    int h = -1;
    for (int i = BW - 1; i >= 0; --i)
        if (a.w[i]) {
            h = i;
            break;
        }
    if (h < 0) return 0.0;
    int top = 64 * h + 63 - __clzll(a.w[h]);  // index of the highest set bit
    u64 win = big_bits64(a, top - 63);          // bits [top-63, top]
    u64 mant = win >> 11;                       // 53 bits
    bool rb = (win >> 10) & 1ull;
    bool sticky = (win & 0x3FFull) != 0ull || big_any_below(a, top - 63);
    if (rb && (sticky || (mant & 1ull))) mant += 1ull;
    return ldexp((double)mant, top - 52 + BBASE);
}

struct FsFinal {
    int S_lo, S_hi;  // range of sign strategies to score
    int k_lo, nk;
    int fl_lo, nfl;
    int ew0;
};

// sat(|x| >= T 2^-fl) contribution of a set with moments (n, s1, s2) in units of E:
// s2 2^(2(E-23)) - 2 T s1 2^(E-23-fl) + T^2 n 2^(-2 fl)
__device__ void add_sat(Big& acc, u64 n, U128 s1, U128 s2, int E, int fl, u64 T) {
    big_add(acc, s2, 2 * (E - 23), false);
    if (T) {
        big_add(acc, mul128_64(s1, 2ull * T), E - 23 - fl, true);
        big_add(acc, mul128_64(U128{n, 0ull}, T * T), -2 * fl, false);
    }
}

__global__ void fl_search_cells_kernel(FsParams P, FsFinal F) {
    FsGlobal* g = P.g;
    const int ncell = (F.S_hi - F.S_lo + 1) * F.nk * F.nfl;
    int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx == ncell || idx == ncell + 1) {
        // stats: exact sum and sum of squares
        Big acc;
        big_zero(acc);
        for (int e = 0; e < NE; ++e) {
            int E = e - EOFF;
            if (idx == ncell) {
                big_add(acc, ld128(g->ts1[0][e]), E - 23, false);
                big_add(acc, ld128(g->ts1[1][e]), E - 23, true);
            } else {
                big_add(acc, ld128(g->ts2[0][e]), 2 * (E - 23), false);
                big_add(acc, ld128(g->ts2[1][e]), 2 * (E - 23), false);
            }
        }
        if (idx == ncell) {
            // the sum may be negative: round |sum| and restore the sign
            bool neg = (long long)acc.w[BW - 1] < 0;
            if (neg) {
                u64 c = 1;
                for (int i = 0; i < BW; ++i) {
                    u64 t = ~acc.w[i] + c;
                    c = (c && t == 0) ? 1ull : 0ull;
                    acc.w[i] = t;
                }
            }
            double v = big_to_double(acc);
            g->stat_sum = neg ? -v : v;
        } else {
            g->stat_sumsq = big_to_double(acc);
        }
        return;
    }
    if (idx >= ncell) return;
    const int S = F.S_lo + idx / (F.nk * F.nfl);
    const int rem = idx % (F.nk * F.nfl);
    const int k = F.k_lo + rem / F.nfl;
    const int fi = rem % F.nfl;
    const int fl = F.fl_lo + fi;

    Big acc;
    big_zero(acc);
    for (int sg = 0; sg < 2; ++sg) {
        // clip level T = 2^t - 1 (x >= 0, boundary by leading ones) or 2^t (x < 0, S = 1); S = 0, x < 0: T = 0
        const bool minus_one = (sg == 0);
        const int t = (sg == 0) ? (S ? k - 1 : k) : (k - 1);
        const u64 T = minus_one ? ((1ull << t) - 1ull) : (1ull << t);
        for (int e = 0; e < NE; ++e) {
            const u64 n = g->tn[sg][e];
            if (n == 0) continue;
            const int E = e - EOFF;
            const U128 s1 = ld128(g->ts1[sg][e]), s2 = ld128(g->ts2[sg][e]);
            if (sg == 1 && S == 0) {  // clipped to 0: error x^2
                big_add(acc, s2, 2 * (E - 23), false);
                continue;
            }
            const int q = E + fl;
            if (q >= t) {  // all saturated
                add_sat(acc, n, s1, s2, E, fl, T);
            } else if (minus_one && q == t - 1) {  // boundary: LO >= t saturates, the rest rounds
                const int wi = E - F.ew0;
                const int l = t < NLO ? t : NLO - 1;
                add_sat(acc, g->wsn[wi][l], ld128(g->wss1[wi][l]), ld128(g->wss2[wi][l]), E, fl, T);
                big_add(acc, ld128(g->r0[sg][q + 1][fi]), 2 * (E - 23), false);
            } else if (q <= -2) {  // |y| < 1/2: rounds to 0
                big_add(acc, s2, 2 * (E - 23), false);
            } else {  // -1 <= q <= t-2 (or t-1 for x < 0): unsaturated, every leading-ones class
                big_add(acc, ld128(g->r0[sg][q + 1][fi]), 2 * (E - 23), false);
                if (sg == 0) big_add(acc, ld128(g->r1[q + 1][fi]), 2 * (E - 23), false);
            }
        }
    }
    g->cells[S][k - 2][fi] = big_to_double(acc);
}

__global__ void fl_search_select_kernel(FsParams P, FsFinal F, int is_signed, double* err, int* best,
                                        fxpq_stats* stats, int* status) {
    FsGlobal* g = P.g;
    const float mn = g->mn == 0xFFFFFFFFu ? 0.0f : order_key_inv(g->mn);
    const float mx = g->mx == 0u ? 0.0f : order_key_inv(g->mx);
    const int S = is_signed >= 0 ? is_signed : (mn < 0.0f ? 1 : 0);
    int i = threadIdx.x;
    if (i < F.nk) {
        const int k = F.k_lo + i;
        double bv = 0.0;
        int bf = F.fl_lo;
        for (int fi = 0; fi < F.nfl; ++fi) {
            double v = g->cells[S][k - 2][fi];
            err[(long long)i * F.nfl + fi] = v;
            if (fi == 0 || v < bv) {
                bv = v;
                bf = F.fl_lo + fi;
            }
        }
        best[i] = bf;
    }
    if (i == 0) {
        if (g->nonfinite) latch_status(status, FXPQ_ERR_NONFINITE);
        if (stats) {
            stats->min = mn;
            stats->max = mx;
            stats->is_signed = S;
            stats->nonfinite = g->nonfinite ? 1 : 0;
            stats->sum = g->stat_sum;
            stats->sumsq = g->stat_sumsq;
            stats->n = P.n;
        }
    }
}

}  // namespace

static QParams make_qparams(const fxpq_fmt& f) {
    QParams p;
    p.scale = ldexpf(1.0f, f.fl);
    p.lo = (float)qmin_of(f);
    p.hi = (float)qmax_of(f);
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
    if (n < 0 || (n > 0 && (!d_x || !d_codes)) || !fmt_ok(f, 32)) return FXPQ_ERR_INVALID_ARG;
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
    if (dtype == FXPQ_DT_F16) {
        quantize_rows_f16_kernel<<<grid_for(n, T), T, 0, s>>>(d_x, 1, (int)n, (int)n, planes_of(f), p,
                                                              static_cast<__half*>(d_codes));
        return after_launch("quantize_rows_f16");
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
    quantize_rows_f16_kernel<<<grid_for(rows * Cp, 256), 256, 0, as_stream(stream)>>>(
        d_x, rows, C, Cp, planes_of(f), p, static_cast<__half*>(d_y));
    return after_launch("quantize_rows_f16");
}

extern "C" fxpq_status fxpq_quantize_images(const float* d_x_nchw, int32_t N, int32_t C, int32_t H, int32_t W,
                                            fxpq_fmt f, int32_t c_pad, void* d_y, void* stream) {
    if (N < 0 || C < 1 || H < 1 || W < 1 || c_pad < C || (c_pad % 8) || !fmt_ok(f)) return FXPQ_ERR_INVALID_ARG;
    if (N == 0) return FXPQ_OK;
    if (!d_x_nchw || !d_y) return FXPQ_ERR_INVALID_ARG;
    QParams p = make_qparams(f);
    long long npix = (long long)N * H * W;
    quantize_images_kernel<<<grid_for(npix, 256), 256, 0, as_stream(stream)>>>(d_x_nchw, N, C, H, W, c_pad,
                                                                                planes_of(f), p,
                                                                                static_cast<__half*>(d_y));
    return after_launch("quantize_images");
}

extern "C" size_t fxpq_fl_search_workspace(int64_t n) {
    (void)n;
    return (sizeof(FsGlobal) + 255) / 256 * 256;
}

extern "C" fxpq_status fxpq_fl_search(const float* d_x, int64_t n, int32_t is_signed, int32_t k_lo, int32_t k_hi,
                                      int32_t fl_lo, int32_t fl_hi, double* d_err, int32_t* d_best,
                                      fxpq_stats* d_stats, void* d_ws, size_t ws_bytes, void* stream) {
    if (n < 0 || n > (int64_t(1) << 31)) return FXPQ_ERR_INVALID_ARG;
    if (is_signed < -1 || is_signed > 1) return FXPQ_ERR_INVALID_ARG;
    if (k_lo < 2 || k_hi > 16 || k_lo > k_hi) return FXPQ_ERR_INVALID_ARG;
    if (fl_lo < -32 || fl_hi > 40 || fl_lo > fl_hi || fl_hi - fl_lo + 1 > MAXFL) return FXPQ_ERR_INVALID_ARG;
    if (!d_err || !d_best || (n > 0 && !d_x)) return FXPQ_ERR_INVALID_ARG;
    if (!d_ws || ws_bytes < fxpq_fl_search_workspace(n) || !aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    cudaStream_t s = as_stream(stream);
    FsGlobal* g = static_cast<FsGlobal*>(d_ws);
    if (cudaMemsetAsync(g, 0, sizeof(FsGlobal), s) != cudaSuccess) return FXPQ_ERR_CUDA;
    if (cudaMemsetAsync(&g->mn, 0xFF, sizeof(unsigned), s) != cudaSuccess) return FXPQ_ERR_CUDA;

    FsParams P;
    P.x = d_x;
    P.n = n;
    long long per = (n + 152LL * 4 - 1) / (152LL * 4);
    long long chunk = (per + 1023) / 1024 * 1024;
    if (chunk < 1024) chunk = 1024;
    if (chunk > 65536) chunk = 65536;  // keeps every per-block 64-bit bin below 2^64
    P.chunk = (int)chunk;
    P.fl_lo = fl_lo;
    P.nfl = fl_hi - fl_lo + 1;
    P.ew0 = k_lo - 2 - fl_hi;  // boundary exponents E = t - 1 - fl, t in [k_lo - 1, k_hi]
    if (k_hi - 1 - fl_lo - P.ew0 + 1 > WE) return FXPQ_ERR_INVALID_ARG;
    const int S_lo = is_signed < 0 ? 0 : is_signed, S_hi = is_signed < 0 ? 1 : is_signed;
    P.jmax_pos = (S_lo == 0) ? k_hi - 1 : k_hi - 2;
    P.jmax_neg = (S_hi == 1) ? k_hi - 2 : -2;
    P.g = g;
    if (n > 0) {
        int grid = (int)((n + chunk - 1) / chunk);
        bool vec = aligned(d_x, 16);
        if (vec)
            fl_search_bins_kernel<true><<<grid, FS_THREADS, 0, s>>>(P);
        else
            fl_search_bins_kernel<false><<<grid, FS_THREADS, 0, s>>>(P);
        fxpq_status st = after_launch("fl_search_bins");
        if (st != FXPQ_OK) return st;
    }
    fl_search_totals_kernel<<<(2 * NE + WE + 127) / 128, 128, 0, s>>>(P);
    fxpq_status st = after_launch("fl_search_totals");
    if (st != FXPQ_OK) return st;
    FsFinal F;
    F.S_lo = S_lo;
    F.S_hi = S_hi;
    F.k_lo = k_lo;
    F.nk = k_hi - k_lo + 1;
    F.fl_lo = fl_lo;
    F.nfl = P.nfl;
    F.ew0 = P.ew0;
    int ncell = (S_hi - S_lo + 1) * F.nk * F.nfl + 2;
    fl_search_cells_kernel<<<(ncell + 31) / 32, 32, 0, s>>>(P, F);
    st = after_launch("fl_search_cells");
    if (st != FXPQ_OK) return st;
    fl_search_select_kernel<<<1, 32, 0, s>>>(P, F, is_signed, d_err, d_best, d_stats, status_ptr());
    return after_launch("fl_search_select");
}

extern "C" fxpq_status fxpq_fl_init(const fxpq_stats* h_stats, int32_t bits, int32_t strategy, fxpq_fmt* h_out) {
    if (!h_stats || !h_out || bits < 2 || bits > 32 || strategy < 0 || strategy > 2) return FXPQ_ERR_INVALID_ARG;
    const double mn = h_stats->min, mx = h_stats->max;
    const int S = mn < 0.0 ? 1 : 0;
    double psi = 0.0;
    if (S == 0) {
        psi = mx / (ldexp(1.0, bits) - 1.0);
    } else {
        double a = mn / -ldexp(1.0, bits - 1), b = mx / (ldexp(1.0, bits - 1) - 1.0);
        psi = (a > 0 && b > 0) ? fmin(a, b) : (a > 0 ? a : b);
    }
    if (!(psi > 0.0) || !isfinite(psi)) return FXPQ_ERR_INVALID_ARG;
    const double bh = -log2(psi);
    double beta = strategy == 0 ? floor(bh) : (strategy == 1 ? nearbyint(bh) : ceil(bh));
    if (beta < -32 || beta > 40) return FXPQ_ERR_RANGE;
    h_out->bits = bits;
    h_out->is_signed = S;
    h_out->fl = (int32_t)beta;
    return FXPQ_OK;
}

// ------------------------------------------------------------------------------------------
// FL search without a caller workspace.
//
// Some callers cannot allocate device memory: a plug-in hosted by an application that owns the
// whole device memory pool, or a latency-critical loop that must never enter the allocator
// (cudaMalloc may synchronise the device).  For them the FL search's scratch (the exact integer
// bins and per-candidate cells, a fixed size independent of n) lives in this file-scope array,
// which every GPU that loads the library keeps until the process exits.
// ------------------------------------------------------------------------------------------
namespace {
constexpr size_t kFlSearchStaticBytes = (sizeof(FsGlobal) + 255) / 256 * 256;
static __device__ __align__(256) unsigned char g_fl_search_scratch[kFlSearchStaticBytes];

std::mutex g_fl_static_mu;
void* g_fl_static_addr[64] = {nullptr};

// Device address of g_fl_search_scratch on the current device, looked up once per device.
fxpq_status fl_search_scratch_ptr(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FXPQ_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_fl_static_mu);
    if (!g_fl_static_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_fl_search_scratch) != cudaSuccess || !p) return FXPQ_ERR_CUDA;
        g_fl_static_addr[dev] = p;
    }
    *out = g_fl_static_addr[dev];
    return FXPQ_OK;
}
}  // namespace

extern "C" fxpq_status fxpq_fl_search_noalloc(const float* d_x, int64_t n, int32_t is_signed, int32_t k_lo,
                                              int32_t k_hi, int32_t fl_lo, int32_t fl_hi, double* d_err,
                                              int32_t* d_best, fxpq_stats* d_stats, void* stream) {
    if (n < 0 || n > (int64_t(1) << 31)) return FXPQ_ERR_INVALID_ARG;  // the largest tensor the bins can hold
    if (k_lo < 2 || k_hi > 16 || k_lo > k_hi || fl_lo > fl_hi || fl_hi - fl_lo + 1 > MAXFL)
        return FXPQ_ERR_INVALID_ARG;  // the largest candidate grid the array holds: 15 x 32
    if (fxpq_fl_search_workspace(n) > kFlSearchStaticBytes) return FXPQ_ERR_WORKSPACE;
    void* scratch = nullptr;
    fxpq_status st = fl_search_scratch_ptr(&scratch);
    if (st != FXPQ_OK) return st;
    // fxpq_fl_search clears the bins it accumulates into before its first kernel.
    return fxpq_fl_search(d_x, n, is_signed, k_lo, k_hi, fl_lo, fl_hi, d_err, d_best, d_stats, scratch,
                          kFlSearchStaticBytes, stream);
}
