// fxpq_flsearch.cu -- batched FL search (Sec. IV-C, Eq. DSB_QE; sign strategy Sec. IV-A.3).
//
// Every candidate (k, FL) is scored exactly: L(k, FL) = sum_i (x_i - Q(x_i) 2^-FL)^2 as an exact
// rational, rounded once to nearest-even double.
//
// Decomposition.  Write fp32 x = (-1)^sg M 2^(E-23) (M the 24-bit significand, u_E = 2^(E-23)).
// For a candidate, y = |x| 2^FL has integer exponent q = E + FL, and Q clips at T (in y units):
// S=1: 2^t - 1 with t = k-1 for x >= 0, 2^t with t = k-1 for x < 0; S=0: 2^t - 1 with t = k for
// x >= 0, T = 0 for x < 0.  The element's error is (|x| - T 2^-FL)^2 when |y| >= T (saturated) and
// r^2 otherwise, r = y - round_half_even(y).  Hence, per (sign, E):
//   q >= t            every element saturates: a polynomial in T of the moments (n, sum M, sum M^2);
//   q == t-1, T=2^t-1 boundary: an element saturates iff M >= thr = (2^t - 1) 2^(24-t); its error
//                     is (M - thr)^2 u_E^2 if so, r^2 otherwise -- one "boundary remainder" sum Rb;
//   q <= -2           |y| < 1/2 rounds to 0: error x^2 = M^2 u_E^2 (a moment);
//   -1 <= q < bound   r^2 in units u_E^2 is the integer (M mod-round 2^(23-q))^2: a remainder sum R.
// All sums are integers; the finalize kernel adds one candidate's terms in a 768-bit fixed-point
// accumulator and rounds once.
//
// Pass structure (one HBM read of x).  Each block sorts a tile of 8192 elements by (sign, E) in
// shared memory (histogram, scan, scatter; the scatter re-reads the tile from L2); each warp then
// walks a contiguous run of the sorted tile, so runs of equal
// exponent are accumulated in registers (one slot per j = q) and reduced across the warp only when
// the exponent changes.  Block totals go to the workspace bins with integer atomics.
#include <math.h>

#include <algorithm>

#include <mutex>

#include "fxpq_common.cuh"

namespace fxpq {
namespace {

typedef unsigned long long u64;

constexpr int NKEY = 512;  // key = sign * 256 + biased exponent field (0..254; 255 = non-finite)
constexpr int NJ = 17;     // j = q in [-1, 15]
constexpr int MAXFL = 32;  // candidates per wordlength
constexpr int MAXK = 16;   // k in [1, 16]
constexpr int FS_THREADS = 256;
constexpr int FS_WARPS = FS_THREADS / 32;
constexpr int TILE = 8192;  // 32 elements per thread, read in sub-rounds of 16
constexpr int FS_BLOCKS_PER_SM = 3;
constexpr int CHUNK_MAX = 65536;  // per-block element cap: keeps every 64-bit block bin below 2^64
// Phase E balances the warps' shares of the sorted tile by elements plus this many per key they touch
// (a key change costs the warp a flush of its accumulators, about as long as this many elements).
constexpr unsigned FS_FLUSH_ELEMS = 128;

struct FsSmem {
    float sorted[TILE];
    unsigned cnt[NKEY];  // histogram, then running scatter offsets
    unsigned pn[NKEY];
    unsigned ps1[NKEY][2];  // 64-bit sums as {lo, hi} 32-bit words
    unsigned ps2[NKEY][2];
    unsigned r[2][NJ][MAXFL][2];
    unsigned rb[NJ][MAXFL][2];
    unsigned mn, mx, nonfinite, live;
    unsigned wbeg[FS_WARPS + 1];  // phase E: warp w walks sorted[wbeg[w], wbeg[w + 1])
};

// Workspace: exact bins, then per-candidate scores.  A sum bin is three 64-bit words w0, w1, w2 that
// stand for w0 + w1 2^32 + w2 2^64 (w2 two's complement): every contribution is split into 32-bit
// limbs and added with plain (non-returning) atomics, so no carry has to be propagated between
// words, and the sum of at most 2^32 limbs stays below 2^64 in every word.
struct FsGlobal {
    u64 pn[NKEY];
    u64 ps1[NKEY][3];
    u64 ps2[NKEY][3];
    u64 r[2][NJ][MAXFL][3];
    u64 rb[NJ][MAXFL][3];
    unsigned mn_inv, mx, nonfinite, fin_done;  // mn_inv = ~(smallest order key), 0: no finite element;
                                               // fin_done: finalize blocks done
    u64 nzero;                            // finite zeros (+-0.0): no key, but a binary-quantizer error
    double cells[2][MAXK][MAXFL];         // [S][k - 1][fl - fl_lo]
    double stat_sum, stat_sumsq;
    // Exact sums of squares by biased exponent eb, weight 2^(2(eb - 150)), that belong to every L2
    // cell and to the sum of squares but to no key's moments (the histogram kernel's sum of L^2)
    u64 cband[256][3];
};

struct FsParams {
    const float* x;
    long long n;
    int chunk;
    int fl_lo, nfl;
    int jmax_pos, jmax_neg;  // largest j whose remainder sum R is needed (x >= 0 / x < 0)
    int jb_lo, jb_hi;        // j range of the boundary sum Rb (x >= 0)
    // histogram kernel (fxpq_flsearch_hist.cuh): split bit s, the window's lowest biased exponent and
    // its keys per sign
    int hs_s;
    int hs_eb_lo;
    int hs_w;
    FsGlobal* g;
};

// A batch of independent searches (one per tensor) run by the same three launches.  Blocks of the
// bins kernel and warps of the cells kernel are assigned to items by the prefix arrays.
constexpr int FS_MAX_ITEMS = 32;

struct FsFinal {
    int S_lo, S_hi;
    int k_lo, nk;
    int fl_lo, nfl;
    int l1;  // score: 0 = L2 (Eq. DSB_QE), 1 = L1 (Eq. MAE as a sum)
};

struct FsBatch {
    int n_items;
    int blk0[FS_MAX_ITEMS + 1];   // first bins block of each item (bins launches cover item ranges)
    int cell0[FS_MAX_ITEMS + 1];  // first cell of each item in the finalize launch
    int fin0[FS_MAX_ITEMS + 1];   // first finalize block of each item
    FsParams p[FS_MAX_ITEMS];
    FsFinal f[FS_MAX_ITEMS];
};

__device__ __forceinline__ int batch_item(const int* start, int n, int idx) {
    int it = 0;
    while (it + 1 < n && idx >= start[it + 1]) ++it;
    return it;
}

__device__ __forceinline__ unsigned order_key(float x) {
    unsigned u = __float_as_uint(x);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float order_key_inv(unsigned k) {
    unsigned u = (k & 0x80000000u) ? (k & 0x7fffffffu) : ~k;
    return __uint_as_float(u);
}

// 64-bit add into {lo, hi} 32-bit shared words (native 32-bit atomics only)
__device__ __forceinline__ void sadd64(unsigned* p, u64 v) {
    if (!v) return;
    const unsigned lo = (unsigned)v;
    unsigned hi = (unsigned)(v >> 32);
    const unsigned old = atomicAdd(p, lo);
    hi += (old + lo < old) ? 1u : 0u;
    if (hi) atomicAdd(p + 1, hi);
}

// v into a three-limb sum bin (v >= 0)
__device__ __forceinline__ void gaddL(u64* p, u64 v) {
    if (!v) return;
    atomicAdd(p, v & 0xFFFFFFFFull);
    if (v >> 32) atomicAdd(p + 1, v >> 32);
}
// v (two's complement, |v| < 2^95) into a three-limb sum bin
__device__ __forceinline__ void gaddLs(u64* p, __int128 v) {
    if (!v) return;
    const unsigned __int128 w = (unsigned __int128)v;
    const u64 l0 = (u64)w & 0xFFFFFFFFull, l1 = (u64)(w >> 32) & 0xFFFFFFFFull;
    const long long l2 = (long long)(v >> 64);
    if (l0) atomicAdd(p, l0);
    if (l1) atomicAdd(p + 1, l1);
    if (l2) atomicAdd(p + 2, (u64)l2);
}

// Sum of a per-lane value v < 2^63 over the full warp (three 21-bit pieces, exact).
__device__ __forceinline__ u64 warp_sum64(u64 v) {
    const unsigned a = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v & 0x1FFFFFu));
    const unsigned b = __reduce_add_sync(0xFFFFFFFFu, (unsigned)((v >> 21) & 0x1FFFFFu));
    const unsigned c = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v >> 42));
    return (u64)a + ((u64)b << 21) + ((u64)c << 42);
}

__device__ __forceinline__ int key_of(float x) {
    const unsigned u = __float_as_uint(x);
    const unsigned eb = (u >> 23) & 0xFFu;
    if (eb == 0xFFu || (u & 0x7FFFFFFFu) == 0u) return NKEY;  // non-finite or zero: contributes nothing
    return (int)((u >> 31) * 256u + eb);
}

struct KeyInfo {
    int sg, E;
    unsigned validR, validRb;  // bit jj set: slot jj (j = jj - 1) is needed for this key
};

// Boundary sums of a narrow wordlength range (at most two boundary positions j = jb_lo, jb_lo + 1):
// per position the remainder mask and modulus of y's fraction and the saturation threshold of M.
struct RbC {
    unsigned mask[2], full[2], thr[2];
};

__device__ __forceinline__ RbC make_rbc(const FsParams& P) {
    RbC c;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int j = min(P.jb_lo + i, 15);  // j in [0, 15]; a position past jb_hi is never flushed
        c.full[i] = 1u << (23 - j);
        c.mask[i] = c.full[i] - 1u;
        c.thr[i] = ((2u << j) - 1u) << (23 - j);
    }
    return c;
}

__device__ __forceinline__ unsigned slot_mask(int jlo, int jhi) {
    // slots jj = j + 1 for j in [jlo, jhi] (empty when jhi < jlo)
    if (jhi < jlo) return 0u;
    return ((2u << (jhi + 1)) - 1u) & ~((1u << (jlo + 1)) - 1u);
}

__device__ __forceinline__ KeyInfo key_info(int key, const FsParams& P) {
    KeyInfo k;
    k.sg = key >> 8;
    const int eb = key & 255;
    k.E = eb ? eb - 127 : -126;
    // candidate FL in [fl_lo, fl_lo + nfl) puts j = E + FL in [E + fl_lo, E + fl_lo + nfl - 1]
    const int cand_lo = k.E + P.fl_lo, cand_hi = k.E + P.fl_lo + P.nfl - 1;
    const int jmax = k.sg ? P.jmax_neg : P.jmax_pos;
    k.validR = slot_mask(max(-1, cand_lo), min(min(jmax, NJ - 2), cand_hi));
    k.validRb = k.sg == 0 ? slot_mask(max(max(P.jb_lo, 0), cand_lo), min(min(P.jb_hi, NJ - 2), cand_hi)) : 0u;
    return k;
}

// Per-lane accumulators of the warp's current key; NS slots cover j = -1 .. NS-2.  Boundary sums:
// NRB = NS slots indexed like r (any wordlength range), or NRB = 2 slots for j = jb_lo, jb_lo + 1.
template <int NS, int NRB>
struct Acc {
    u64 r[NS];
    u64 rb[NRB];
    u64 s1, s2;
    unsigned n;
};

template <int NS, int NRB>
__device__ __forceinline__ void acc_zero(Acc<NS, NRB>& a) {
#pragma unroll
    for (int jj = 0; jj < NS; ++jj) a.r[jj] = 0ull;
#pragma unroll
    for (int i = 0; i < NRB; ++i) a.rb[i] = 0ull;
    a.s1 = a.s2 = 0ull;
    a.n = 0u;
}

// Narrow wordlength range: every remainder slot is computed without branches (slots the key does not
// use are never flushed).  The rounding error's magnitude is min(t, 2^p - t) for the fraction t of y
// in units of 2^-p, whichever way a tie rounds, so the parity of y's integer part is not needed.
// L1: first powers of the remainders (the L1 score), otherwise squares.
template <int NS, bool L1>
__device__ __forceinline__ void acc_add_narrow(Acc<NS, 2>& a, unsigned M, bool rb_on, const RbC& c) {
    a.n += 1u;
    a.s1 += M;
    a.s2 += (u64)M * M;
#pragma unroll
    for (int jj = 0; jj < NS; ++jj) {
        const unsigned full = 1u << (24 - jj);  // p = 23 - j bits below y's binary point
        const unsigned t = M & (full - 1u);
        const unsigned r = min(t, full - t);
        a.r[jj] += L1 ? (u64)r : (u64)r * r;
    }
    if (rb_on) {
        // boundary: saturated iff M >= thr, error (M - thr) u_E; otherwise the rounding error
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const unsigned t = M & c.mask[i];
            const unsigned r = min(t, c.full[i] - t);
            const unsigned rb = M >= c.thr[i] ? M - c.thr[i] : r;
            a.rb[i] += L1 ? (u64)rb : (u64)rb * rb;
        }
    }
}

// Add one element (significand M of the warp's current key) to this lane's accumulators.
template <int NS, bool L1>
__device__ __forceinline__ void acc_add(Acc<NS, NS>& a, unsigned M, const KeyInfo& k) {
    a.n += 1u;
    a.s1 += M;
    a.s2 += (u64)M * M;
#pragma unroll
    for (int jj = 0; jj < NS; ++jj) {
        const int j = jj - 1;
        const int p = 23 - j;  // bits of M below the binary point of y: 24 .. 8
        if (((k.validR | k.validRb) >> jj) & 1u) {
            const unsigned t = M & ((1u << p) - 1u);
            const unsigned odd = (M >> p) & 1u;
            const bool up = (t + odd) > (1u << (p - 1));
            const unsigned r = up ? (1u << p) - t : t;
            if ((k.validR >> jj) & 1u) a.r[jj] += L1 ? (u64)r : (u64)r * r;
            if (j >= 0 && ((k.validRb >> jj) & 1u)) {
                // boundary t' = j + 1: saturated iff M >= (2^(j+1) - 1) 2^(23-j)
                const unsigned thr = ((2u << j) - 1u) << (23 - j);
                const unsigned rb = M >= thr ? M - thr : r;
                a.rb[jj] += L1 ? (u64)rb : (u64)rb * rb;
            }
        }
    }
}

// Sum of 16 per-lane 64-bit values over the warp, scattered: on return v[0] of lanes 2 i and 2 i + 1
// holds the total of value i.  Four halving exchange stages (each lane keeps the half selected by one
// of its lane bits and adds its partner's copy of it), then one pairwise add.
__device__ __forceinline__ void warp_reduce_scatter16(u64 (&v)[16], unsigned lane) {
#pragma unroll
    for (int st = 0; st < 4; ++st) {
        const int half = 8 >> st;
        const unsigned o = 16u >> st;
        const bool b = (lane & o) != 0u;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const u64 mine = b ? v[half + i] : v[i];
            const u64 other = b ? v[i] : v[half + i];
            v[i] = mine + __shfl_xor_sync(0xFFFFFFFFu, other, o);
        }
    }
    v[0] += __shfl_xor_sync(0xFFFFFFFFu, v[0], 1);
}

// Warp totals of the current key's accumulators into the block bins.
// Narrow ranges (NRB = 2): the values (count, moments, remainder slots, boundary sums) are reduced in
// groups of 16 by exchange stages, and each even lane adds one total into its bin.  Wide ranges: every
// total by warp reductions first (independent, they pipeline), then one round of shared-memory
// atomics, value v by lane v % 32 (a second value per lane past 32).
template <int NS, int NRB>
__device__ __forceinline__ void acc_flush(FsSmem& sm, Acc<NS, NRB>& a, int key, const KeyInfo& k, const FsParams& P,
                                          unsigned lane) {
    if constexpr (NRB == 2) {
        constexpr int NV = 3 + NS + 2;  // count, s1, s2, r[0 .. NS), rb[0 .. 2)
        constexpr int NG = (NV + 15) / 16;
#pragma unroll
        for (int grp = 0; grp < NG; ++grp) {
            u64 v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int idx = 16 * grp + i;
                v[i] = idx == 0 ? (u64)a.n
                                : idx == 1 ? a.s1
                                           : idx == 2 ? a.s2
                                                      : idx < 3 + NS ? a.r[(idx - 3) < NS ? idx - 3 : 0]
                                                                     : idx < NV ? a.rb[(idx - 3 - NS) & 1] : 0ull;
            }
            warp_reduce_scatter16(v, lane);
            const int idx = 16 * grp + (int)(lane >> 1);
            if ((lane & 1u) || idx >= NV) continue;
            const u64 tot = v[0];
            if (idx == 0) {
                atomicAdd(&sm.pn[key], (unsigned)tot);
            } else if (idx == 1) {
                sadd64(sm.ps1[key], tot);
            } else if (idx == 2) {
                sadd64(sm.ps2[key], tot);
            } else if (idx < 3 + NS) {
                const int jj = idx - 3;
                if ((k.validR >> jj) & 1u) sadd64(sm.r[k.sg][jj][jj - 1 - k.E - P.fl_lo], tot);
            } else {
                const int jj = P.jb_lo + (idx - 3 - NS) + 1;
                if (jj < NJ && ((k.validRb >> jj) & 1u)) sadd64(sm.rb[jj][jj - 1 - k.E - P.fl_lo], tot);
            }
        }
    } else {
        const unsigned n = __reduce_add_sync(0xFFFFFFFFu, a.n);
        u64 v0 = 0ull, v1 = 0ull;  // this lane's totals
        unsigned o0 = 0u, o1 = 0u;  // and the byte offsets of their {lo, hi} bins in sm (0: none)
        char* const base = reinterpret_cast<char*>(&sm);
        auto take = [&](int idx, u64 v, unsigned* d) {
            if (lane == (unsigned)(idx & 31)) {
                const unsigned off = (unsigned)(reinterpret_cast<char*>(d) - base);
                if (idx < 32) {
                    v0 = v;
                    o0 = off;
                } else {
                    v1 = v;
                    o1 = off;
                }
            }
        };
        take(1, warp_sum64(a.s1), sm.ps1[key]);
        take(2, warp_sum64(a.s2), sm.ps2[key]);
#pragma unroll
        for (int jj = 0; jj < NS; ++jj) {
            const int fi = jj - 1 - k.E - P.fl_lo;
            if ((k.validR >> jj) & 1u) take(3 + jj, warp_sum64(a.r[jj]), sm.r[k.sg][jj][fi]);
            if ((k.validRb >> jj) & 1u) take(3 + NS + jj, warp_sum64(a.rb[jj < NRB ? jj : 0]), sm.rb[jj][fi]);
        }
        if (lane == 0) atomicAdd(&sm.pn[key], n);
        if (o0) sadd64(reinterpret_cast<unsigned*>(base + o0), v0);
        if (o1) sadd64(reinterpret_cast<unsigned*>(base + o1), v1);
    }
}

// 16 consecutive-by-thread elements of sub-round `sub` of the tile starting at tb: values and keys
// (NKEY for zeros, non-finite values and positions past the end).
template <bool VEC>
__device__ __forceinline__ void load16(const FsParams& P, long long tb, int sub, long long end, float (&v)[16],
                                       int (&key)[16]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const long long idx = tb + (long long)sub * 4096 + 1024LL * i + 4LL * threadIdx.x;
        if (VEC && idx + 3 < end) {
            const float4 f = __ldg(reinterpret_cast<const float4*>(P.x + idx));
            v[4 * i] = f.x, v[4 * i + 1] = f.y, v[4 * i + 2] = f.z, v[4 * i + 3] = f.w;
#pragma unroll
            for (int e = 0; e < 4; ++e) key[4 * i + e] = key_of(v[4 * i + e]);
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool in = idx + e < end;
                v[4 * i + e] = in ? P.x[idx + e] : 0.0f;
                key[4 * i + e] = in ? key_of(v[4 * i + e]) : NKEY;
            }
        }
    }
}

template <bool VEC, int NS, int NRB, bool L1>
__global__ void __launch_bounds__(FS_THREADS, NRB == 2 ? FS_BLOCKS_PER_SM : 2)
    fl_search_bins_kernel(const __grid_constant__ FsBatch B, int item0, int item1) {
    // this launch covers items [item0, item1); blk0 holds their block offsets relative to the launch
    const int item = item0 + batch_item(B.blk0 + item0, item1 - item0, (int)blockIdx.x);
    const FsParams& P = B.p[item];
    const int blk = (int)blockIdx.x - B.blk0[item];
    extern __shared__ __align__(16) unsigned char fs_smem_raw[];
    FsSmem& sm = *reinterpret_cast<FsSmem*>(fs_smem_raw);
    const unsigned lane = threadIdx.x & 31u, warp = threadIdx.x >> 5;
    {
        unsigned* z = reinterpret_cast<unsigned*>(&sm.cnt[0]);
        const int nz = (int)((sizeof(FsSmem) - sizeof(sm.sorted)) / 4);
        for (int i = threadIdx.x; i < nz; i += FS_THREADS) z[i] = 0u;
    }
    __syncthreads();
    if (threadIdx.x == 0) sm.mn = 0xFFFFFFFFu;
    unsigned tmn = 0xFFFFFFFFu, tmx = 0u;
    unsigned tz = 0u;  // finite zeros
    bool tnf = false;

    const long long start = (long long)blk * P.chunk;
    const long long end = min(start + (long long)P.chunk, P.n);
    const RbC rbc = make_rbc(P);
    for (long long tb = start; tb < end; tb += TILE) {
        // ---- A+B: read the tile (16 elements per thread per sub-round), stats, key histogram
        for (int sub = 0; sub < TILE / 4096; ++sub) {
            float v[16];
            int key[16];
            load16<VEC>(P, tb, sub, end, v, key);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                const long long idx = tb + (long long)sub * 4096 + 1024LL * (e / 4) + 4LL * threadIdx.x + (e % 4);
                if (idx < end) {
                    const unsigned u = __float_as_uint(v[e]);
                    if (((u >> 23) & 0xFFu) == 0xFFu) {
                        tnf = true;
                    } else {
                        const unsigned ok = order_key(v[e]);
                        tmn = min(tmn, ok);
                        tmx = max(tmx, ok);
                        tz += (u & 0x7FFFFFFFu) == 0u ? 1u : 0u;
                    }
                }
                // per-element shared-memory reduction (no value returned); lanes with equal keys
                // serialise in the memory pipe instead of a warp-wide match
                if (key[e] < NKEY) atomicAdd(&sm.cnt[key[e]], 1u);
            }
        }
        __syncthreads();
        // ---- C: exclusive scan of the 512 counts (warp 0)
        if (warp == 0) {
            unsigned loc[NKEY / 32];
            unsigned s = 0;
#pragma unroll
            for (int i = 0; i < NKEY / 32; ++i) {
                loc[i] = sm.cnt[lane * (NKEY / 32) + i];
                s += loc[i];
            }
            unsigned incl = s;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const unsigned o = __shfl_up_sync(0xFFFFFFFFu, incl, off);
                if (lane >= (unsigned)off) incl += o;
            }
            unsigned run = incl - s;
            const unsigned first = run;  // sorted position of this lane's first key
#pragma unroll
            for (int i = 0; i < NKEY / 32; ++i) {
                sm.cnt[lane * (NKEY / 32) + i] = run;
                run += loc[i];
            }
            if (lane == 31) sm.live = incl;
            // the warps' shares of phase E: equal in elements plus FS_FLUSH_ELEMS per key present
            unsigned e = 0;
#pragma unroll
            for (int i = 0; i < NKEY / 32; ++i) e += loc[i] + (loc[i] ? FS_FLUSH_ELEMS : 0u);
            unsigned eincl = e;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const unsigned o = __shfl_up_sync(0xFFFFFFFFu, eincl, off);
                if (lane >= (unsigned)off) eincl += o;
            }
            const unsigned eexcl = eincl - e, etot = __shfl_sync(0xFFFFFFFFu, eincl, 31);
            const unsigned total = __shfl_sync(0xFFFFFFFFu, incl, 31);
            if (lane < FS_WARPS) sm.wbeg[lane] = 0u;
            if (lane == 0) sm.wbeg[FS_WARPS] = total;
            __syncwarp();
            // every lane checks its own keys against the FS_WARPS - 1 boundaries (each falls in one key)
            unsigned ec = eexcl, pos = first;
#pragma unroll
            for (int i = 0; i < NKEY / 32; ++i) {
                const unsigned ke = loc[i] + (loc[i] ? FS_FLUSH_ELEMS : 0u);
#pragma unroll
                for (int w = 1; w < FS_WARPS; ++w) {
                    const unsigned T = (unsigned)(((unsigned long long)etot * (unsigned)w) / FS_WARPS);
                    if (T >= ec && T < ec + ke) sm.wbeg[w] = pos + min(T - ec, loc[i]);
                }
                ec += ke;
                pos += loc[i];
            }
        }
        __syncthreads();
        // ---- D: scatter into key order (the tile is read again; it is L2-resident)
        for (int sub = 0; sub < TILE / 4096; ++sub) {
            float v[16];
            int key[16];
            load16<VEC>(P, tb, sub, end, v, key);
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                // each element takes the next free position of its key (order within a key is
                // immaterial: every sum is exact)
                if (key[e] < NKEY) sm.sorted[atomicAdd(&sm.cnt[key[e]], 1u)] = v[e];
            }
        }
        __syncthreads();
        // ---- E: each warp walks a contiguous run of the sorted tile
        const int w0 = (int)sm.wbeg[warp], w1 = (int)sm.wbeg[warp + 1];
        Acc<NS, NRB> acc;
        acc_zero(acc);
        int ck = -1;
        KeyInfo ki;
        ki.sg = 0, ki.E = 0, ki.validR = ki.validRb = 0u;
        // one step of lookahead: the next group's shared-memory load is in flight while this one is
        // accumulated
        float xn = w0 + (int)lane < w1 ? sm.sorted[w0 + lane] : 0.0f;
        for (int pos = w0; pos < w1; pos += 32) {
            const int p = pos + (int)lane;
            const bool live = p < w1;
            const float xv = xn;
            xn = p + 32 < w1 ? sm.sorted[p + 32] : 0.0f;
            const int kx = live ? key_of(xv) : NKEY;
            const unsigned u = __float_as_uint(xv);
            const unsigned eb = (u >> 23) & 0xFFu;
            const unsigned M = eb ? ((u & 0x7FFFFFu) | 0x800000u) : (u & 0x7FFFFFu);
            // common case: every lane is live and continues the current key
            if (__all_sync(0xFFFFFFFFu, kx == ck)) {
                if constexpr (NRB == 2)
                    acc_add_narrow<NS, L1>(acc, M, ki.validRb != 0u, rbc);
                else
                    acc_add<NS, L1>(acc, M, ki);
                continue;
            }
            unsigned rem = __ballot_sync(0xFFFFFFFFu, live);
            while (rem) {
                const int kk = __shfl_sync(0xFFFFFFFFu, kx, __ffs(rem) - 1);
                const unsigned in = __ballot_sync(0xFFFFFFFFu, live && kx == kk);
                if (kk != ck) {
                    if (ck >= 0) {
                        acc_flush(sm, acc, ck, ki, P, lane);
                        acc_zero(acc);
                    }
                    ck = kk;
                    ki = key_info(ck, P);
                }
                if ((in >> lane) & 1u) {
                    if constexpr (NRB == 2)
                        acc_add_narrow<NS, L1>(acc, M, ki.validRb != 0u, rbc);
                    else
                        acc_add<NS, L1>(acc, M, ki);
                }
                rem &= ~in;
            }
        }
        if (ck >= 0) acc_flush(sm, acc, ck, ki, P, lane);
        __syncthreads();
        for (int i = threadIdx.x; i < NKEY; i += FS_THREADS) sm.cnt[i] = 0u;
        __syncthreads();
    }
    atomicMin(&sm.mn, tmn);
    atomicMax(&sm.mx, tmx);
    if (tnf) sm.nonfinite = 1u;
    {
        const unsigned zw = __reduce_add_sync(0xFFFFFFFFu, tz);
        if (lane == 0 && zw) atomicAdd(&P.g->nzero, (u64)zw);
    }
    __syncthreads();

    // ---- block bins -> exact workspace bins
    FsGlobal* g = P.g;
    for (int i = threadIdx.x; i < NKEY; i += FS_THREADS) {
        if (!sm.pn[i]) continue;
        atomicAdd(&g->pn[i], (u64)sm.pn[i]);
        gaddL(g->ps1[i], ((u64)sm.ps1[i][1] << 32) | sm.ps1[i][0]);
        gaddL(g->ps2[i], ((u64)sm.ps2[i][1] << 32) | sm.ps2[i][0]);
    }
    for (int i = threadIdx.x; i < 2 * NJ * MAXFL; i += FS_THREADS) {
        const int s = i / (NJ * MAXFL), j = (i / MAXFL) % NJ, f = i % MAXFL;
        gaddL(g->r[s][j][f], ((u64)sm.r[s][j][f][1] << 32) | sm.r[s][j][f][0]);
    }
    for (int i = threadIdx.x; i < NJ * MAXFL; i += FS_THREADS) {
        const int j = i / MAXFL, f = i % MAXFL;
        gaddL(g->rb[j][f], ((u64)sm.rb[j][f][1] << 32) | sm.rb[j][f][0]);
    }
    if (threadIdx.x == 0) {
        if (sm.mn != 0xFFFFFFFFu) atomicMax(&g->mn_inv, ~sm.mn);
        atomicMax(&g->mx, sm.mx);
        if (sm.nonfinite) atomicOr(&g->nonfinite, 1u);
    }
}

}  // namespace
}  // namespace fxpq

#include "fxpq_flsearch_hist.cuh"

namespace fxpq {
namespace {

// ------------------------------------------------------------------ exact finalize
struct U128 {
    u64 lo, hi;
};
// (a * m) for a 128-bit a and 64-bit m: the callers' bounds keep the product below 2^128
__device__ __forceinline__ U128 mul128_64(U128 a, u64 m) {
    U128 r;
    r.lo = a.lo * m;
    r.hi = __umul64hi(a.lo, m) + a.hi * m;
    return r;
}

// 768-bit two's complement fixed point: word i weighs 2^(64 i - 320)
constexpr int BW = 12;
constexpr int BBASE = -320;

struct Big {
    u64 w[BW];
};

// A cell's exact sum is gathered in 24 signed 64-bit columns in shared memory, column c weighing
// 2^(32 c + BBASE): every term is cut into 32-bit pieces added to their columns (shared-memory
// atomics, so the lanes of a warp share one set), and one carry pass turns the columns into the
// 768-bit two's complement value.  A column takes well under 2^31 pieces, so it cannot overflow;
// pieces above column 23 weigh multiples of 2^(768 + BBASE) and drop, as modulo 2^768 they must.
constexpr int NCOL = 2 * BW;

// col += (neg ? -1 : 1) * v * 2^e for a 128-bit magnitude v
__device__ __forceinline__ void col_add(u64* col, U128 v, int e, bool neg) {
    if ((v.lo | v.hi) == 0ull) return;
    const int pos = e - BBASE;
    const int ci = pos >> 5;
    const unsigned b = (unsigned)pos & 31u;
    const unsigned x0 = (unsigned)v.lo, x1 = (unsigned)(v.lo >> 32), x2 = (unsigned)v.hi,
                   x3 = (unsigned)(v.hi >> 32);
    const unsigned c[5] = {x0 << b, __funnelshift_l(x0, x1, b), __funnelshift_l(x1, x2, b),
                           __funnelshift_l(x2, x3, b), __funnelshift_l(x3, 0u, b)};
#pragma unroll
    for (int j = 0; j < 5; ++j)
        if (c[j] && ci + j < NCOL) atomicAdd(&col[ci + j], neg ? (u64)(-(long long)c[j]) : (u64)c[j]);
}

// The columns' value as a 768-bit two's complement number.
__device__ void col_to_big(const u64* col, Big& a) {
    long long carry = 0;
#pragma unroll
    for (int i = 0; i < BW; ++i) {
        const long long t0 = (long long)col[2 * i] + carry;
        const long long t1 = (long long)col[2 * i + 1] + (t0 >> 32);
        carry = t1 >> 32;
        a.w[i] = (u64)(unsigned)t0 | ((u64)(unsigned)t1 << 32);
    }
}

// a += (neg ? -1 : 1) * m * 2^e * (the three-limb bin at p).  The top limb is signed: the histogram
// kernel's remainder sums leave out the sum of L^2 that its exponent band carries, so one key's
// share of a cell may be negative.
__device__ __forceinline__ void col_add_L3(u64* a, const u64* p, int e, bool neg, u64 m = 1ull) {
    col_add(a, mul128_64(U128{p[0], 0ull}, m), e, neg);
    col_add(a, mul128_64(U128{p[1], 0ull}, m), e + 32, neg);
    const long long w2 = (long long)p[2];
    if (w2) col_add(a, mul128_64(U128{w2 < 0 ? (u64)(-w2) : (u64)w2, 0ull}, m), e + 64, neg != (w2 < 0));
}

__device__ u64 big_bits64(const Big& a, int pos) {  // bits [pos, pos + 64), zero below bit 0
    const int wi = pos >= 0 ? (pos >> 6) : -((-pos + 63) >> 6);
    const int b = pos - wi * 64;
    const u64 lo = (wi >= 0 && wi < BW) ? a.w[wi] : 0ull;
    const u64 hi = (wi + 1 >= 0 && wi + 1 < BW) ? a.w[wi + 1] : 0ull;
    return b ? ((lo >> b) | (hi << (64 - b))) : lo;
}

__device__ bool big_any_below(const Big& a, int pos) {
    if (pos <= 0) return false;
    const int wi = pos >> 6, b = pos & 63;
    for (int i = 0; i < wi && i < BW; ++i)
        if (a.w[i]) return true;
    return wi < BW && b && (a.w[wi] & ((1ull << b) - 1ull));
}

// round a non-negative accumulator to nearest-even double (negative -> -1, a sentinel)
__device__ double big_to_double(const Big& a) {
    if ((long long)a.w[BW - 1] < 0) return -1.0;
    int h = -1;
    for (int i = BW - 1; i >= 0; --i)
        if (a.w[i]) {
            h = i;
            break;
        }
    if (h < 0) return 0.0;
    const int top = 64 * h + 63 - __clzll(a.w[h]);
    const u64 win = big_bits64(a, top - 63);
    u64 mant = win >> 11;
    const bool rb = (win >> 10) & 1ull;
    const bool sticky = (win & 0x3FFull) != 0ull || big_any_below(a, top - 63);
    if (rb && (sticky || (mant & 1ull))) mant += 1ull;
    return ldexp((double)mant, top - 52 + BBASE);
}

__device__ void big_negate(Big& a) {
    u64 c = 1ull;
    for (int i = 0; i < BW; ++i) {
        const u64 t = ~a.w[i] + c;
        c = (c && t == 0ull) ? 1ull : 0ull;
        a.w[i] = t;
    }
}

// saturated set with moments (n, s1, s2) at exponent E: s2 2^(2(E-23)) - 2 T s1 2^(E-23-fl) + T^2 n 2^(-2fl)
__device__ void add_sat(u64* acc, u64 n, const u64* s1, const u64* s2, int E, int fl, u64 T) {
    col_add_L3(acc, s2, 2 * (E - 23), false);
    if (T) {
        col_add_L3(acc, s1, E - 23 - fl, true, 2ull * T);
        col_add(acc, mul128_64(U128{n, 0ull}, T * T), -2 * fl, false);
    }
}

// ------------------------------------------------------------------ finalize: scores, argmin, stats
constexpr int FIN_T = 256;            // threads per finalize block
constexpr int FIN_WARPS = FIN_T / 32;  // cells per finalize block, one per warp

// The keys with elements and the non-zero exponent sums of squares of one item, staged per block,
// and every warp's column accumulator.
struct FinSmem {
    unsigned nkey, nband, last;
    unsigned key[NKEY];
    u64 n[NKEY];
    u64 s1[NKEY][3];
    u64 s2[NKEY][3];
    unsigned beb[256];
    u64 band[256][3];
    u64 col[FIN_WARPS][NCOL];
};

__device__ void fin_stage(FinSmem& sm, const FsGlobal* g) {
    if (threadIdx.x == 0) sm.nkey = sm.nband = 0u;
    __syncthreads();
    for (int key = threadIdx.x; key < NKEY; key += blockDim.x) {
        const u64 n = g->pn[key];
        if (!n) continue;
        const unsigned i = atomicAdd(&sm.nkey, 1u);
        sm.key[i] = (unsigned)key;
        sm.n[i] = n;
#pragma unroll
        for (int w = 0; w < 3; ++w) {
            sm.s1[i][w] = g->ps1[key][w];
            sm.s2[i][w] = g->ps2[key][w];
        }
    }
    for (int eb = threadIdx.x; eb < 256; eb += blockDim.x) {
        const u64 a = g->cband[eb][0], b = g->cband[eb][1], c = g->cband[eb][2];
        if (!(a | b | c)) continue;
        const unsigned i = atomicAdd(&sm.nband, 1u);
        sm.beb[i] = (unsigned)eb;
        sm.band[i][0] = a;
        sm.band[i][1] = b;
        sm.band[i][2] = c;
    }
    __syncthreads();
}

// The exact value of one cell (candidate (S, k, FL), or the two stats cells) added to a warp's
// columns: the lanes split the staged keys.
__device__ void fin_cell(u64* acc, const FinSmem& sm, const FsGlobal* g, const FsFinal& F, int cell, int ncell,
                         int lane, int nlanes) {
    // the exponent-indexed sums of squares that belong to every L2 cell and to the sum of squares
    const bool with_band = cell == ncell + 1 || (cell < ncell && !F.l1);
    if (with_band)
        for (unsigned i = lane; i < sm.nband; i += nlanes) col_add_L3(acc, sm.band[i], 2 * ((int)sm.beb[i] - 150), false);
    if (cell >= ncell) {
        const bool sq = cell == ncell + 1;
        for (unsigned i = lane; i < sm.nkey; i += nlanes) {
            const int key = (int)sm.key[i];
            const int eb = key & 255, E = eb ? eb - 127 : -126;
            if (sq)
                col_add_L3(acc, sm.s2[i], 2 * (E - 23), false);
            else
                col_add_L3(acc, sm.s1[i], E - 23, (key >> 8) != 0);
        }
    } else if (F.k_lo == 1 && F.S_lo + cell / (F.nk * F.nfl) == 1 && (cell % (F.nk * F.nfl)) / F.nfl == 0) {
        // k = 1, S = 1: the binary quantizer (Eq. fp_1_bit_quantization), every value decoded to
        // +-c with c = 2^-fl, so the error of x is | |x| - c |: from the moments alone, zeros included
        const int fl = F.fl_lo + cell % F.nfl;
        if (lane == 0) {
            const U128 nz{g->nzero, 0ull};
            col_add(acc, nz, F.l1 ? -fl : -2 * fl, false);
        }
        for (unsigned i = lane; i < sm.nkey; i += nlanes) {
            const int key = (int)sm.key[i];
            const u64 n = sm.n[i];
            const int eb = key & 255, E = eb ? eb - 127 : -126;
            if (!F.l1) {
                add_sat(acc, n, sm.s1[i], sm.s2[i], E, fl, 1ull);  // sum (|x| - c)^2
            } else {
                // |x| >= 2^E >= c when E >= -fl, else |x| < 2^(E+1) <= c
                const bool above = E >= -fl;
                col_add_L3(acc, sm.s1[i], E - 23, !above);
                col_add(acc, U128{n, 0ull}, -fl, above);
            }
        }
    } else {
        const int S = F.S_lo + cell / (F.nk * F.nfl);
        const int rem = cell % (F.nk * F.nfl);
        const int k = F.k_lo + rem / F.nfl;
        const int fi = rem % F.nfl;
        const int fl = F.fl_lo + fi;
        // L2 terms weigh u_E^2 = 2^(2(E-23)), L1 terms u_E = 2^(E-23)
        const int pw = F.l1 ? 1 : 2;
        for (unsigned i = lane; i < sm.nkey; i += nlanes) {
            const int key = (int)sm.key[i];
            const u64 n = sm.n[i];
            const int sg = key >> 8, eb = key & 255, E = eb ? eb - 127 : -126;
            const u64* s1 = sm.s1[i];
            const u64* s2 = sm.s2[i];
            if (sg == 1 && S == 0) {  // clipped to code 0: error |x|
                col_add_L3(acc, F.l1 ? s1 : s2, pw * (E - 23), false);
                continue;
            }
            const int t = (sg == 0) ? (S ? k - 1 : k) : (k - 1);
            const u64 T = (sg == 0) ? ((1ull << t) - 1ull) : (1ull << t);
            const int q = E + fl;
            if (q >= t) {
                if (F.l1) {  // |x| >= T 2^-fl: sum |x| - n T 2^-fl
                    col_add_L3(acc, s1, E - 23, false);
                    col_add(acc, U128{n * T, 0ull}, -fl, true);
                } else {
                    add_sat(acc, n, s1, s2, E, fl, T);
                }
            } else if (sg == 0 && q == t - 1) {
                col_add_L3(acc, g->rb[q + 1][fi], pw * (E - 23), false);
            } else if (q <= -2) {
                col_add_L3(acc, F.l1 ? s1 : s2, pw * (E - 23), false);
            } else {
                col_add_L3(acc, g->r[sg][q + 1][fi], pw * (E - 23), false);
            }
        }
    }
}

// Per-item outputs.
struct FsOut {
    double* err;
    int* best;
    fxpq_stats* stats;
    int is_signed;
};
struct FsOutBatch {
    FsOut o[FS_MAX_ITEMS];
};

// Finalize: one warp per cell of one item (the cells of every S, k, FL, then the two stats cells),
// FIN_WARPS cells per block.  The block stages the item's keys once; each warp's lanes score their
// share of the keys into the warp's columns, and lane 0 turns them into the exact 768-bit value and
// its nearest double.  The item's last block to finish (completion ticket) writes the scores, the
// argmin per wordlength (exact ties keep the smaller FL) and the stats.
__global__ void __launch_bounds__(FIN_T) fl_search_final_kernel(const __grid_constant__ FsBatch B,
                                                                 const __grid_constant__ FsOutBatch O, int* status) {
    const int item = batch_item(B.fin0, B.n_items, (int)blockIdx.x);
    const FsParams& P = B.p[item];
    const FsFinal& F = B.f[item];
    const FsOut& out = O.o[item];
    FsGlobal* g = P.g;
    __shared__ FinSmem sm;
    const int nblk = B.fin0[item + 1] - B.fin0[item];
    const int ncell = (F.S_hi - F.S_lo + 1) * F.nk * F.nfl;
    const int tid = (int)threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int cell = ((int)blockIdx.x - B.fin0[item]) * FIN_WARPS + warp;
    u64* col = sm.col[warp];
    if (lane < NCOL) col[lane] = 0ull;
    fin_stage(sm, g);
    if (cell < ncell + 2) {  // warp-uniform
        fin_cell(col, sm, g, F, cell, ncell, lane, 32);
        __syncwarp();
        if (lane == 0) {
            Big acc;
            col_to_big(col, acc);
            if (cell == ncell) {
                const bool neg = (long long)acc.w[BW - 1] < 0;
                if (neg) big_negate(acc);
                const double v = big_to_double(acc);
                g->stat_sum = neg ? -v : v;
            } else if (cell == ncell + 1) {
                g->stat_sumsq = big_to_double(acc);
            } else {
                const int S = F.S_lo + cell / (F.nk * F.nfl);
                const int rem = cell % (F.nk * F.nfl);
                g->cells[S][F.k_lo + rem / F.nfl - 1][rem % F.nfl] = big_to_double(acc);
            }
            __threadfence();
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        sm.last = atomicAdd(&g->fin_done, 1u) == (unsigned)(nblk - 1) ? 1u : 0u;
    }
    __syncthreads();
    if (!sm.last) return;
    __threadfence();
    const float mn = g->mn_inv == 0u ? 0.0f : order_key_inv(~g->mn_inv);
    const float mx = g->mx == 0u ? 0.0f : order_key_inv(g->mx);
    const int S = out.is_signed >= 0 ? out.is_signed : (mn < 0.0f ? 1 : 0);
    for (int i = warp; i < F.nk; i += FIN_T / 32) {  // one warp per wordlength, one lane per FL
        const int k = F.k_lo + i;
        double v = __longlong_as_double(0x7FF0000000000000ll);
        if (lane < F.nfl) {
            v = __ldcg(&g->cells[S][k - 1][lane]);
            out.err[(long long)i * F.nfl + lane] = v;
        }
        int bf = lane;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const double ov = __shfl_down_sync(0xFFFFFFFFu, v, off);
            const int of = __shfl_down_sync(0xFFFFFFFFu, bf, off);
            if (ov < v || (ov == v && of < bf)) {  // exact ties keep the smaller FL
                v = ov;
                bf = of;
            }
        }
        if (lane == 0) out.best[i] = F.fl_lo + bf;
    }
    if (threadIdx.x == 0) {
        if (g->nonfinite) latch_status(status, FXPQ_ERR_NONFINITE);
        if (out.stats) {
            out.stats->min = mn;
            out.stats->max = mx;
            out.stats->is_signed = S;
            out.stats->nonfinite = g->nonfinite ? 1 : 0;
            out.stats->sum = __ldcg(&g->stat_sum);
            out.stats->sumsq = __ldcg(&g->stat_sumsq);
            out.stats->n = P.n;
        }
    }
}

}  // namespace
}  // namespace fxpq

using namespace fxpq;

namespace {
std::mutex g_fs_attr_mu;
bool g_fs_attr_done = false;
// The bins kernel's shared memory exceeds the 48 KB default; raise the limit once per process.
void st_attr_once() {
    std::lock_guard<std::mutex> lk(g_fs_attr_mu);
    if (g_fs_attr_done) return;
    const int sb = (int)sizeof(FsSmem);
#define FXPQ_FS_ATTR(V, L1)                                                                                      \
    cudaFuncSetAttribute(fl_search_bins_kernel<V, 10, 2, L1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sb); \
    cudaFuncSetAttribute(fl_search_bins_kernel<V, NJ, 2, L1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sb); \
    cudaFuncSetAttribute(fl_search_bins_kernel<V, NJ, NJ, L1>, cudaFuncAttributeMaxDynamicSharedMemorySize, sb);
    FXPQ_FS_ATTR(true, false)
    FXPQ_FS_ATTR(false, false)
    FXPQ_FS_ATTR(true, true)
    FXPQ_FS_ATTR(false, true)
#undef FXPQ_FS_ATTR
    const int hb = (int)HS_SMEM;
    cudaFuncSetAttribute(fl_search_hist_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, hb);
    cudaFuncSetAttribute(fl_search_hist_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, hb);
    cudaFuncSetAttribute(fl_search_hist_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, hb);
    cudaFuncSetAttribute(fl_search_hist_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, hb);
    g_fs_attr_done = true;
}
}  // namespace

namespace {
constexpr size_t kFsGlobalBytes = (sizeof(FsGlobal) + 255) / 256 * 256;

// One search of a batch, prepared on the host.
struct FsItemHost {
    FsParams p;
    FsFinal f;
    FsOut o;
    int variant;  // bins kernel instance: bit 0 vec, bit 1 small (k_hi <= 9), bit 2 narrow boundary range,
                  // bit 3 L1 score, bit 4 the histogram kernel (then bits 1-2 are clear)
    int grid;     // bins blocks
};

// The histogram kernel serves a search when every slot it needs has j <= 7: split bit
// s = min(16, 22 - jneed) >= 15.  Window: the exponents E with a needed slot for some candidate FL,
// E in [-1 - fl_hi, jneed - fl_lo]; below it every candidate rounds to zero, above it every one
// saturates.  Both signs take the same window and split (negative keys of an unsigned-only search
// need their moments alone).
bool hs_configure(FsParams& P, int S_hi) {
    const int fl_hi = P.fl_lo + P.nfl - 1;
    const int jneed = max(max(P.jmax_pos, P.jb_hi), S_hi == 1 ? P.jmax_neg : -1);
    if (jneed > 7) return false;
    P.hs_s = min(16, 22 - max(jneed, -1));
    const int e_lo = -1 - fl_hi, e_hi = max(jneed, -1) - P.fl_lo;
    P.hs_eb_lo = e_lo + 127;
    P.hs_w = e_hi - e_lo + 1;
    // every window exponent is a normal one (fl in [-32, 40], j <= 7)
    return P.hs_eb_lo >= 1 && P.hs_eb_lo + P.hs_w - 1 <= 254;
}

fxpq_status fs_prepare(const fxpq_fl_search_item& it, FsGlobal* g, FsItemHost& h) {
    const int64_t n = it.n;
    if (n < 0 || n > (int64_t(1) << 31)) return FXPQ_ERR_INVALID_ARG;
    if (it.is_signed < -1 || it.is_signed > 1) return FXPQ_ERR_INVALID_ARG;
    if (it.k_lo < 1 || it.k_hi > 16 || it.k_lo > it.k_hi) return FXPQ_ERR_INVALID_ARG;
    if (it.score != FXPQ_SCORE_L2 && it.score != FXPQ_SCORE_L1) return FXPQ_ERR_INVALID_ARG;
    if (it.fl_lo < -32 || it.fl_hi > 40 || it.fl_lo > it.fl_hi || it.fl_hi - it.fl_lo + 1 > MAXFL)
        return FXPQ_ERR_INVALID_ARG;
    if (!it.d_err || !it.d_best || (n > 0 && !it.d_x)) return FXPQ_ERR_INVALID_ARG;
    const int S_lo = it.is_signed < 0 ? 0 : it.is_signed, S_hi = it.is_signed < 0 ? 1 : it.is_signed;
    FsParams& P = h.p;
    P.x = it.d_x;
    P.n = n;
    // whole waves of resident blocks, each chunk at most CHUNK_MAX elements
    const long long resident = 152LL * FS_BLOCKS_PER_SM;
    const long long waves = n > 0 ? (n + resident * CHUNK_MAX - 1) / (resident * CHUNK_MAX) : 1;
    const long long per = (n + resident * waves - 1) / (resident * waves);
    long long chunk = (per + TILE - 1) / TILE * TILE;
    if (chunk < TILE) chunk = TILE;
    if (chunk > CHUNK_MAX) chunk = CHUNK_MAX;
    P.chunk = (int)chunk;
    P.fl_lo = it.fl_lo;
    P.nfl = it.fl_hi - it.fl_lo + 1;
    // x >= 0 rounds (no clip) for q <= t-2 with t = k-1 (S=1) or k (S=0); x < 0 (S=1) for q <= k-2
    P.jmax_pos = (S_lo == 0) ? it.k_hi - 2 : it.k_hi - 3;
    P.jmax_neg = (S_hi == 1) ? it.k_hi - 2 : -2;
    // boundary q = t-1 for x >= 0
    P.jb_lo = (S_hi == 1) ? it.k_lo - 2 : it.k_lo - 1;
    P.jb_hi = (S_lo == 0) ? it.k_hi - 1 : it.k_hi - 2;
    if (P.jb_lo < 0) P.jb_lo = 0;
    P.g = g;
    h.f.S_lo = S_lo;
    h.f.S_hi = S_hi;
    h.f.k_lo = it.k_lo;
    h.f.nk = it.k_hi - it.k_lo + 1;
    h.f.fl_lo = it.fl_lo;
    h.f.nfl = P.nfl;
    h.f.l1 = it.score == FXPQ_SCORE_L1 ? 1 : 0;
    h.o.err = it.d_err;
    h.o.best = it.d_best;
    h.o.stats = it.d_stats;
    h.o.is_signed = it.is_signed;
    h.grid = (int)((n + chunk - 1) / chunk);
    h.variant = (aligned(it.d_x, 16) ? 1 : 0) | (it.k_hi <= 9 ? 2 : 0) | (P.jb_hi - P.jb_lo + 1 <= 2 ? 4 : 0) |
                (h.f.l1 ? 8 : 0);
    if (hs_configure(P, S_hi) && hs_fits(P)) {
        // one block per SM, at most HS_CHUNK_MAX elements each: whole iterations per block except the
        // last where a block gets one or more (the partial pass exposes a load latency), else equal
        // chunks below one iteration (multiples of 4 elements: 16-byte aligned starts), at least one
        // float4 per thread
        const long long waves = n > 0 ? (n + 152LL * HS_CHUNK_MAX - 1) / (152LL * HS_CHUNK_MAX) : 1;
        long long per = (n + 152 * waves - 1) / (152 * waves);
        per = per >= HS_ITER ? (per + HS_ITER - 1) / HS_ITER * HS_ITER : (per + 3) / 4 * 4;
        if (per < HS_CHUNK_MIN) per = HS_CHUNK_MIN;
        if (per > HS_CHUNK_MAX) per = HS_CHUNK_MAX;
        P.chunk = (int)per;
        h.grid = n > 0 ? (int)((n + per - 1) / per) : 0;
        h.variant = 16 | (aligned(it.d_x, 16) ? 1 : 0) | (h.f.l1 ? 8 : 0);
    } else {
        P.hs_s = 16;
        P.hs_eb_lo = 0;
        P.hs_w = 0;
    }
    return FXPQ_OK;
}

void fs_bins_launch(int variant, int grid, const FsBatch& B, int i0, int i1, cudaStream_t s) {
    if (variant & 16) {
        const size_t hb = HS_SMEM;
        const bool vec = variant & 1, l1 = variant & 8;
        if (vec && !l1)
            fl_search_hist_kernel<true, false><<<grid, HS_T, hb, s>>>(B, i0, i1);
        else if (!l1)
            fl_search_hist_kernel<false, false><<<grid, HS_T, hb, s>>>(B, i0, i1);
        else if (vec)
            fl_search_hist_kernel<true, true><<<grid, HS_T, hb, s>>>(B, i0, i1);
        else
            fl_search_hist_kernel<false, true><<<grid, HS_T, hb, s>>>(B, i0, i1);
        return;
    }
    const size_t sb = sizeof(FsSmem);
    const bool vec = variant & 1, small = variant & 2, narrow = variant & 4, l1 = variant & 8;
#define FXPQ_FS_LAUNCH(V, L1)                                                            \
    if (narrow && small)                                                                 \
        fl_search_bins_kernel<V, 10, 2, L1><<<grid, FS_THREADS, sb, s>>>(B, i0, i1);     \
    else if (narrow)                                                                     \
        fl_search_bins_kernel<V, NJ, 2, L1><<<grid, FS_THREADS, sb, s>>>(B, i0, i1);     \
    else                                                                                 \
        fl_search_bins_kernel<V, NJ, NJ, L1><<<grid, FS_THREADS, sb, s>>>(B, i0, i1);
    if (vec && !l1) {
        FXPQ_FS_LAUNCH(true, false)
    } else if (!l1) {
        FXPQ_FS_LAUNCH(false, false)
    } else if (vec) {
        FXPQ_FS_LAUNCH(true, true)
    } else {
        FXPQ_FS_LAUNCH(false, true)
    }
#undef FXPQ_FS_LAUNCH
}

// Runs up to FS_MAX_ITEMS prepared searches whose bins live at g[0..n): one clear, one bins launch
// per run of items sharing a kernel instance (items are ordered by instance), one cells launch, one
// select launch.
fxpq_status fs_run(FsItemHost* h, int n, FsGlobal* g, cudaStream_t s) {
    if (n == 0) return FXPQ_OK;
    if (cudaMemsetAsync(g, 0, kFsGlobalBytes * n, s) != cudaSuccess) return FXPQ_ERR_CUDA;
    // order by kernel instance, each item keeping its own bins; within an instance the items with the
    // largest chunk per block come first, so that their long blocks start in the first wave and the
    // many short blocks of small items fill in behind them (longest-first scheduling of one launch)
    int order[FS_MAX_ITEMS];
    int m = 0;
    for (int v = 0; v < 32; ++v) {
        const int m0 = m;
        for (int i = 0; i < n; ++i)
            if (h[i].variant == v) order[m++] = i;
        std::stable_sort(order + m0, order + m, [&](int x, int y) {
            const long long wx = h[x].grid > 0 ? (h[x].p.n + h[x].grid - 1) / h[x].grid : 0;
            const long long wy = h[y].grid > 0 ? (h[y].p.n + h[y].grid - 1) / h[y].grid : 0;
            return wx > wy;
        });
    }
    FsBatch B;
    FsOutBatch O;
    B.n_items = n;
    int cells = 0, fblocks = 0;
    for (int j = 0; j < n; ++j) {
        const FsItemHost& it = h[order[j]];
        B.p[j] = it.p;
        B.p[j].g = reinterpret_cast<FsGlobal*>(reinterpret_cast<char*>(g) + kFsGlobalBytes * order[j]);
        B.f[j] = it.f;
        O.o[j] = it.o;
        B.cell0[j] = cells;
        B.fin0[j] = fblocks;
        const int nc = (it.f.S_hi - it.f.S_lo + 1) * it.f.nk * it.f.nfl + 2;
        cells += nc;
        fblocks += (nc + FIN_WARPS - 1) / FIN_WARPS;  // one finalize warp per cell
    }
    B.cell0[n] = cells;
    B.fin0[n] = fblocks;
    st_attr_once();
    for (int j0 = 0; j0 < n;) {
        const int v = h[order[j0]].variant;
        int j1 = j0, blocks = 0;
        while (j1 < n && h[order[j1]].variant == v) {
            B.blk0[j1] = blocks;  // relative to this launch
            blocks += h[order[j1]].grid;
            ++j1;
        }
        B.blk0[j1] = blocks;
        if (blocks > 0) {
            fs_bins_launch(v, blocks, B, j0, j1, s);
            const fxpq_status st = after_launch("fl_search_bins");
            if (st != FXPQ_OK) return st;
        }
        j0 = j1;
    }
    fl_search_final_kernel<<<fblocks, FIN_T, 0, s>>>(B, O, status_ptr());
    return after_launch("fl_search_final");
}
}  // namespace

extern "C" size_t fxpq_fl_search_workspace(int64_t n) {
    (void)n;
    return kFsGlobalBytes;
}

extern "C" fxpq_status fxpq_fl_search(const float* d_x, int64_t n, int32_t is_signed, int32_t k_lo, int32_t k_hi,
                                      int32_t fl_lo, int32_t fl_hi, double* d_err, int32_t* d_best,
                                      fxpq_stats* d_stats, void* d_ws, size_t ws_bytes, void* stream) {
    const fxpq_fl_search_item it = {d_x, n, is_signed, k_lo, k_hi, fl_lo, fl_hi, d_err, d_best, d_stats, FXPQ_SCORE_L2};
    FsItemHost h;
    const fxpq_status st = fs_prepare(it, static_cast<FsGlobal*>(d_ws), h);
    if (st != FXPQ_OK) return st;
    if (!d_ws || ws_bytes < fxpq_fl_search_workspace(n) || !aligned(d_ws, 256)) return FXPQ_ERR_WORKSPACE;
    return fs_run(&h, 1, static_cast<FsGlobal*>(d_ws), as_stream(stream));
}

extern "C" size_t fxpq_fl_search_batch_workspace(int32_t n_items) {
    return n_items > 0 ? kFsGlobalBytes * (size_t)n_items : 0;
}

extern "C" fxpq_status fxpq_fl_search_batch(const fxpq_fl_search_item* h_items, int32_t n_items, void* d_ws,
                                            size_t ws_bytes, void* stream) {
    if (n_items < 0 || (n_items > 0 && !h_items)) return FXPQ_ERR_INVALID_ARG;
    if (n_items == 0) return FXPQ_OK;
    if (!d_ws || ws_bytes < fxpq_fl_search_batch_workspace(n_items) || !aligned(d_ws, 256))
        return FXPQ_ERR_WORKSPACE;
    FsItemHost h[FS_MAX_ITEMS];
    FsGlobal* g = static_cast<FsGlobal*>(d_ws);
    // validate everything before the first launch
    for (int i = 0; i < n_items; ++i) {
        FsItemHost tmp;
        const fxpq_status st = fs_prepare(h_items[i], g, tmp);
        if (st != FXPQ_OK) return st;
    }
    cudaStream_t s = as_stream(stream);
    for (int i0 = 0; i0 < n_items; i0 += FS_MAX_ITEMS) {
        const int m = n_items - i0 < FS_MAX_ITEMS ? n_items - i0 : FS_MAX_ITEMS;
        FsGlobal* gi = reinterpret_cast<FsGlobal*>(reinterpret_cast<char*>(g) + kFsGlobalBytes * i0);
        for (int i = 0; i < m; ++i) fs_prepare(h_items[i0 + i], gi, h[i]);
        const fxpq_status st = fs_run(h, m, gi, s);
        if (st != FXPQ_OK) return st;
    }
    return FXPQ_OK;
}

extern "C" fxpq_status fxpq_fl_init(const fxpq_stats* h_stats, int32_t bits, int32_t strategy, fxpq_fmt* h_out) {
    if (!h_stats || !h_out || bits < 2 || bits > 32 || strategy < 0 || strategy > 2) return FXPQ_ERR_INVALID_ARG;
    const double mn = h_stats->min, mx = h_stats->max;
    const int S = mn < 0.0 ? 1 : 0;
    double psi = 0.0;
    if (S == 0) {
        psi = mx / (ldexp(1.0, bits) - 1.0);
    } else {
        const double a = mn / -ldexp(1.0, bits - 1), b = mx / (ldexp(1.0, bits - 1) - 1.0);
        psi = (a > 0 && b > 0) ? fmin(a, b) : (a > 0 ? a : b);
    }
    if (!(psi > 0.0) || !isfinite(psi)) return FXPQ_ERR_INVALID_ARG;
    const double bh = -log2(psi);
    const double beta = strategy == 0 ? floor(bh) : (strategy == 1 ? nearbyint(bh) : ceil(bh));
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
    if (k_lo < 1 || k_hi > 16 || k_lo > k_hi || fl_lo > fl_hi || fl_hi - fl_lo + 1 > MAXFL)
        return FXPQ_ERR_INVALID_ARG;  // the largest candidate grid the array holds: 16 x 32 (k in [1, 16])
    if (fxpq_fl_search_workspace(n) > kFlSearchStaticBytes) return FXPQ_ERR_WORKSPACE;
    void* scratch = nullptr;
    const fxpq_status st = fl_search_scratch_ptr(&scratch);
    if (st != FXPQ_OK) return st;
    // fxpq_fl_search clears the bins it accumulates into before its first kernel.
    return fxpq_fl_search(d_x, n, is_signed, k_lo, k_hi, fl_lo, fl_hi, d_err, d_best, d_stats, scratch,
                          kFlSearchStaticBytes, stream);
}
