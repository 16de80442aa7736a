// fxpq_flsearch_hist.cuh -- FL search by a moment histogram of the fp32 bit patterns (Sec. IV-C,
// Eq. DSB_QE and Eq. MAE).  Included by fxpq_flsearch.cu after the workspace types; it fills the
// same exact per-key workspace bins (counts, moments, remainder sums) as the sorting kernel there,
// so the same cells and select kernels finish both.
//
// Scope: searches whose remainder slots all lie at j <= 7 (k <= 8 when the sign strategy may pick
// unsigned codes, k <= 9 for signed ones) -- every per-layer search of the networks' weights and
// activations.  Wider ranges (the 9..16-bit rows) keep the sorting kernel.
//
// The algebra.  Write an element's significand M = Hf 2^s + L with L < 2^s and s in {15, 16}
// chosen so that every needed slot j has its rounding bit (bit 22 - j of M) in Hf (s <= 22 - j).
// At slot j (p = 23 - j bits below y's binary point) the rounding error's magnitude is
//     r = A 2^s + L_b,   L_b = L if b = 0, 2^s - L if b = 1,
// where b is the rounding bit and A the bits of Hf below it (complemented when b = 1); both depend
// on Hf alone.  Hence over the elements of one bin (sign, exponent E, h = Hf - 2^(23-s)):
//     sum r^2 = 2^(2s) (A^2 + b) n + 2^(s+1) (A sum L_b - b sum L) + sum L^2,
//     sum r   = 2^s A n + sum L_b,
// with n the bin's count and sum L_b = b (n 2^s) + (1 - 2b) sum L.  The boundary slot (saturation
// at T = 2^t - 1, Sec. IV-B clip) saturates exactly the bins whose top t bits of Hf are all ones,
// where the error M - thr has the same form with A = Hf - thr 2^-s and b = 0.  The moments
// (sum M, sum M^2) are the same kind of polynomial in (Hf, n, sum L).  So the per-element work is
// two 32-bit shared-memory reductions into the element's bin.
//
// sum L^2 enters every class of every candidate of the L2 score with coefficient one (rounding,
// boundary, saturation, rounding to zero), so only its total over the window's keys, weighted by
// u_E^2 = 2^(2(E-23)), is needed: elements whose exponent lies in a band of up to 16 exponents
// inside the window, chosen per block, accumulate (L 2^e)^2 (e = E - band mod 8) exactly in two
// per-lane 64-bit registers, whose block sums go to the exponent-indexed workspace bins `cband`
// (added to every L2 cell and to the sum of squares by the cells kernel).  Window elements outside
// the band add L^2, as two 16-bit halves, to per-key shared bins striped over 16 lanes, which are
// folded into their key's sums.
//
// Keys outside the window (saturated for every candidate FL, or rounded to zero for every one) and
// subnormals need only their moments: they go straight to the workspace by global atomics, and
// non-finite values set the flag.  In the hot loop every element outside the window, zeros
// included, lands in a per-lane scratch bin; the rare ones that need more (outside the band, or
// outside the window and not zero) are handled after each group of 16 in a separate pass over the
// same registers.  Zeros are the scratch count less those.
//
// After its chunk each block converts its bins, one key per warp: the moments, then the remainder
// sums level by level from the coarsest rounding bit down, the bins folded over their top bit
// between levels (level pb holds g = Hf mod 2^pb, enough for slot j = 23 - s - pb).

namespace fxpq {
namespace {

constexpr int HS_T = 1024;                 // threads per block (one block per SM)
constexpr int HS_ITER = 16 * HS_T;         // elements per block iteration (four float4 per thread)
constexpr int HS_CHUNK_MAX = 1 << 20;      // per-block elements: keeps stripe sums below 2^32
constexpr int HS_CHUNK_MIN = 4 * HS_T;  // at least one float4 per thread
constexpr int HS_STRIPE = 16;              // per-key L^2 bins, by lane % 16
constexpr unsigned HS_CNT_LIMIT = 65536u;  // a bin this full may have wrapped its 32-bit sum of L
constexpr int HS_OVF_MAX = HS_CHUNK_MAX / (int)HS_CNT_LIMIT;
constexpr int HS_MAX_W = 40;               // window keys per sign (j <= 7 and 32 FLs)
constexpr int HS_MAX_BINS = 2 * HS_MAX_W * 256;

// Shared-memory layout in words, fixed so that a bin's sum of L sits a constant distance from its
// count: counts (HS_MAX_BINS + 32 scratch), sums of L (the same), L^2 stripes, misc.
constexpr int HS_O_SL = HS_MAX_BINS + 32;
constexpr int HS_O_L2LO = 2 * HS_O_SL;
constexpr int HS_O_L2HI = HS_O_L2LO + 2 * HS_MAX_W * HS_STRIPE;
constexpr int HS_O_MISC = HS_O_L2HI + 2 * HS_MAX_W * HS_STRIPE;
constexpr int HM_WSUM = 64;  // the warps' band sums (2 x 32 u64)
constexpr int HS_MISC = HM_WSUM + 4 * (HS_T / 32);  // band, min, max, counters, overflow list and its 64-bit sums
constexpr size_t HS_SMEM = (size_t)(HS_O_MISC + HS_MISC) * 4u;
static_assert(HS_O_MISC % 2 == 0, "misc holds 64-bit sums");
constexpr int HM_BAND = 0, HM_MN = 1, HM_MX = 2, HM_NOVF = 3, HM_COLD = 4, HM_NF = 5, HM_OVF_IDX = 8,
              HM_OVF_SUM = 24;  // 16 x u64

struct HsLayout {
    int nH, nbins, nkeys;
};

__host__ __device__ inline HsLayout hs_layout(const FsParams& P) {
    HsLayout y;
    y.nH = 1 << (23 - P.hs_s);
    y.nkeys = 2 * P.hs_w;
    y.nbins = y.nkeys * y.nH;
    return y;
}

__host__ __device__ inline bool hs_fits(const FsParams& P) { return P.hs_w <= HS_MAX_W && P.hs_s >= 15; }

struct HsLane {
    u64 acc0, acc1;   // sum (L 2^e)^2 for E - band in [0, 8) (e = E - band) and [8, 16) (e = E - band - 8)
    unsigned mn, mx;  // order keys (non-finite values are corrected for after the chunk)
};

// Per-item constants of the hot loop.
struct HsK {
    unsigned s1;       // split bit + 1 (the bin index is taken from u << 1)
    unsigned lmask;    // 2^s - 1
    unsigned eblo24;   // lowest window biased exponent << 24
    unsigned w24;      // window keys per sign << 24
    unsigned noff;     // first bin of the negative keys: w 2^(23-s)
    unsigned scratch;  // this lane's scratch bin
    unsigned band24;   // band's lowest biased exponent << 24
    unsigned lim0, lim1;  // band exponents accumulated in acc0 (e < lim0) and acc1 (e - 8 < lim1)
    unsigned span;     // lim0 + lim1
};

// One element of the hot loop: its bin's count and sum of L (a scratch bin outside the window), its
// share of sum L^2 u_E^2 when its exponent is in the band, the stats.  Returns true when the element
// needs the cold pass (window element outside the band, or a non-zero element outside the window).
__device__ __forceinline__ bool hs_elem(unsigned u, unsigned* cnt, const HsK& K, HsLane& st) {
    const unsigned z = u << 1;              // (eb, mantissa, 0)
    const unsigned zw = z - K.eblo24;       // window slot d in the top byte
    const bool in = zw < K.w24;
    const unsigned sgm = (unsigned)((int)u >> 31);
    // zw >> (s + 1) = d 2^(23-s) + h; negative keys follow the w positive ones
    const unsigned idx = in ? (zw >> K.s1) + (sgm & K.noff) : K.scratch;
    const unsigned L = u & K.lmask;
    atomicAdd(&cnt[idx], 1u);
    atomicAdd(&cnt[idx + HS_O_SL], L);
    const unsigned eo = (z - K.band24) >> 24;  // E - band (large when below the band)
    const unsigned Le = L << (eo & 7u);        // < 2^23
    // branch-free: the operand is zeroed outside each half of the band
    const unsigned L0 = eo < K.lim0 ? Le : 0u;
    const unsigned L1 = eo - 8u < K.lim1 ? Le : 0u;
    st.acc0 += (u64)L0 * L0;
    st.acc1 += (u64)L1 * L1;
    const unsigned ok = u ^ (sgm | 0x80000000u);
    st.mn = min(st.mn, ok);
    st.mx = max(st.mx, ok);
    return eo >= K.span && z != 0u;  // the band lies inside the window
}

// The cold pass of one element (see hs_elem): L^2 of a window element outside the band into its
// key's stripe; exact moments of a key outside the window (or a subnormal) into the workspace; the
// flag for a non-finite value.  Returns 1 for a non-zero element that took a scratch bin.
__device__ __noinline__ unsigned hs_cold(unsigned u, const HsK& K, unsigned* smem, FsGlobal* g, unsigned lane) {
    const unsigned z = u << 1;
    const unsigned eo = (z - K.band24) >> 24;
    if (eo < K.span || z == 0u) return 0u;
    const unsigned zw = z - K.eblo24;
    if (zw < K.w24) {
        const unsigned L = u & K.lmask;
        const unsigned q = L * L;  // < 2^32
        const unsigned ks = (zw >> 24) + (((unsigned)((int)u >> 31)) & (K.w24 >> 24));
        const unsigned c = ks * HS_STRIPE + (lane & (HS_STRIPE - 1));
        atomicAdd(&smem[HS_O_L2LO + c], q & 0xFFFFu);
        atomicAdd(&smem[HS_O_L2HI + c], q >> 16);
        return 0u;
    }
    const unsigned eb = z >> 24;
    if (eb == 0xFFu) {
        smem[HS_O_MISC + HM_NF] = 1u;
        atomicOr(&g->nonfinite, 1u);
        return 1u;
    }
    const unsigned mant = u & 0x7FFFFFu;
    const u64 M = eb ? (mant | 0x800000u) : mant;
    const unsigned key = u >> 23;
    atomicAdd(&g->pn[key], 1ull);
    gaddL(g->ps1[key], M);
    gaddL(g->ps2[key], M * M);
    return 1u;
}

// Bin of a window element, or -1 (for the overflow recount).
__device__ __forceinline__ int hs_bin(unsigned u, const HsK& K, unsigned& L) {
    const unsigned zw = (u << 1) - K.eblo24;
    if (zw >= K.w24) return -1;
    L = u & K.lmask;
    return (int)((zw >> K.s1) + (((unsigned)((int)u >> 31)) & K.noff));
}

// Warp sum of per-lane values below 2^52, as two 26-bit pieces (each piece sum stays below 2^31).
__device__ __forceinline__ u64 hs_wsum52(u64 v) {
    const unsigned lo = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v & 0x3FFFFFFull));
    const unsigned hi = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v >> 26));
    return (u64)lo + ((u64)hi << 26);
}
// Warp sum of per-lane values below 2^63 (three 21-bit pieces), exact in 128 bits.
__device__ __forceinline__ unsigned __int128 hs_wsum128(u64 v) {
    const unsigned a = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v & 0x1FFFFFull));
    const unsigned b = __reduce_add_sync(0xFFFFFFFFu, (unsigned)((v >> 21) & 0x1FFFFFull));
    const unsigned c = __reduce_add_sync(0xFFFFFFFFu, (unsigned)(v >> 42));
    return (unsigned __int128)a + ((unsigned __int128)b << 21) + ((unsigned __int128)c << 42);
}
// ... of signed per-lane values with |v| < 2^45.
__device__ __forceinline__ long long hs_wsum_s(long long v) {
    return (long long)hs_wsum52((u64)(v + (1ll << 45))) - (1ll << 50);
}

// In-range rounding (b, A) of the level-pb value g = Hf mod 2^pb.
__device__ __forceinline__ void hs_round(unsigned g, int pb, unsigned& A, unsigned& b) {
    const unsigned m = (1u << (pb - 1)) - 1u;
    b = (g >> (pb - 1)) & 1u;
    A = (g & m) ^ (b ? m : 0u);
}

// Accumulate one level entry (n, sum L) with rounding (A, b) into the slot sums.
template <bool L1>
__device__ __forceinline__ void hs_term(u64& X, long long& Y, unsigned A, unsigned b, unsigned n, u64 sL, int s) {
    const u64 nS = (u64)n << s;
    const u64 Lb = b ? nS - sL : sL;
    if constexpr (L1) {
        X += (u64)A * n;
        Y += (long long)Lb;
    } else {
        X += ((u64)A * A + b) * n;
        Y += (long long)((u64)A * Lb) - (b ? (long long)sL : 0ll);
    }
}

// One warp converts window key ks of the block's bins (split bit s = 23 - HB) into the workspace.
// Every level's total ends up in one lane (lane 0: sum M, 1: sum M^2, 2 + level: the remainder sum,
// 12 + j: the boundary sum of slot j), and the lanes add them to the workspace together.
template <bool L1, int HB>
__device__ void hs_convert_key(const FsParams& P, const unsigned* smem, const u64* ovf_sum, const unsigned* ovf_idx,
                               unsigned novf, int ks, unsigned lane) {
    constexpr int s = 23 - HB;
    constexpr int nH = 1 << HB;
    constexpr int NE = nH >> 5;  // entries per lane at level HB
    const unsigned* cnt = smem;
    const unsigned* slb = smem + HS_O_SL;
    const int sg = ks >= P.hs_w ? 1 : 0;
    const int E = P.hs_eb_lo + ks - sg * P.hs_w - 127;
    const int key = sg * 256 + E + 127;
    const int base = ks * nH;
    unsigned n[NE];
    u64 sl[NE];
    unsigned nl = 0;
#pragma unroll
    for (int i = 0; i < NE; ++i) {
        const int b = base + (int)lane + 32 * i;
        n[i] = cnt[b];
        sl[i] = slb[b];
        if (n[i] >= HS_CNT_LIMIT)
            for (unsigned q = 0; q < novf; ++q)
                if (ovf_idx[q] == (unsigned)b) sl[i] = ovf_sum[q];
        nl += n[i];
    }
    const unsigned ntot = __reduce_add_sync(0xFFFFFFFFu, nl);
    if (ntot == 0u) return;
    // sum of L^2 of this key's elements outside the block's band
    u64 l2 = 0ull;
    if (lane < (unsigned)HS_STRIPE) {
        const int c = ks * HS_STRIPE + (int)lane;
        l2 = (u64)smem[HS_O_L2LO + c] + ((u64)smem[HS_O_L2HI + c] << 16);
    }
    l2 = hs_wsum52(l2);
    u64* dst = nullptr;
    __int128 val = 0;
    {
        u64 s1h = 0, slt = 0, s2a = 0, s2b = 0;
#pragma unroll
        for (int i = 0; i < NE; ++i) {
            const u64 hf = (u64)(nH + (int)lane + 32 * i);
            s1h += hf * n[i];
            slt += sl[i];
            s2a += hf * hf * n[i];
            s2b += hf * sl[i];
        }
        s1h = hs_wsum52(s1h);
        slt = hs_wsum52(slt);
        s2a = hs_wsum52(s2a);
        s2b = hs_wsum52(s2b);
        if (lane == 0) {
            atomicAdd(&P.g->pn[key], (u64)ntot);
            dst = P.g->ps1[key];
            val = ((__int128)s1h << s) + (__int128)slt;
        } else if (lane == 1) {
            dst = P.g->ps2[key];
            val = ((__int128)s2a << (2 * s)) + ((__int128)s2b << (s + 1)) + (__int128)l2;
        }
    }
    // live slots of this key: j = E + FL for FL in range, within the needed slots
    const int cand_lo = E + P.fl_lo, cand_hi = E + P.fl_lo + P.nfl - 1;
    const int jmax = sg ? P.jmax_neg : P.jmax_pos;
    const int jlo = max(-1, cand_lo), jhi = min(jmax, cand_hi);
    const int jblo = sg ? 1 : max(max(P.jb_lo, 0), cand_lo), jbhi = sg ? 0 : min(P.jb_hi, cand_hi);
    constexpr int pa = L1 ? s : 2 * s, pbw = L1 ? 0 : s + 1;
    const __int128 z = L1 ? 0 : (__int128)l2;
    // levels pb = HB + 1 (slot j = -1) down to 1 (slot j = 22 - s)
#pragma unroll
    for (int lv = 0; lv <= HB; ++lv) {
        const int pb = HB + 1 - lv;
        const int j = 23 - s - pb;
        const bool live = j >= jlo && j <= jhi;
        const bool blive = lv > 0 && j >= jblo && j <= jbhi;  // boundary slots have j >= 0
        if (live || blive) {
            u64 X = 0;
            long long Y = 0;
            if (lv == 0) {
                // g = Hf = 2^HB + h: the rounding bit is the implicit one, A = 2^HB - 1 - h
#pragma unroll
                for (int i = 0; i < NE; ++i) hs_term<L1>(X, Y, (unsigned)(nH - 1 - ((int)lane + 32 * i)), 1u, n[i], sl[i], s);
            } else if (pb >= 6) {
                // entry i holds g = lane + 32 i: its rounding bit (bit pb - 1 >= 5) is bit pb - 6 of i
#pragma unroll
                for (int i = 0; i < ((1 << pb) >> 5); ++i) {
                    const unsigned b = ((unsigned)i >> (pb - 6)) & 1u;
                    const unsigned m = (1u << (pb - 1)) - 1u;
                    const unsigned A = ((lane + 32u * i) & m) ^ (b ? m : 0u);
                    hs_term<L1>(X, Y, A, b, n[i], sl[i], s);
                }
            } else if (pb == 5) {
                unsigned A, b;
                hs_round(lane, pb, A, b);
                hs_term<L1>(X, Y, A, b, n[0], sl[0], s);
            } else if (lane < (1u << pb)) {
                unsigned A, b;
                hs_round(lane, pb, A, b);
                hs_term<L1>(X, Y, A, b, n[0], sl[0], s);
            }
            if (blive) {
                // the bins whose top (HB + 1 - pb) bits of Hf are all ones saturate: h in
                // [nH - 2^pb, nH), with Hf - thr 2^-s = g; their in-range terms give way to saturated ones
                u64 Xd = 0;
                long long Yd = 0;
                for (int g = (int)lane; g < (1 << pb); g += 32) {
                    const int b0 = base + nH - (1 << pb) + g;
                    const unsigned nn = cnt[b0];
                    u64 ss = slb[b0];
                    if (nn >= HS_CNT_LIMIT)
                        for (unsigned q = 0; q < novf; ++q)
                            if (ovf_idx[q] == (unsigned)b0) ss = ovf_sum[q];
                    u64 Xi = 0, Xs = 0;
                    long long Yi = 0, Ys = 0;
                    unsigned A, b;
                    hs_round((unsigned)g, pb, A, b);
                    hs_term<L1>(Xi, Yi, A, b, nn, ss, s);
                    hs_term<L1>(Xs, Ys, (unsigned)g, 0u, nn, ss, s);
                    Xd += Xs - Xi;
                    Yd += Ys - Yi;
                }
                const u64 Xb = hs_wsum52(X + Xd);  // every lane's X + Xd >= 0
                const long long Yb = hs_wsum_s(Y + Yd);
                if (lane == 12u + (unsigned)j) {
                    dst = P.g->rb[j + 1][j - cand_lo];
                    val = ((__int128)Xb << pa) + ((__int128)Yb << pbw) + z;
                }
            }
            if (live) {
                const u64 Xt = hs_wsum52(X);
                const long long Yt = hs_wsum_s(Y);
                if (lane == 2u + (unsigned)lv) {
                    dst = P.g->r[sg][j + 1][j - cand_lo];
                    val = ((__int128)Xt << pa) + ((__int128)Yt << pbw) + z;
                }
            }
        }
        // fold to level pb - 1 (levels HB + 1 and HB share the entries)
        if (lv > 0 && pb >= 2) {
            if (pb > 5) {
                const int half = (1 << pb) >> 6;
#pragma unroll
                for (int i = 0; i < NE / 2; ++i) {
                    if (i < half) {
                        n[i] += n[i + half];
                        sl[i] += sl[i + half];
                    }
                }
            } else {
                const unsigned o = 1u << (pb - 1);
                n[0] += __shfl_down_sync(0xFFFFFFFFu, n[0], o);
                sl[0] += __shfl_down_sync(0xFFFFFFFFu, sl[0], o);
            }
        }
    }
    if (dst) gaddLs(dst, val);
}

template <bool VEC>
__device__ __forceinline__ void hs_load4(const float* __restrict__ x, long long i0, uint4 (&d)[4]) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const long long i = i0 + 4LL * HS_T * q;
        if (VEC) {
            d[q] = __ldg(reinterpret_cast<const uint4*>(x + i));
        } else {
            d[q].x = __float_as_uint(__ldg(x + i));
            d[q].y = __float_as_uint(__ldg(x + i + 1));
            d[q].z = __float_as_uint(__ldg(x + i + 2));
            d[q].w = __float_as_uint(__ldg(x + i + 3));
        }
    }
}

// The same slots as hs_load4 for the block's last, partial iteration: the elements below `end`
// (bit 4 q + c of the returned mask), zeros elsewhere.
template <bool VEC>
__device__ __forceinline__ unsigned hs_load4p(const float* __restrict__ x, long long i0, long long end,
                                              uint4 (&d)[4]) {
    unsigned m = 0u;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const long long i = i0 + 4LL * HS_T * q;
        d[q] = make_uint4(0u, 0u, 0u, 0u);
        if (VEC && i + 4 <= end) {
            d[q] = __ldg(reinterpret_cast<const uint4*>(x + i));
            m |= 0xFu << (4 * q);
        } else {
            if (i < end) d[q].x = __float_as_uint(__ldg(x + i)), m |= 1u << (4 * q);
            if (i + 1 < end) d[q].y = __float_as_uint(__ldg(x + i + 1)), m |= 2u << (4 * q);
            if (i + 2 < end) d[q].z = __float_as_uint(__ldg(x + i + 2)), m |= 4u << (4 * q);
            if (i + 3 < end) d[q].w = __float_as_uint(__ldg(x + i + 3)), m |= 8u << (4 * q);
        }
    }
    return m;
}

template <bool VEC, bool L1>
__global__ void __launch_bounds__(HS_T, 1) fl_search_hist_kernel(const __grid_constant__ FsBatch B, int item0, int item1) {
    const int item = item0 + batch_item(B.blk0 + item0, item1 - item0, (int)blockIdx.x);
    const FsParams& P = B.p[item];
    const int blk = (int)blockIdx.x - B.blk0[item];
    extern __shared__ __align__(16) unsigned hs_smem[];
    unsigned* misc = hs_smem + HS_O_MISC;
    u64* ovf_sum = reinterpret_cast<u64*>(misc + HM_OVF_SUM);
    u64* wsum = reinterpret_cast<u64*>(misc + HM_WSUM);
    const unsigned tid = threadIdx.x, lane = tid & 31u, warp = tid >> 5;
    FsGlobal* g = P.g;
    const HsLayout Ly = hs_layout(P);

    {
        uint4* z4 = reinterpret_cast<uint4*>(hs_smem);
        for (int i = (int)tid; i < HS_O_MISC / 4; i += HS_T) z4[i] = make_uint4(0u, 0u, 0u, 0u);
        if (tid < (unsigned)HS_MISC) misc[tid] = tid == HM_MN ? 0xFFFFFFFFu : 0u;
    }
    __syncthreads();

    HsK K;
    K.s1 = (unsigned)P.hs_s + 1u;
    K.lmask = (1u << P.hs_s) - 1u;
    K.eblo24 = (unsigned)P.hs_eb_lo << 24;
    K.w24 = (unsigned)P.hs_w << 24;
    K.noff = (unsigned)P.hs_w << (23 - P.hs_s);
    K.scratch = (unsigned)HS_MAX_BINS + lane;

    const long long start = (long long)blk * P.chunk;
    const long long end = min(start + (long long)P.chunk, P.n);
    // whole iterations, then at most one partial one
    const long long nit = end > start ? (end - start + HS_ITER - 1) / HS_ITER : 0;
    const long long nfull = end > start ? (end - start) / HS_ITER : 0;
    HsLane st;
    st.acc0 = st.acc1 = 0ull;
    st.mn = 0xFFFFFFFFu;
    st.mx = 0u;
    unsigned nout = 0u;

    uint4 va[4], vb[4];
    unsigned ma = 0xFFFFu;  // valid elements of the first iteration
    const long long t0 = start + 4LL * tid;
    if (nfull > 0)
        hs_load4<VEC>(P.x, t0, va);
    else
        ma = nit > 0 ? hs_load4p<VEC>(P.x, t0, end, va) : 0u;
    // the block's band: up to 16 exponents of the window ending at the largest window exponent of its
    // first iteration
    {
        unsigned m = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const unsigned w4[4] = {va[q].x, va[q].y, va[q].z, va[q].w};
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const unsigned zw = (w4[c] << 1) - K.eblo24;
                if (((ma >> (4 * q + c)) & 1u) && zw < K.w24) m = max(m, (w4[c] >> 23) & 0xFFu);
            }
        }
        m = __reduce_max_sync(0xFFFFFFFFu, m);
        if (lane == 0 && m) atomicMax(&misc[HM_BAND], m);
    }
    __syncthreads();
    const unsigned span = (unsigned)min(16, P.hs_w);
    const unsigned eb_lo = (unsigned)P.hs_eb_lo;
    unsigned band = misc[HM_BAND] ? misc[HM_BAND] + 1u - span : eb_lo;
    band = max(band, eb_lo);  // inside the window: [band, band + span) within [eb_lo, eb_lo + w)
    K.band24 = band << 24;
    K.lim0 = min(8u, span);
    K.lim1 = span - K.lim0;
    K.span = span;

    // One group of 16 elements as a single basic block; the rare ones that need the cold pass are
    // marked in a mask and handled after the group, each at a compile-time register index.
    auto cold = [&](const uint4 (&v)[4], unsigned cm) {
        if (cm) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (cm & (1u << (4 * q))) nout += hs_cold(v[q].x, K, hs_smem, g, lane);
                if (cm & (2u << (4 * q))) nout += hs_cold(v[q].y, K, hs_smem, g, lane);
                if (cm & (4u << (4 * q))) nout += hs_cold(v[q].z, K, hs_smem, g, lane);
                if (cm & (8u << (4 * q))) nout += hs_cold(v[q].w, K, hs_smem, g, lane);
            }
        }
    };
    auto body = [&](const uint4 (&v)[4]) {
        unsigned cm = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            cm |= hs_elem(v[q].x, hs_smem, K, st) ? 1u << (4 * q) : 0u;
            cm |= hs_elem(v[q].y, hs_smem, K, st) ? 2u << (4 * q) : 0u;
            cm |= hs_elem(v[q].z, hs_smem, K, st) ? 4u << (4 * q) : 0u;
            cm |= hs_elem(v[q].w, hs_smem, K, st) ? 8u << (4 * q) : 0u;
        }
        cold(v, cm);
    };
    // two buffers in rotation: one iteration of loads in flight (1024 threads x 64 B per SM) while the
    // other is binned
    for (long long it = 0; it < nfull; it += 2) {
        if (it + 1 < nfull) hs_load4<VEC>(P.x, t0 + (it + 1) * HS_ITER, vb);
        body(va);
        if (it + 1 >= nfull) break;
        if (it + 2 < nfull) hs_load4<VEC>(P.x, t0 + (it + 2) * HS_ITER, va);
        body(vb);
    }
    // the partial iteration (the only one of a chunk below HS_ITER elements): its valid elements
    if (nit > nfull) {
        if (nfull > 0) ma = hs_load4p<VEC>(P.x, t0 + nfull * HS_ITER, end, va);
        unsigned cm = 0u;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if ((ma >> (4 * q)) & 1u) cm |= hs_elem(va[q].x, hs_smem, K, st) ? 1u << (4 * q) : 0u;
            if ((ma >> (4 * q)) & 2u) cm |= hs_elem(va[q].y, hs_smem, K, st) ? 2u << (4 * q) : 0u;
            if ((ma >> (4 * q)) & 4u) cm |= hs_elem(va[q].z, hs_smem, K, st) ? 4u << (4 * q) : 0u;
            if ((ma >> (4 * q)) & 8u) cm |= hs_elem(va[q].w, hs_smem, K, st) ? 8u << (4 * q) : 0u;
        }
        cold(va, cm);
    }

    // per-lane results: stats, band sums, elements outside the window that were not zeros
    {
        const unsigned mn = __reduce_min_sync(0xFFFFFFFFu, st.mn), mx = __reduce_max_sync(0xFFFFFFFFu, st.mx);
        const unsigned no = __reduce_add_sync(0xFFFFFFFFu, nout);
        const u64 a0 = warp_sum64(st.acc0), a1 = warp_sum64(st.acc1);  // < 2^61 per warp
        if (lane == 0) {
            atomicMin(&misc[HM_MN], mn);
            atomicMax(&misc[HM_MX], mx);
            if (no) atomicAdd(&misc[HM_COLD], no);
            wsum[warp] = a0;
            wsum[HS_T / 32 + warp] = a1;
        }
    }
    __syncthreads();
    if (warp == 0) {  // the block's band sums (< 2^66), one workspace add each
        const unsigned __int128 b0 = hs_wsum128(wsum[lane]), b1 = hs_wsum128(wsum[HS_T / 32 + lane]);
        if (lane == 0) {
            gaddLs(g->cband[band], (__int128)b0);
            gaddLs(g->cband[band + 8u], (__int128)b1);
        }
    }
    if (misc[HM_NF]) {
        // a non-finite value reached the order keys: take min and max again over the finite ones
        __syncthreads();
        if (tid == 0) {
            misc[HM_MN] = 0xFFFFFFFFu;
            misc[HM_MX] = 0u;
        }
        __syncthreads();
        unsigned mn = 0xFFFFFFFFu, mx = 0u;
        for (long long i = start + tid; i < end; i += HS_T) {
            const unsigned u = __float_as_uint(__ldg(P.x + i));
            if (((u >> 23) & 0xFFu) == 0xFFu) continue;
            const unsigned ok = u ^ ((unsigned)((int)u >> 31) | 0x80000000u);
            mn = min(mn, ok);
            mx = max(mx, ok);
        }
        mn = __reduce_min_sync(0xFFFFFFFFu, mn);
        mx = __reduce_max_sync(0xFFFFFFFFu, mx);
        if (lane == 0) {
            atomicMin(&misc[HM_MN], mn);
            atomicMax(&misc[HM_MX], mx);
        }
        __syncthreads();
    }
    if (warp == 0) {
        // zeros: every element outside the window took a scratch bin
        const unsigned zs = __reduce_add_sync(0xFFFFFFFFu, hs_smem[HS_MAX_BINS + lane]);
        if (lane == 0) {
            const unsigned nz = zs - misc[HM_COLD];
            if (nz) atomicAdd(&g->nzero, (u64)nz);
            if (misc[HM_MN] != 0xFFFFFFFFu) atomicMax(&g->mn_inv, ~misc[HM_MN]);
            if (misc[HM_MX]) atomicMax(&g->mx, misc[HM_MX]);
        }
    }
    // bins that may have wrapped their 32-bit sum of L: recount those sums in 64 bits (rare)
    for (int i = (int)tid; i < Ly.nbins; i += HS_T) {
        if (hs_smem[i] >= HS_CNT_LIMIT) {
            const unsigned q = atomicAdd(&misc[HM_NOVF], 1u);
            if (q < (unsigned)HS_OVF_MAX) misc[HM_OVF_IDX + q] = (unsigned)i;
        }
    }
    __syncthreads();
    const unsigned novf = min(misc[HM_NOVF], (unsigned)HS_OVF_MAX);
    if (novf) {
        for (long long i = start + tid; i < end; i += HS_T) {
            unsigned L = 0u;
            const int b = hs_bin(__float_as_uint(__ldg(P.x + i)), K, L);
            if (b >= 0 && hs_smem[b] >= HS_CNT_LIMIT)
                for (unsigned q = 0; q < novf; ++q)
                    if (misc[HM_OVF_IDX + q] == (unsigned)b) atomicAdd(&ovf_sum[q], (u64)L);
        }
        __syncthreads();
    }
    // convert the bins, one key per warp
    for (int ks = (int)warp; ks < Ly.nkeys; ks += HS_T / 32) {
        if (P.hs_s == 15)
            hs_convert_key<L1, 8>(P, hs_smem, ovf_sum, misc + HM_OVF_IDX, novf, ks, lane);
        else
            hs_convert_key<L1, 7>(P, hs_smem, ovf_sum, misc + HM_OVF_IDX, novf, ks, lane);
    }
}

}  // namespace
}  // namespace fxpq
