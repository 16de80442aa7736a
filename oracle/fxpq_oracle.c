/*
 * fxpq_oracle.c -- plain, slow CPU oracle for the dynamic fixed-point
 * evaluation path of FxP-QNet (Shawahna et al., IEEE Access 2022,
 * arXiv 2203.12091).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header or table with the CUDA library; it is compiled on its own
 * with gcc.
 *
 * Every function follows the paper's definition written out with plain loops:
 *   - Sec. II-A, Eq. (fixed_point): value = code * 2^-beta, k = alpha + beta.
 *   - Sec. IV-B, Eq. (fp_k_bit_quantization), Eq. (clip), Eq. (quantization_
 *     levels): code = clip(round_half_even(x * 2^beta), Qmin, Qmax) with
 *     Qmin = -S * 2^(k-S), Qmax = 2^(k-S) - 1.
 *   - Sec. IV-C, Eq. (DSB_QE): L(X) = || X - X~ ||_2^2 (a sum, not a mean).
 *   - Sec. IV-B (C-Block arithmetic): MAC of integer codes, exact.
 *
 * The L2 error is summed EXACTLY: every term (x - c)^2 is expanded as
 * x*x - 2*x*c + c*c whose three products are exact doubles for fp32 x and
 * 16-bit codes, and the terms go into a long fixed-point accumulator
 * (Kulisch).  The exact sum is rounded once, to nearest even, to a double.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Exact long accumulator (Kulisch): signed 32-bit digits held in int64.    */
/* Digit i has weight 2^(32*i + KA_BASE).  Covers every finite double and   */
/* every product of two fp32 values.                                        */
/* ------------------------------------------------------------------------ */
#define KA_DIGITS 72
#define KA_BASE (-1184) /* lowest weight 2^-1184 < smallest subnormal double 2^-1074 */

typedef struct {
    int64_t d[KA_DIGITS];
    int64_t adds; /* additions since the last carry normalisation */
} ka_t;

static void ka_zero(ka_t* a) { memset(a, 0, sizeof(*a)); }

/* propagate carries so every digit except the top one is in [0, 2^32) */
static void ka_normalise(ka_t* a) {
    for (int i = 0; i < KA_DIGITS - 1; ++i) {
        int64_t carry = a->d[i] >> 32; /* arithmetic shift: floor division */
        a->d[i] -= carry * ((int64_t)1 << 32);
        a->d[i + 1] += carry;
    }
    a->adds = 0;
}

/* add the double v exactly */
static void ka_add(ka_t* a, double v) {
    if (v == 0.0) return;
    int e;
    double f = frexp(v, &e);               /* v = f * 2^e, 0.5 <= |f| < 1 */
    int64_t m = (int64_t)ldexp(f, 53);     /* exact: |m| < 2^53          */
    int lsb = e - 53;                      /* v = m * 2^lsb               */
    int off = lsb - KA_BASE;               /* bit offset of m's lsb       */
    int idx = off >> 5, sh = off & 31;
    int neg = m < 0;
    uint64_t mag = (uint64_t)(neg ? -m : m);
    unsigned __int128 t = (unsigned __int128)mag << sh; /* < 2^85 */
    for (int i = 0; i < 3; ++i) {
        int64_t dig = (int64_t)(uint64_t)(t & 0xffffffffu);
        t >>= 32;
        if (idx + i < KA_DIGITS) a->d[idx + i] += neg ? -dig : dig;
    }
    if (++a->adds >= ((int64_t)1 << 29)) ka_normalise(a);
}

/* round the exact accumulated value once, to nearest even, to a double */
static double ka_to_double(ka_t* a) {
    ka_normalise(a);
    int neg = a->d[KA_DIGITS - 1] < 0;
    int64_t dd[KA_DIGITS];
    memcpy(dd, a->d, sizeof(dd));
    if (neg) { /* two's complement negate across the digit vector */
        int64_t carry = 1;
        for (int i = 0; i < KA_DIGITS; ++i) {
            int64_t v = (i < KA_DIGITS - 1) ? ((~dd[i]) & 0xffffffff) : -dd[i] - 1;
            v += carry;
            if (i < KA_DIGITS - 1) {
                carry = v >> 32;
                v &= 0xffffffff;
            }
            dd[i] = v;
        }
    }
    int top = -1;
    for (int i = KA_DIGITS - 1; i >= 0; --i)
        if (dd[i] != 0) { top = i; break; }
    if (top < 0) return 0.0;
    /* gather the top 96 bits (three digits) into an unsigned 128-bit integer */
    unsigned __int128 t = 0;
    int lo_digit = top - 2;
    for (int i = top; i >= lo_digit; --i) {
        t <<= 32;
        if (i >= 0) t |= (uint64_t)dd[i];
    }
    int sticky = 0;
    for (int i = lo_digit - 1; i >= 0; --i)
        if (dd[i] != 0) { sticky = 1; break; }
    /* bit length of t */
    int len = 0;
    for (unsigned __int128 u = t; u != 0; u >>= 1) ++len;
    int drop = len - 53; /* bits below the 53-bit significand */
    uint64_t mant;
    if (drop > 0) {
        unsigned __int128 q = t >> drop;
        unsigned __int128 rem = t - (q << drop);
        unsigned __int128 half = (unsigned __int128)1 << (drop - 1);
        /* above half (or exactly half with nonzero lower digits): up;
         * exactly half: to even; below half: down */
        int up = rem > half || (rem == half && (sticky || (q & 1)));
        mant = (uint64_t)q + (uint64_t)up;
    } else {
        mant = (uint64_t)(t << (-drop));
    }
    /* value = t * 2^(32*lo_digit + KA_BASE) ~= mant * 2^(drop + 32*lo_digit + KA_BASE) */
    int exp2 = drop + 32 * lo_digit + KA_BASE;
    double r = ldexp((double)mant, exp2);
    return neg ? -r : r;
}

/* ------------------------------------------------------------------------ */
/* Quantizer Q, Sec. IV-B.                                                  */
/* ------------------------------------------------------------------------ */

/* Eq. (quantization_levels): Qmin = -S * 2^(k-S), Qmax = 2^(k-S) - 1 */
static int64_t ora_qmin(int k, int S) { return S ? -((int64_t)1 << (k - S)) : 0; }
static int64_t ora_qmax(int k, int S) { return ((int64_t)1 << (k - S)) - 1; }

/* round to nearest integer, halves to the even neighbour (Sec. IV-B) */
static double round_half_even(double y) {
    double f = floor(y);
    double d = y - f; /* exact for |y| < 2^52 */
    if (d > 0.5) return f + 1.0;
    if (d < 0.5) return f;
    return (fmod(f, 2.0) == 0.0) ? f : f + 1.0;
}

/* Eq. (fp_k_bit_quantization) + Eq. (clip) for one element; a signed 1-bit data-structure takes the
 * binary quantizer of Eq. (fp_1_bit_quantization): -1 for x < 0, 0 otherwise */
static int64_t ora_q1(float x, int k, int S, int beta) {
    if (k == 1 && S == 1) return x < 0.0f ? -1 : 0;
    double y = ldexp((double)x, beta); /* exact in double */
    double m = round_half_even(y);
    double lo = (double)ora_qmin(k, S), hi = (double)ora_qmax(k, S);
    if (m < lo) m = lo;
    if (m > hi) m = hi;
    return (int64_t)m;
}

/* the value a code stands for: code * 2^-beta, or for the binary quantizer the decoded sign
 * (0 -> +1, -1 -> -1) times 2^-beta */
static double ora_value(int64_t code, int k, int S, int beta) {
    if (k == 1 && S == 1) return ldexp((double)(2 * code + 1), -beta);
    return ldexp((double)code, -beta);
}

void ora_quantize(const float* x, int64_t n, int k, int S, int beta, int32_t* codes) {
    for (int64_t i = 0; i < n; ++i) codes[i] = (int32_t)ora_q1(x[i], k, S, beta);
}

/* Eq. (DSB_QE): L = sum_i (x_i - code_i * 2^-beta)^2, exact then rounded once */
double ora_l2_error(const float* x, int64_t n, int k, int S, int beta) {
    ka_t acc;
    ka_zero(&acc);
    for (int64_t i = 0; i < n; ++i) {
        double xi = (double)x[i];
        double c = ora_value(ora_q1(x[i], k, S, beta), k, S, beta); /* value of the code */
        ka_add(&acc, xi * xi);        /* exact: 48-bit product        */
        ka_add(&acc, -2.0 * xi * c);  /* exact: 24 x 17-bit product   */
        ka_add(&acc, c * c);          /* exact: 17 x 17-bit product   */
    }
    return ka_to_double(&acc);
}

/* Eq. (MAE) without the 1/N: sum_i |x_i - value_i|, exact then rounded once.  Both x_i and the value
 * are exact doubles, so the sign of each difference is decided exactly and each is added with it. */
double ora_l1_error(const float* x, int64_t n, int k, int S, int beta) {
    ka_t acc;
    ka_zero(&acc);
    for (int64_t i = 0; i < n; ++i) {
        double xi = (double)x[i];
        double c = ora_value(ora_q1(x[i], k, S, beta), k, S, beta);
        if (xi >= c) {
            ka_add(&acc, xi);
            ka_add(&acc, -c);
        } else {
            ka_add(&acc, c);
            ka_add(&acc, -xi);
        }
    }
    return ka_to_double(&acc);
}

/* exact sum of a double vector, rounded once (used by the oracle's stats and
 * by tests that pin the accumulator itself) */
double ora_exact_sum(const double* v, int64_t n) {
    ka_t acc;
    ka_zero(&acc);
    for (int64_t i = 0; i < n; ++i) ka_add(&acc, v[i]);
    return ka_to_double(&acc);
}

/*
 * FL search over a grid of candidates: for every wordlength k in [k_lo,k_hi]
 * and fractional length beta in [fl_lo, fl_hi], L(X; k, beta, S) by
 * Eq. (DSB_QE) (score 0) or the L1 error of Eq. (MAE) as a sum (score 1); best[k] = the beta with the
 * smallest score, exact ties going to
 * the smallest beta.  err is row-major [k][beta].
 * S = -1 picks the sign strategy by Sec. IV-A.3: S = 1 iff min(X) < 0.
 * stats = {min, max, sum, sumsq} (sum and sumsq exact, rounded once).
 * Returns the S used.
 */
int ora_fl_search(const float* x, int64_t n, int S, int k_lo, int k_hi, int fl_lo, int fl_hi,
                  double* err, int32_t* best, double* stats, int score) {
    float mn = INFINITY, mx = -INFINITY;
    ka_t s1, s2;
    ka_zero(&s1);
    ka_zero(&s2);
    for (int64_t i = 0; i < n; ++i) {
        if (x[i] < mn) mn = x[i];
        if (x[i] > mx) mx = x[i];
        ka_add(&s1, (double)x[i]);
        ka_add(&s2, (double)x[i] * (double)x[i]);
    }
    if (n == 0) { mn = 0.0f; mx = 0.0f; }
    if (S < 0) S = (mn < 0.0f) ? 1 : 0;
    int nfl = fl_hi - fl_lo + 1;
    int nk = k_hi - k_lo + 1;
    /* every candidate is scored independently (OpenMP only spreads the candidates) */
#pragma omp parallel for schedule(dynamic, 1)
    for (int c = 0; c < nk * nfl; ++c)
        err[c] = score == 1 ? ora_l1_error(x, n, k_lo + c / nfl, S, fl_lo + c % nfl)
                            : ora_l2_error(x, n, k_lo + c / nfl, S, fl_lo + c % nfl);
    for (int k = k_lo; k <= k_hi; ++k) {
        double bestv = INFINITY;
        int bestfl = fl_lo;
        for (int b = fl_lo; b <= fl_hi; ++b) {
            double e = err[(int64_t)(k - k_lo) * nfl + (b - fl_lo)];
            if (e < bestv) { bestv = e; bestfl = b; } /* strict: exact ties keep the smaller FL */
        }
        best[k - k_lo] = bestfl;
    }
    stats[0] = (double)mn;
    stats[1] = (double)mx;
    stats[2] = ka_to_double(&s1);
    stats[3] = ka_to_double(&s2);
    return S;
}

/* ------------------------------------------------------------------------ */
/* Integer C-Block contraction, Sec. IV-B: exact MAC of codes (int64).      */
/* Activations NHWC, weights KRSC (out, kh, kw, in), output acc[N][P][Q][K].*/
/* Taps outside the input are zero codes (= value 0).                       */
/* ------------------------------------------------------------------------ */
void ora_conv2d(const int32_t* x, int N, int H, int W, int C, const int32_t* w, int K, int R,
                int S, int stride, int pad, int P, int Q, int64_t* acc) {
#pragma omp parallel for collapse(2) schedule(static)
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < Q; ++q)
                for (int k = 0; k < K; ++k) {
                    int64_t sum = 0;
                    for (int r = 0; r < R; ++r) {
                        int h = p * stride + r - pad;
                        if (h < 0 || h >= H) continue;
                        for (int s = 0; s < S; ++s) {
                            int ww = q * stride + s - pad;
                            if (ww < 0 || ww >= W) continue;
                            const int32_t* xa = x + (((int64_t)n * H + h) * W + ww) * C;
                            const int32_t* wa = w + (((int64_t)k * R + r) * S + s) * C;
                            for (int c = 0; c < C; ++c) sum += (int64_t)xa[c] * (int64_t)wa[c];
                        }
                    }
                    acc[(((int64_t)n * P + p) * Q + q) * K + k] = sum;
                }
}
