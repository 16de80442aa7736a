/*
 * fxpq.h -- C ABI of libfxpq.so: the data-parallel hot path of evaluating a CNN under a
 * dynamic fixed-point configuration (FxP-QNet, Shawahna et al., IEEE Access 2022,
 * arXiv 2203.12091), on one NVIDIA GB300 (sm_103a).
 *
 * Conventions shared by every entry point
 *   - Pointers named d_* are device pointers; h_* are host pointers.  The caller owns every
 *     buffer.  The library allocates no device memory: scratch comes from the caller's
 *     workspace, sized by the matching *_workspace() query.
 *   - Calls are asynchronous on the caller's stream (a cudaStream_t passed as void*;
 *     NULL = the legacy default stream), except where a function says it synchronises.
 *   - Arguments are validated on the host before any launch; a failed check returns an error
 *     code and launches nothing.  Errors detected on the device (non-finite input, a bounded
 *     wait that ran out) are latched in a device status word read by fxpq_get_device_status().
 *   - Results are deterministic: no floating-point atomics; repeated calls are bit-identical.
 *
 * Notation follows the paper: a data-structure is a group of k-bit integer codes sharing the
 * scale 2^-FL ("beta" in the paper); k = alpha + beta (Sec. II-A); S is the sign strategy
 * (0 = unsigned U(alpha, beta), 1 = two's complement S(alpha, beta)).
 *
 * Code storage ("fp16 code tensors").  Inside the network path every code tensor is stored as
 * fp16 values that are exact integers.  A format with k <= 8 bits uses one plane (|code| <= 255).
 * A format with 9..16 bits uses two planes, hi and lo, with code = 256*hi + lo, lo in [0, 255]
 * and hi = floor(code / 256).  Planes are stored plane-major: the whole hi tensor, then the whole
 * lo tensor of the same shape (for an NHWC tensor [N,H,W,Cp] the lo plane starts N*H*W*Cp
 * elements after the hi plane).  Channel counts are padded to a multiple of 8 with zero codes.
 */
#ifndef FXPQ_H
#define FXPQ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define FXPQ_API __attribute__((visibility("default")))
#else
#define FXPQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FXPQ_OK = 0,
    FXPQ_ERR_INVALID_ARG = 1, /* a null/misaligned pointer, a size or a format out of range     */
    FXPQ_ERR_UNSUPPORTED = 2, /* a valid request this build does not implement                  */
    FXPQ_ERR_NONFINITE = 3,   /* fl_search / quantize saw a NaN or Inf (latched on the device)  */
    FXPQ_ERR_TIMEOUT = 4,     /* a bounded device-side wait gave up (latched on the device)     */
    FXPQ_ERR_CUDA = 5,        /* a CUDA runtime call failed                                     */
    FXPQ_ERR_WORKSPACE = 6,   /* the workspace is null or smaller than the query returned       */
    FXPQ_ERR_RANGE = 7        /* an integer bound the exact arithmetic relies on would not hold */
} fxpq_status;

/* Storage of integer codes in device memory. */
typedef enum {
    FXPQ_DT_I8 = 0,  /* int8   : signed formats, k <= 8       */
    FXPQ_DT_U8 = 1,  /* uint8  : unsigned formats, k <= 8     */
    FXPQ_DT_I16 = 2, /* int16  : signed formats, k <= 16      */
    FXPQ_DT_U16 = 3, /* uint16 : unsigned formats, k <= 16    */
    FXPQ_DT_I32 = 4, /* int32  : any format                   */
    FXPQ_DT_F16 = 5  /* fp16 code tensor (see the file header): one or two limb planes */
} fxpq_dtype;

/* Quantization parameters of one data-structure (Sec. IV-A.3 / IV-B): wordlength k = bits,
 * sign strategy S = is_signed, fractional length beta = fl; alpha = bits - fl. */
typedef struct {
    int32_t bits;      /* 2..16 (32 is accepted for biases, which are int32 codes) */
    int32_t is_signed; /* 0: U(alpha, beta), codes in [0, 2^k - 1]; 1: S(alpha, beta), [-2^(k-1), 2^(k-1) - 1] */
    int32_t fl;        /* beta, in [-32, 40] */
} fxpq_fmt;

/* Statistics gathered by the FL-search pass over a tensor. */
typedef struct {
    float min, max;     /* exact                                                          */
    int32_t is_signed;  /* sign strategy of Sec. IV-A.3: 1 iff min < 0                     */
    int32_t nonfinite;  /* 1 if a NaN/Inf was seen (the scores are then not meaningful)    */
    double sum, sumsq;  /* exact sums rounded once to double                               */
    int64_t n;
} fxpq_stats;

/* ---------------------------------------------------------------------------------------- */
/* Quantizer Q (Sec. IV-B, Eq. fp_k_bit_quantization, Eq. clip, Eq. quantization_levels):   */
/*   code_i = clip(round_half_even(x_i * 2^fl), Qmin, Qmax),                                */
/*   Qmin = -S * 2^(k-S), Qmax = 2^(k-S) - 1.                                                */
/* d_x: n fp32 values.  d_codes: n codes in storage `dtype` (I8/U8/I16/U16/I32 must be wide   */
/* enough and of the right signedness; F16 writes an fp16 code tensor: plane hi at [0, n) and */
/* plane lo at [n, 2n) when k > 8).  n may be 0.                                             */
/* NaN/Inf inputs latch FXPQ_ERR_NONFINITE and produce code 0.                               */
/* f.bits may be 1: S = 0 gives the levels {0, 1}; S = 1 the binary quantizer of             */
/* Eq. fp_1_bit_quantization, code -1 for x < 0 and 0 otherwise (-0.0 included), decoded     */
/* 0 -> +1 before use, so the values are +-2^-fl.  fxpq_pack_codes stores it in one bit.     */
/* ---------------------------------------------------------------------------------------- */
FXPQ_API fxpq_status fxpq_quantize(const float* d_x, int64_t n, fxpq_fmt f, int32_t dtype, void* d_codes,
                          void* stream);

/* Quantize a row-major [rows, C] fp32 tensor (e.g. KRSC weights with C innermost) into an fp16
 * code tensor: planes (per f.bits, see the file header) of [rows, Cp]; channels C..Cp-1 are zero
 * codes.  Cp is a multiple of 8 and >= C. */
FXPQ_API fxpq_status fxpq_quantize_rows(const float* d_x, int64_t rows, int32_t C, fxpq_fmt f, int32_t Cp, void* d_y,
                               void* stream);

/* Parameter quantization in one launch, with formats that stay on the device: each item's S and
 * FL are read from device memory (typically the d_stats / d_best results of fxpq_fl_search_batch),
 * so no host round trip separates the FL search from the quantization (Sec. IV-C: weights and
 * biases are quantized with the FL the search picked).  Item kinds:
 *   FXPQ_QB_ROWS_F16: `rows` rows of C fp32 values -> fp16 code planes [rows, Cp] (as
 *                     fxpq_quantize_rows); with d_l1 (bits <= 8) the largest L1 norm over groups
 *                     of rows_per_group consecutive rows (an output channel of KRSC weights:
 *                     rows_per_group = R*S) is atomically max-ed into *d_l1 (initialise it).
 *                     C == Cp needs d_x and d_out 16-byte aligned; rows % rows_per_group == 0.
 *   FXPQ_QB_FLAT_I32: `rows` fp32 values -> int32 codes (biases, the avg-pool reciprocal).
 * Non-finite inputs latch FXPQ_ERR_NONFINITE and produce code 0.  Not part of the paper's
 * statement beyond Q itself: it batches Eq. fp_k_bit_quantization over many tensors. */
enum { FXPQ_QB_ROWS_F16 = 0, FXPQ_QB_FLAT_I32 = 1 };
typedef struct {
    const float* d_x;
    void* d_out;
    int32_t kind;             /* FXPQ_QB_*                                                     */
    int32_t bits;             /* k (2..16)                                                     */
    int64_t rows;             /* ROWS_F16: rows of C values; FLAT_I32: element count           */
    int32_t C, Cp;            /* ROWS_F16 geometry                                             */
    int32_t rows_per_group;   /* ROWS_F16: rows per L1 group                                   */
    int32_t reserved;
    const int32_t* d_fl;      /* device int32: FL                                              */
    const fxpq_stats* d_stats; /* device: is_signed gives S                                    */
    int64_t* d_l1;            /* ROWS_F16, bits <= 8: L1 bound output, or NULL                 */
} fxpq_quantize_item;

FXPQ_API fxpq_status fxpq_quantize_batch(const fxpq_quantize_item* h_items, int32_t n_items, void* stream);

/* Largest L1 norm over the rows of a one-plane fp16 code tensor [rows, L] (fmt.bits <= 8):
 * *d_out = max_r sum_j |code[r, j]| as an int64 on the device (0 when rows == 0).  For KRSC
 * weights with L = R*S*Cp it is the w_l1 bound of fxpq_conv_desc.  Exact integer arithmetic;
 * d_codes 16-byte aligned and L a multiple of 8.  Not part of the paper: it feeds the
 * implementation's exact-accumulation planning. */
FXPQ_API fxpq_status fxpq_code_l1max(const void* d_codes, int64_t rows, int64_t L, int64_t* d_out, void* stream);

/* Quantize + transpose + pack fp32 images NCHW -> NHWC fp16 code tensor with the channel count
 * padded to c_pad (a multiple of 8, >= C) with zero codes: the FxP-QLayer inserted at the input
 * of the network (Sec. IV-A.2).  d_y (16-byte aligned) holds planes x [N, H, W, c_pad] fp16
 * values. */
FXPQ_API fxpq_status fxpq_quantize_images(const float* d_x_nchw, int32_t N, int32_t C, int32_t H, int32_t W,
                                 fxpq_fmt f, int32_t c_pad, void* d_y, void* stream);

/* ---------------------------------------------------------------------------------------- */
/* FL search (Sec. IV-C, Eq. DSB_QE; sign strategy Sec. IV-A.3).                             */
/* One pass over d_x scores every candidate (k, fl), k in [k_lo, k_hi] and fl in              */
/* [fl_lo, fl_hi]:  L(k, fl) = sum_i (x_i - Q(x_i; k, fl) * 2^-fl)^2  -- the exact sum,       */
/* rounded once to nearest-even double.                                                      */
/*   is_signed: 0 or 1 fixes S; -1 picks S = 1 iff min(x) < 0.                                */
/*   d_err  : device double[(k_hi-k_lo+1) * (fl_hi-fl_lo+1)], row-major [k][fl].              */
/*   d_best : device int32[k_hi-k_lo+1]: the fl with the smallest L per k, exact ties to the  */
/*            smallest fl.                                                                   */
/*   d_stats: device fxpq_stats (may be NULL).                                               */
/* k = 1 with S = 1 scores the binary quantizer of Eq. fp_1_bit_quantization (every value     */
/* decoded to +-2^-fl: error | |x| - 2^-fl |, zeros included); k = 1 with S = 0 the levels    */
/* {0, 1}.                                                                                   */
/* Limits: 1 <= k_lo <= k_hi <= 16; -32 <= fl_lo <= fl_hi <= 40; fl_hi - fl_lo <= 31;         */
/* 0 <= n <= 2^31.  Non-finite inputs latch FXPQ_ERR_NONFINITE.                              */
/* Workspace: fxpq_fl_search_workspace() bytes, 256-byte aligned; contents are scratch.       */
/* ---------------------------------------------------------------------------------------- */
FXPQ_API size_t fxpq_fl_search_workspace(int64_t n);
FXPQ_API fxpq_status fxpq_fl_search(const float* d_x, int64_t n, int32_t is_signed, int32_t k_lo, int32_t k_hi,
                           int32_t fl_lo, int32_t fl_hi, double* d_err, int32_t* d_best,
                           fxpq_stats* d_stats, void* d_ws, size_t ws_bytes, void* stream);

/* Several independent FL searches (e.g. every weight and bias tensor of a network, Sec. IV-C's
 * per-data-structure search) in one set of launches: each item has the arguments, results and
 * limits of fxpq_fl_search.  Every item is validated before the first launch.  The batch runs in
 * groups of up to 32 items, each group as three kernels on `stream`.
 * Workspace: fxpq_fl_search_batch_workspace(n_items) bytes, 256-byte aligned; scratch. */
typedef struct {
    const float* d_x;      /* device tensor of n fp32 values                                  */
    int64_t n;
    int32_t is_signed;     /* 0, 1, or -1 (S = 1 iff min(x) < 0)                              */
    int32_t k_lo, k_hi;
    int32_t fl_lo, fl_hi;
    double* d_err;         /* device double[(k_hi-k_lo+1) * (fl_hi-fl_lo+1)]                  */
    int32_t* d_best;       /* device int32[k_hi-k_lo+1]                                       */
    fxpq_stats* d_stats;   /* device fxpq_stats or NULL                                       */
    int32_t score;         /* FXPQ_SCORE_L2: Eq. DSB_QE; FXPQ_SCORE_L1: sum_i |x_i - Q(x_i)|,   */
                           /* the L1 error of Eq. MAE times N (same argmin), exact, rounded once */
} fxpq_fl_search_item;

enum { FXPQ_SCORE_L2 = 0, FXPQ_SCORE_L1 = 1 };

FXPQ_API size_t fxpq_fl_search_batch_workspace(int32_t n_items);
FXPQ_API fxpq_status fxpq_fl_search_batch(const fxpq_fl_search_item* h_items, int32_t n_items, void* d_ws,
                                          size_t ws_bytes, void* stream);

/* fxpq_fl_search for callers that cannot allocate device memory -- for instance a plug-in whose
 * host application owns the whole device memory pool, or a latency-critical loop that must never
 * enter the allocator (cudaMalloc may synchronise the device).  The paper has no counterpart: this
 * is a deployment variant of fxpq_fl_search with the same arguments, results and limits, minus
 * the workspace.  It allocates nothing.  Its scratch is a file-scope device array of about
 * 81 KiB inside libfxpq.so that every GPU which loads the library holds until the process exits.
 *   - Limits: n <= 2^31 elements and at most 16 x 32 candidates (k in [1,16], fl_hi-fl_lo <= 31);
 *     larger requests return FXPQ_ERR_INVALID_ARG before any launch.
 *   - The first call on a device looks up the array's device address (cudaGetSymbolAddress) with
 *     that device current; make that first call before any stream capture begins.
 *   - All calls share the one array and each call clears it before use.  Calls that overlap on the
 *     GPU (concurrent streams, or several host threads) race on it and give wrong results:
 *     serialise them, or use fxpq_fl_search with a workspace per stream. */
FXPQ_API fxpq_status fxpq_fl_search_noalloc(const float* d_x, int64_t n, int32_t is_signed, int32_t k_lo,
                                            int32_t k_hi, int32_t fl_lo, int32_t fl_hi, double* d_err,
                                            int32_t* d_best, fxpq_stats* d_stats, void* stream);

/* Initial quantization parameters (Sec. IV-A.3, Eq. initial_quantization_parameters), a host
 * helper on statistics already copied to the host: psi from the range, beta_hat = -log2(psi),
 * beta = floor (strategy 0, conservative) / round half-even (1, neutral) / ceil (2, aggressive).
 * Where one of the two signed candidates for psi is not positive it is dropped. */
FXPQ_API fxpq_status fxpq_fl_init(const fxpq_stats* h_stats, int32_t bits, int32_t strategy, fxpq_fmt* h_out);

/* ---------------------------------------------------------------------------------------- */
/* C-Block: convolution / FC on codes with exact integer accumulation and the fused epilogue */
/* (Sec. IV-B, the C-Block paragraph and its figure; FxP-QLayer placement Sec. IV-A.2):      */
/*   acc[n,p,q,o] = sum_{r,s,c} X[n, p*st+r-pad, q*st+s-pad, c] * W[o, r, s, c]    (exact)    */
/*   value scale s = fl_x + fl_w; bias aligned with delta = s - fl_b: delta >= 0 adds          */
/*   B << delta, delta < 0 shifts acc left by -delta first (no bit is dropped);               */
/*   ReLU = max(., 0) if relu;                                                               */
/*   out_mode CODES : FxP-QLayer -> round_half_even(v * 2^(fl_y - s)), clip to fmt_y,         */
/*                    written as an fp16 code tensor NHWC [N,P,Q,K] (K a multiple of 8);      */
/*   out_mode ACC64 : no QLayer (last layer): int64 v, NHWC [N,P,Q,K]; its scale exponent is   */
/*                    returned in *h_out_scale;                                               */
/*   out_mode F32   : fp32 nearest-even image of v * 2^-s (for calibrating fmt_y.fl).          */
/* X: fp16 code tensor NHWC [N,H,W,Cp] (planes per fmt_x.bits); W: fp16 code tensor KRSC       */
/* [K,R,S,Cp] (planes per fmt_w.bits); d_bias: int32 codes [K] or NULL.  X, W, Y 16-byte      */
/* aligned.                                                                                  */
/* An FC layer is a convolution whose window covers the whole input map (R = H, S = W).      */
/* Returns FXPQ_ERR_RANGE if |acc| could exceed 2^62 after alignment.                         */
/* w_l1 (optional, one-plane weights only): an upper bound on max_o sum_{r,s,c} |W[o,r,s,c]|, */
/* e.g. from fxpq_code_l1max, 0 = none.  Every partial sum of output channel o is then at     */
/* most max|x code| * w_l1, which lets the tensor-core path keep longer reductions in exact    */
/* fp32 groups and the epilogue in 32-bit arithmetic.  A value below the true norm voids the  */
/* exactness guarantee; not part of the paper (an implementation bound).                      */
/* Scale layer (optional; Sec. IV-A.1: a BN layer rewritten as aleph1 * A + aleph2, its two    */
/* per-channel parameters quantized like weights and biases; Sec. IV-B: integer multiply and  */
/* accumulate in the C-Block): when d_scale != NULL, after the bias alignment the value v of  */
/* scale s becomes v * aleph1_code[o] of scale s + fmt_scale.fl, and aleph2_code[o] is aligned  */
/* to it like the bias (delta2 = that scale - fmt_shift.fl, the same two cases); ReLU and the  */
/* FxP-QLayer follow.  d_scale and d_shift are int32 code arrays [K], both set or both NULL.   */
/* d_wpacked (optional; Sec. V-E.2: k-bit storage of the read-only data-structures): the       */
/* weights of d_w, one plane of fmt_w.bits <= 8, as fxpq_pack_weights' tiles.  Layers whose A   */
/* operand is the stored activations themselves (FC layers: R = H, S = W, pad 0; 1x1 stride-1   */
/* without padding) and whose output tiles are too few for the SMs (the split reduction) then   */
/* read k bits per weight from memory instead of a 2-byte fp16 code; other layers ignore it.    */
/* d_w stays required (every other path reads it); d_wpacked must hold exactly d_w's codes,     */
/* 16-byte aligned.                                                                             */
/* ---------------------------------------------------------------------------------------- */
enum { FXPQ_OUT_CODES = 0, FXPQ_OUT_ACC64 = 1, FXPQ_OUT_F32 = 2 };

typedef struct {
    int32_t N, H, W, C;        /* input geometry; C = true channel count                    */
    int32_t Cp;                /* stored channel count of X and W (multiple of 8, >= C)      */
    int32_t K, R, S;           /* output channels, window                                   */
    int32_t stride, pad;
    int32_t relu;
    int32_t out_mode;          /* FXPQ_OUT_*                                                 */
    fxpq_fmt fmt_x, fmt_w, fmt_b, fmt_y;
    int64_t w_l1;              /* optional weight-code L1 bound (see above), 0 = none        */
    fxpq_fmt fmt_scale, fmt_shift;  /* Scale layer aleph1 / aleph2 formats (if d_scale)      */
    const int32_t* d_scale;    /* Scale layer aleph1 codes [K], or NULL (no Scale layer)     */
    const int32_t* d_shift;    /* Scale layer aleph2 codes [K] (NULL iff d_scale is NULL)    */
    const void* d_wpacked;     /* optional: the same weights packed by fxpq_pack_weights, or NULL */
} fxpq_conv_desc;

FXPQ_API size_t fxpq_conv_workspace(const fxpq_conv_desc* h_desc);
FXPQ_API fxpq_status fxpq_conv_fwd(const fxpq_conv_desc* h_desc, const void* d_x, const void* d_w,
                          const int32_t* d_bias, void* d_y, int32_t* h_out_scale, void* d_ws,
                          size_t ws_bytes, void* stream);

/* FC layer as a GEMM: X [M, Kdim] (fp16 codes, Kdim padded to 8), W [N, Kdim]; same epilogue. */
FXPQ_API fxpq_status fxpq_gemm(const void* d_x, fxpq_fmt fmt_x, const void* d_w, fxpq_fmt fmt_w,
                      const int32_t* d_bias, fxpq_fmt fmt_b, int32_t M, int32_t N, int32_t Kdim,
                      int32_t relu, int32_t out_mode, fxpq_fmt fmt_y, void* d_y, int32_t* h_out_scale,
                      void* d_ws, size_t ws_bytes, void* stream);

/* MAX-POOL on codes (Sec. IV-A.2: no FxP-QLayer follows; the format is unchanged).  Window
 * k x k, stride, pad; taps outside the map are ignored.  X, Y: fp16 code tensors NHWC with
 * Cp channels (planes per fmt.bits, pooled as whole codes). */
FXPQ_API fxpq_status fxpq_maxpool(const void* d_x, int32_t N, int32_t H, int32_t W, int32_t Cp, fxpq_fmt fmt,
                         int32_t k, int32_t stride, int32_t pad, void* d_y, void* stream);

/* Eltwise C-Block (Sec. IV-A.2, residual add): both inputs aligned to max(fl_a, fl_b) by an
 * exact left shift, added, optional ReLU, then the FxP-QLayer to fmt_y (or F32 / ACC64 as in
 * fxpq_conv_fwd).  A, B, Y: NHWC with Cp channels, count = n_pix * Cp codes. */
FXPQ_API fxpq_status fxpq_eltwise(const void* d_a, fxpq_fmt fmt_a, const void* d_b, fxpq_fmt fmt_b, int64_t n_pix,
                         int32_t Cp, int32_t relu, int32_t out_mode, fxpq_fmt fmt_y, void* d_y,
                         int32_t* h_out_scale, void* stream);

/* FxP-QLayer (Sec. IV-A.2 and the requantization paragraph of Sec. IV-B) as a standalone op: n int64
 * C-Block values v with scale 2^-s (e.g. the ACC64 output of fxpq_conv_fwd) become
 *   out_mode CODES: round_half_even(v * 2^(fl_y - s)) clipped to fmt_y, as an fp16 code tensor of n
 *                   codes (plane-major when fmt_y.bits > 8);
 *   out_mode F32  : the fp32 nearest-even image of v * 2^-s;  ACC64: a copy of v.
 * -64 <= s <= 80. */
FXPQ_API fxpq_status fxpq_qlayer(const int64_t* d_v, int64_t n, int32_t s, int32_t out_mode, fxpq_fmt fmt_y,
                                 void* d_y, void* stream);

/* Global AVG-POOL (Sec. IV-A.2: the reciprocal of the patch size is quantized like a parameter):
 * v[n,c] = recip_code * sum_{h,w} X[n,h,w,c], scale fl_x + fmt_recip.fl, then the FxP-QLayer to
 * fmt_y (or F32 / ACC64).  Output NHWC with H = W = 1. */
FXPQ_API fxpq_status fxpq_avgpool(const void* d_x, int32_t N, int32_t H, int32_t W, int32_t Cp, fxpq_fmt fmt_x,
                         int32_t recip_code, fxpq_fmt fmt_recip, int32_t out_mode, fxpq_fmt fmt_y,
                         void* d_y, int32_t* h_out_scale, void* stream);

/* Packed k-bit code storage (the footprint of Sec. V-E.2's memory model: k bits per code, Eq. mfp).
 * Codes are taken in groups of 32 (the last zero-padded); group g occupies k = fmt.bits uint32 words,
 * word g*k + b holding bit b of the k-bit two's-complement field of code 32g + i at bit i (a bit-plane
 * layout: a warp packs a group with k ballots and unpacks it with k shuffles).  Unpacking sign-extends
 * when fmt.is_signed.  d_codes: fp16 code tensor of n codes (plane-major when fmt.bits > 8), 2-byte
 * aligned; d_words: ceil(n / 32) * fmt.bits words, 4-byte aligned.  Codes outside fmt's range are
 * truncated to their low k bits (they cannot come from the quantizer). */
FXPQ_API fxpq_status fxpq_pack_codes(const void* d_codes, int64_t n, fxpq_fmt fmt, uint32_t* d_words, void* stream);
FXPQ_API fxpq_status fxpq_unpack_codes(const uint32_t* d_words, int64_t n, fxpq_fmt fmt, void* d_codes,
                                       void* stream);

/* Packed weights for the contraction (Sec. V-E.2: a data-structure of k-bit values occupies k bits
 * per value).  d_w: one plane of fp16 weight codes [K][L] (L = R*S*Cp, KRSC order), fmt_w.bits in
 * [1, 8].  d_packed receives the codes' k-bit two's-complement fields as bit planes of tiles of 256
 * output channels x 64 reduction steps: words [ceil(L / 64)][K_pad / 256][k][256][2], K_pad = K
 * rounded up to a multiple of 256; word (kb, t, b, o, h) holds at bit i bit b of the field of code
 * W[256 t + o][64 kb + 32 h + i] (zero past L and past K).  These are fxpq_pack_codes' words for the
 * codes rearranged as [ceil(L / 64)][K_pad][64], with each tile's words ordered plane-major.  One tile
 * is a single contiguous run of 2 KiB per plane, which the contraction copies to shared memory and
 * expands there.  fxpq_packed_weights_bytes gives the size (k bits per code of the padded tensor);
 * d_packed 16-byte aligned. */
FXPQ_API size_t fxpq_packed_weights_bytes(fxpq_fmt fmt_w, int32_t K, int32_t L);
FXPQ_API fxpq_status fxpq_pack_weights(const void* d_w, fxpq_fmt fmt_w, int32_t K, int32_t L, void* d_packed,
                                       void* stream);

/* BN -> Scale preprocessing (Sec. IV-A.1, the BatchNorm rewrite): per channel,
 *   aleph1 = gamma / sqrt(var + eps),  aleph2 = beta - (gamma * mean) / sqrt(var + eps),
 * each operation one correctly rounded fp32 step in that order.  Inputs: fp32 device arrays of n
 * channels (running statistics and the affine parameters); outputs: fp32 device arrays of n, which
 * the FL search and fxpq_quantize turn into the Scale layer's codes.  eps >= 0. */
FXPQ_API fxpq_status fxpq_bn_to_scale(const float* d_gamma, const float* d_beta, const float* d_mean,
                                      const float* d_var, int64_t n, float eps, float* d_aleph1, float* d_aleph2,
                                      void* stream);

/* ---------------------------------------------------------------------------------------- */
/* Network forward (Sec. IV-A.2: FxP-QLayers as vertices, C-Blocks as edges).                */
/* A network is a list of ops over numbered tensor slots; slot 0 is the input image codes.   */
/* Every op reads its source slot(s) and writes slot `dst`.  The last op must be a CONV with  */
/* last = 1: its int64 accumulator (no QLayer, Sec. IV-A.2) is written to d_logits            */
/* [batch, K] and its scale exponent to *h_logits_scale.                                      */
/* ---------------------------------------------------------------------------------------- */
enum { FXPQ_OP_CONV = 0, FXPQ_OP_MAXPOOL = 1, FXPQ_OP_ELTWISE = 2, FXPQ_OP_AVGPOOL = 3 };

typedef struct {
    int32_t op;              /* FXPQ_OP_*                                                    */
    int32_t src0, src1;      /* source slots (src1: second eltwise operand, else -1)         */
    int32_t dst;             /* destination slot                                             */
    int32_t K, R, S;         /* conv: output channels and window; maxpool: window in R (=S)   */
    int32_t stride, pad;
    int32_t relu;
    int32_t last;            /* 1 for the final conv/FC (int64 logits)                       */
    int32_t recip_code;      /* avgpool: quantized reciprocal of the patch size             */
    fxpq_fmt fmt_w, fmt_b;   /* conv: weight and bias formats; avgpool: fmt_w = reciprocal  */
    fxpq_fmt fmt_y;          /* format of the output QLayer (ignored for maxpool / last)    */
    const void* d_w;         /* conv: fp16 code tensor KRSC [K, R, S, Cp_in]                 */
    const int32_t* d_bias;   /* conv: int32 bias codes [K] or NULL                           */
    int64_t w_l1;            /* conv: optional weight-code L1 bound (fxpq_conv_desc.w_l1)    */
    fxpq_fmt fmt_scale, fmt_shift;  /* conv: Scale layer formats (fxpq_conv_desc)            */
    const int32_t* d_scale;  /* conv: Scale layer aleph1 codes [K] or NULL                   */
    const int32_t* d_shift;  /* conv: Scale layer aleph2 codes [K] or NULL                   */
    const void* d_wpacked;   /* conv: optional packed weights (fxpq_conv_desc.d_wpacked)       */
} fxpq_op_desc;

typedef struct {
    int32_t n_ops;
    int32_t n_slots;
    int32_t C, H, W;          /* input image geometry (NCHW fp32)                           */
    int32_t Cp_in;            /* padded channel count of slot 0                             */
    fxpq_fmt fmt_in;          /* input FxP-QLayer format                                    */
    const fxpq_op_desc* ops;  /* host array of n_ops descriptors                            */
} fxpq_net;

FXPQ_API size_t fxpq_net_workspace(const fxpq_net* h_net, int32_t batch);

/* Memory requirement of one inference (Sec. V-E.2, Eq. mfp, RW_R and RO_R), a host computation on the
 * op list: MFP = nu * k / 2^23 MB for nu elements at k bits (k = 32 for every data-structure when
 * fp32 != 0, the FP32 baseline).  *h_rw_mb = the largest, over ops, of the footprint of the op's input
 * activations (both operands of an eltwise) plus its output activations, per image, with the true
 * channel counts (net->C for the input; the last op's output, which has no FxP-QLayer, at 32 bits);
 * *h_ro_mb = the sum over conv ops of the weights (K*R*S*C), the bias (K, when d_bias) and the Scale
 * layer's aleph1 and aleph2 (K each, when d_scale) at their formats' bits.  The compression rates are
 * ratios of the two calls (fp32 = 1 over fp32 = 0).  No device access. */
FXPQ_API fxpq_status fxpq_net_memory(const fxpq_net* h_net, int32_t fp32, double* h_rw_mb, double* h_ro_mb);
FXPQ_API fxpq_status fxpq_net_forward(const fxpq_net* h_net, const float* d_images_nchw, int32_t batch,
                             int64_t* d_logits, int32_t* h_logits_scale, void* d_ws, size_t ws_bytes,
                             void* stream);

/* Calibration of the activation formats in the forward optimizer's order (Sec. IV-C, which does not
 * say where activation FLs come from; here they are searched on a calibration slice and then
 * frozen): the input FxP-QLayer's FL is searched on the fp32 calibration images, then
 * layer by layer, with every earlier layer already quantized, the FL of each op's output QLayer is
 * searched on the fp32 nearest-even image of its exact C-Block output (conv: the contraction to that
 * image, then again to codes with the searched format, or -- where a time model of output size against
 * input, weight and contraction work favours it, the FC layers and late 3x3 layers at calibration batch
 * sizes -- the contraction once to int64 values and fxpq_qlayer to the image and then to the codes;
 * eltwise / avg-pool: their F32 and CODES modes).  S is
 * picked from the data (Sec. IV-A.3); FLs in [fl_lo, fl_hi], exact ties to the smaller FL.
 *   h_net: every parameter quantized (d_w, d_bias, fmt_w, fmt_b, recip_code, w_l1); fmt_in.bits and
 *          each op's fmt_y.bits give the wordlengths (their S and FL are ignored);
 *   h_fmt_in: the chosen input format; h_fmt_y[n_ops]: each op's output format (a max-pool passes
 *          its input's on; the last op's entry is copied unchanged).
 * The host waits for each search (a stream synchronisation per QLayer; the search writes its result
 * into a mapped pinned host record that the library allocates once and reuses).  Errors: as the
 * calls it makes, FXPQ_ERR_CUDA if the host record cannot be allocated.  Workspace:
 * fxpq_net_calibrate_workspace(h_net, n_calib) bytes, 256-byte aligned. */
FXPQ_API size_t fxpq_net_calibrate_workspace(const fxpq_net* h_net, int32_t n_calib);
FXPQ_API fxpq_status fxpq_net_calibrate(const fxpq_net* h_net, const float* d_calib_nchw, int32_t n_calib,
                                        int32_t fl_lo, int32_t fl_hi, fxpq_fmt* h_fmt_in, fxpq_fmt* h_fmt_y,
                                        void* d_ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------- */
/* Forward optimizer support (Sec. IV-C, Alg. 1 QParamsOpt and its cost F of                */
/* Eq. quantization_parameters_optimization).  While one data-structure's QPs are searched,  */
/* every data-structure after it is FP32: these are the FP32 layers, the conversions between */
/* the two worlds, and the statistics the cost reads.  FP32 tensors are NHWC with the true    */
/* channel count (no padding).                                                               */
/* ---------------------------------------------------------------------------------------- */
typedef struct {
    int32_t N, H, W, C;        /* input geometry                                             */
    int32_t K, R, S;           /* output channels, window                                    */
    int32_t stride, pad;
    int32_t relu;
} fxpq_conv_f32_desc;

/* y[n,p,q,o] = relu?(sum_{r,s,c} x[n, p*st+r-pad, q*st+s-pad, c] * w[o,r,s,c] + bias[o]) in fp32
 * (fused multiply-adds, taps outside the map are zero); w KRSC fp32 [K,R,S,C], bias [K] or NULL. */
FXPQ_API fxpq_status fxpq_conv_f32(const fxpq_conv_f32_desc* h_desc, const float* d_x, const float* d_w,
                                   const float* d_bias, float* d_y, void* stream);
/* k x k max-pool (taps outside the map ignored), element-wise add (+ ReLU), global average pool
 * (fp32 sum over H x W divided by H W); fp32 NHWC. */
FXPQ_API fxpq_status fxpq_maxpool_f32(const float* d_x, int32_t N, int32_t H, int32_t W, int32_t C, int32_t k,
                                      int32_t stride, int32_t pad, float* d_y, void* stream);
FXPQ_API fxpq_status fxpq_eltwise_f32(const float* d_a, const float* d_b, int64_t n, int32_t relu, float* d_y,
                                      void* stream);
FXPQ_API fxpq_status fxpq_avgpool_f32(const float* d_x, int32_t N, int32_t H, int32_t W, int32_t C, float* d_y,
                                      void* stream);
/* fp32 images NCHW -> NHWC (the FP32 network's input). */
FXPQ_API fxpq_status fxpq_nchw_to_nhwc_f32(const float* d_x, int32_t N, int32_t C, int32_t H, int32_t W, float* d_y,
                                           void* stream);
/* Values of an fp16 code tensor [npix, Cp] (planes per fmt.bits) as fp32 [npix, C]: code * 2^-fl
 * (the binary quantizer's codes decoded 0 -> +1 first); exact. */
FXPQ_API fxpq_status fxpq_dequantize(const void* d_codes, int64_t npix, int32_t Cp, int32_t C, fxpq_fmt fmt,
                                     float* d_y, void* stream);
/* In place on fp32 [npix, K]: y += bias[k] (bias may be NULL), then ReLU if relu: the FP32 bias of a
 * layer whose weights are already fixed point (the contraction ran in FXPQ_OUT_F32 mode). */
FXPQ_API fxpq_status fxpq_bias_relu_f32(float* d_y, int64_t npix, int32_t K, const float* d_bias, int32_t relu,
                                        void* stream);
/* Statistics of data-structures, the terms of Eq. CPB_QE (Sec. IV-C), many in one set of launches.
 * Item i: n_samples x nu fp32 values (sample-major) and the QPs under which its error is taken; its
 * record d_out (device double[3 + 2 n_samples]) receives
 *   { L = sum (x - Q(x; fmt))^2 (Eq. DSB_QE, fp64), min, max,
 *     then per sample its mean and its sum of squared deviations from that mean }
 * so that the population deviation of Eq. importance is sqrt(M2 / nu), free of the cancellation
 * of the one-pass form.  Each sum is formed in a fixed order (deterministic, no floating-point
 * atomics).  Items <= 4096, n_samples <= 65535, nu >= 1.  Workspace:
 * fxpq_ds_stats_batch_workspace(items) bytes, 256-byte aligned, scratch. */
typedef struct {
    const float* d_x;   /* device fp32 values, n_samples x nu                                    */
    double* d_out;      /* device record, double[3 + 2 n_samples]                                 */
    int64_t nu;         /* values per sample                                                     */
    int32_t n_samples;  /* samples (1 for a parameter tensor)                                    */
    fxpq_fmt fmt;       /* the QPs of the error L (k = 1..32; k = 1, S = 1 the binary quantizer)  */
} fxpq_ds_item;
FXPQ_API size_t fxpq_ds_stats_batch_workspace(const fxpq_ds_item* h_items, int32_t n_items);
FXPQ_API fxpq_status fxpq_ds_stats_batch(const fxpq_ds_item* h_items, int32_t n_items, void* d_ws, size_t ws_bytes,
                                         void* stream);

/* The cost F = E + UnClass + MisPred of Alg. 1 (Eq. quantization_parameters_optimization) for
 * n_cand candidates at once, on the device.  Term t of candidate c is the fxpq_ds_stats_batch record
 * at d_stats + c * cand_stride + h_terms[t].offset; terms of one layer (equal .layer) share the
 * normaliser of Eq. importance:
 *   sigma_t = mean over samples of sqrt(M2_s / nu), pi_t = sigma_t nu_t / sum over the layer of sigma nu,
 *   E = sum_t pi_t L_t / R_t  (Eq. CPB_QE; R = max - min, Eq. data_range; a term with R = 0 or a
 *       layer with sum sigma nu = 0 adds nothing).
 * d_ties: per candidate N counts |C_i| (fxpq_top1_ties), candidate c at d_ties + c * N:
 *   UnClass = #{i : |C_i| > 1} / N, MisPred = sum (|C_i| - 1) / (N n_classes)
 * (Eqs. unclassified_samples, mispredicted_classes).  d_cost: device double[n_cand][4] =
 * { F, E, UnClass, MisPred }.  n_terms <= 512. */
typedef struct {
    int64_t offset;     /* the term's record, in doubles from the candidate's base               */
    int64_t nu;         /* values per sample                                                     */
    int32_t n_samples;
    int32_t layer;      /* terms with equal layer share the importance normaliser                 */
} fxpq_cost_term;
FXPQ_API fxpq_status fxpq_fopt_cost(const double* d_stats, int64_t cand_stride, const fxpq_cost_term* h_terms,
                                    int32_t n_terms, const int32_t* d_ties, int32_t N, int32_t n_classes,
                                    int32_t n_cand, double* d_cost, void* stream);
/* |C_i| of Eqs. unclassified_samples / mispredicted_classes: per sample the number of classes whose
 * logit equals the largest.  Logits [N, C]: fp32, or exact int64 C-Block values when is_int64. */
FXPQ_API fxpq_status fxpq_top1_ties(const void* d_logits, int32_t is_int64, int32_t N, int32_t C,
                                    int32_t* d_counts, void* stream);

/* Synchronises `stream`, returns and clears the latched device status (FXPQ_OK if none). */
FXPQ_API fxpq_status fxpq_get_device_status(void* stream);

/* Failure-detection check (tests): one thread waits on a shared-memory mbarrier that nothing arrives on,
 * with the same bounded-wait routine that guards every wait of the tensor-core kernels, given up after
 * limit_cycles SM clocks (1 .. 10^8).  The routine latches FXPQ_ERR_TIMEOUT in the device status word
 * and returns, so the next fxpq_get_device_status reports FXPQ_ERR_TIMEOUT (and clears it) and the
 * context stays usable.  No copy or tensor-memory allocation is involved. */
FXPQ_API fxpq_status fxpq_selftest_wait_timeout(int64_t limit_cycles, void* stream);

/* Static English description of a status code. */
FXPQ_API const char* fxpq_status_string(fxpq_status s);

/* Number of kernel launches this library issued since load (instrumentation for benchmarks). */
FXPQ_API int64_t fxpq_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* FXPQ_H */
