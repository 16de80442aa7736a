// fxpq_conv_tc.cu -- host side of the tensor-core C-Block (planning, tensor maps, launch) and the
// kernels without a Scale layer; the kernel itself is in fxpq_conv_tc.cuh.
#include <algorithm>

#include "fxpq_conv_tc.cuh"

namespace fxpq {

using namespace tc;

namespace {

int g_num_sms = 0;
std::mutex g_tc_mu;

// FXPQ_CONV_PATH picks among exact alternatives so that tests can compare them on the same shapes:
// "tc_rows" keeps every layer on 128-row tiles gathered by the producer warps, "tc_patch" takes patch tiles wherever the geometry
// allows them (by default only while they compute few extra rows), "tc_bn128" never takes
// 256-column tiles and "tc_bn256" takes them wherever the layer allows (by default they also need
// enough tiles to keep every SM busy), "tc_win64" keeps window mode's two-limb epilogue in 64-bit
// arithmetic.
bool conv_path_is(const char* name) {
    const char* e = getenv("FXPQ_CONV_PATH");
    return e && strcmp(e, name) == 0;
}
bool g_tc_attr_set = false;

int num_sms() {
    std::lock_guard<std::mutex> lk(g_tc_mu);
    if (g_num_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_num_sms <= 0) g_num_sms = 1;
    }
    return g_num_sms;
}


// Largest |limb| of a format's codes: the only plane (k <= 8) or the hi / lo limb (k > 8).
long long limb_max(const fxpq_fmt& f, int plane) {
    const long long mx = qmax_of(f), mn = -qmin_of(f);
    if (f.bits <= 8) return mx > mn ? mx : mn;
    if (plane == 1) return 255;
    const long long hmx = mx >> 8, hmn = (mn + 255) >> 8;  // |floor(code / 256)|
    return hmx > hmn ? hmx : hmn;
}

}  // namespace

// Builds the group table; returns false if the tensor-core path cannot keep the sums exact.
bool plan_tc(const ConvArgs& a, const fxpq_conv_desc& d, TcParams& P, bool& acc64) {
    P.a = a;
    P.RSC = a.R * a.S * a.Cp;
    const int n_kb = (P.RSC + TC_BK - 1) / TC_BK;
    P.cp64 = (a.Cp % TC_BK) == 0;
    const int pa = planes_of(d.fmt_x), pw = planes_of(d.fmt_w);
    int ng = 0;
    bool shifted = false;
    for (int ia = 0; ia < pa; ++ia)
        for (int iw = 0; iw < pw; ++iw) {
            const long long bound = limb_max(d.fmt_x, ia) * limb_max(d.fmt_w, iw);
            if (bound == 0) continue;
            const long long kmax = ((1LL << 24) - 1) / bound;  // taps per exact fp32 group
            int kb_per = (int)(kmax / TC_BK);
            // every partial sum of channel o is at most max|x limb| * sum_taps |w[o]| <= max|x| * w_l1:
            // below 2^24 the whole reduction is one exact group
            if (d.w_l1 > 0 && d.w_l1 < (1LL << 24) && pw == 1 && limb_max(d.fmt_x, ia) * d.w_l1 < (1LL << 24))
                kb_per = n_kb;
            if (kb_per < 1) return false;
            const int shift = 8 * ((pa - 1 - ia) + (pw - 1 - iw));
            shifted |= shift > 0;
            for (int kb0 = 0; kb0 < n_kb; kb0 += kb_per) {
                if (ng >= TC_MAX_GROUPS) return false;
                P.g[ng++] = TcGroup{kb0, kb0 + kb_per < n_kb ? kb0 + kb_per : n_kb, ia, iw, shift};
            }
        }
    P.n_groups = ng;
    double total = ldexp(1.0, d.fmt_x.bits - d.fmt_x.is_signed) * ldexp(1.0, d.fmt_w.bits - d.fmt_w.is_signed) *
                   (double)a.R * a.S * a.Cp;
    if (d.w_l1 > 0 && pw == 1)
        total = fmin(total, ldexp(1.0, d.fmt_x.bits - d.fmt_x.is_signed) * (double)d.w_l1);
    acc64 = shifted || total >= ldexp(1.0, 31) - 1.0;
    P.status = status_ptr();
    return ng > 0;
}

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link-time driver dependency).
EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    std::lock_guard<std::mutex> lk(g_tc_mu);
    if (!tried) {
        tried = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}
}  // namespace

fxpq_status launch_conv_tc(const ConvArgs& a, const fxpq_conv_desc& d, cudaStream_t st, bool& launched, void* ws,
                           size_t ws_bytes) {
    launched = false;
    TcParams P;
    bool acc64 = false;
    if (!plan_tc(a, d, P, acc64)) return FXPQ_OK;
    const int sms = num_sms();
    // 64-column tiles for int64 sums and for layers with at most 64 output channels; 256-column tiles
    // (one MMA instruction covers twice the work of a 128-column one, which hides its issue cost) for
    // wide layers with enough tiles
    int BN = 128;
    const long long row_tiles_est = (a.M + TC_BM - 1) / TC_BM;
    // Layers whose im2col matrix is the stored activations themselves: 1x1 stride-1 convolutions
    // without padding ([M][Cp] per plane) and kernels covering the whole unpadded map (P = Q = 1,
    // FC layers: [N][H W Cp]).  A 128-row A tile is then one 2-D box of [M][R S Cp].
    const bool one_by_one = a.R == 1 && a.S == 1 && a.stride == 1 && a.pad == 0;
    const bool whole_map = a.R == a.H && a.S == a.W && a.pad == 0 && a.P == 1 && a.Q == 1;
    const bool rows_geom = (one_by_one || whole_map) && a.M > 0 && a.M < (1LL << 31) - TC_BM &&
                           !conv_path_is("tc_rows") && !conv_path_is("tc_patch");
    // ... with few row tiles (FC layers at small batches) they take 256-column tiles and a split
    // reduction fills the SMs: the MMA thread's fixed cost per k-block is then hidden, and the weights
    // stream at the memory's rate
    const bool wide_split = rows_geom && !acc64 && !a.has_scale && ws && a.K > 128 && !conv_path_is("tc_bn128") &&
                            !conv_path_is("tc_nosplit") && row_tiles_est * ((a.K + 255) / 256) * 2 <= sms;
    if (acc64 || a.K <= 64)
        BN = 64;
    else if (wide_split || (a.K > 128 && !conv_path_is("tc_bn128") &&
                            (conv_path_is("tc_bn256") || (a.K % 256 == 0 && row_tiles_est * (a.K / 256) >= sms))))
        BN = 256;
    // packed k-bit weights (k <= 8, one plane) are read by the 256-column TMA-row instances of the
    // split (FC) layers, whose weights stream through once; elsewhere every weight tile is expanded
    // once per row tile and the fp16 codes are read instead
    P.pk = d.d_wpacked && d.fmt_w.bits <= 8 && BN == 256 && wide_split && (reinterpret_cast<uintptr_t>(d.d_wpacked) & 15) == 0 &&
           !conv_path_is("tc_nopack");
    P.wpack = static_cast<const uint32_t*>(d.d_wpacked);
    P.wk = d.fmt_w.bits;
    P.wsigned = d.fmt_w.is_signed;
    P.K_pad = (a.K + 255) / 256 * 256;
    // too few 128-column tiles to occupy every SM (small batches, FC layers): 64-column tiles double
    // the CTA count
    if (BN == 128 && row_tiles_est * ((a.K + 127) / 128) < sms) BN = 64;
    // BN = 256 fills TMEM with two accumulator buffers; with several exact groups per tile it keeps one
    // buffer and the integer running sums
    P.nbuf = (BN == 256 && P.n_groups > 1) ? 1 : 2;
    {
        EncodeTiledFn enc = encode_tiled();
        if (!enc) return FXPQ_OK;  // no tensor-map encoder: the CUDA-core kernel runs instead
        const cuuint64_t dims[3] = {(cuuint64_t)P.RSC, (cuuint64_t)a.K, (cuuint64_t)a.pw};
        const cuuint64_t strides[2] = {(cuuint64_t)P.RSC * 2, (cuuint64_t)a.K * P.RSC * 2};
        const cuuint32_t box[3] = {(cuuint32_t)TC_BK, (cuuint32_t)BN, 1};
        const cuuint32_t es[3] = {1, 1, 1};
        if (enc(&P.tmap_w, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<__half*>(a.w), dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return FXPQ_OK;
        P.patch = 0;
        P.rows_tma = 0;
        P.w32 = 0;
        P.wf32 = 0;
        P.nacc = 1;
        // window mode for 8-channel stride-1 layers with at most 64 output channels: 8 x 16 output
        // patches, one input window per tile and limb plane, weights resident in shared memory, one
        // exact fp32 accumulator per limb pair (R * S2 * 8 products each)
        {
            const int S2 = (a.S + 1) & ~1;
            const int WW = 8 + S2 - 1, WH = 16 + a.R - 1;
            const int win_bytes = (WW * WH * 16 + 127) / 128 * 128;
            bool ok = a.stride == 1 && a.Cp == 8 && a.K <= 64 && a.N > 0 && a.R * S2 <= 16 && 8 * WW <= 256 &&
                      WH <= 256 && a.px * win_bytes <= TC_BM * TC_BK * 2 &&
                      a.pw * a.R * (S2 / 2) * 64 * 32 <= tc_stages(64) * 64 * TC_BK * 2 && !conv_path_is("tc_rows") &&
                      !conv_path_is("tc_nowin");
            for (int ia = 0; ok && ia < a.px; ++ia)
                for (int iw = 0; iw < a.pw; ++iw)
                    if ((double)limb_max(d.fmt_x, ia) * limb_max(d.fmt_w, iw) * a.R * S2 * 8 >= 16777216.0) ok = false;
            if (ok) {
                // the input as [planes][N][H][W * 8]: one window row (WW pixels of 8 channels) is a single
                // 16 WW-byte run of the box rather than WW 16-byte rows
                const cuuint64_t xdims[4] = {(cuuint64_t)a.W * 8, (cuuint64_t)a.H, (cuuint64_t)a.N, (cuuint64_t)a.px};
                const cuuint64_t xstrides[3] = {(cuuint64_t)a.W * 16, (cuuint64_t)a.H * a.W * 16, (cuuint64_t)a.x_ps * 2};
                const cuuint32_t xbox[4] = {(cuuint32_t)(8 * WW), (cuuint32_t)WH, 1, 1};
                // weights as {c, out channel, s, r, plane} (strides in that order, not memory order)
                const cuuint64_t wdims[5] = {8, (cuuint64_t)a.K, (cuuint64_t)a.S, (cuuint64_t)a.R, (cuuint64_t)a.pw};
                const cuuint64_t wstrides[4] = {(cuuint64_t)a.R * a.S * 16, 16, (cuuint64_t)a.S * 16,
                                                (cuuint64_t)a.w_ps * 2};
                const cuuint32_t wbox[5] = {8, 64, 1, 1, 1};  // one tap of one plane
                const cuuint32_t es5[5] = {1, 1, 1, 1, 1};
                CUtensorMap mx, mw;
                if (enc(&mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<__half*>(a.x), xdims, xstrides, xbox, es5,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS &&
                    enc(&mw, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 5, const_cast<__half*>(a.w), wdims, wstrides, wbox, es5,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
                    P.tmap_x = mx;
                    P.tmap_w = mw;
                    P.patch = 3;
                    P.TW = 8;
                    P.TH = 16;
                    P.tiles_p = (a.P + 15) / 16;
                    P.tiles_q = (a.Q + 7) / 8;
                    P.S2 = S2;
                    P.WW = WW;
                    P.WH = WH;
                    P.win_bytes = win_bytes;
                    P.nacc = a.px * a.pw;
                    P.n_groups = 1;
                    P.g[0] = TcGroup{0, 1, 0, 0, 0};
                    P.nbuf = 2;
                    BN = 64;
                    acc64 = true;  // the int64 instance: its TMEM holds two buffers of the limb accumulators
                    // 32-bit epilogue of two-limb x and w (v = 2^16 T + Lo, see the kernel): every limb
                    // sum covers R * S2 * 8 products; L = 2^8 (S_hl + S_lh) + S_ll + Lo(B') and T must stay
                    // below 2^31, the aligned bias must not be finer than the sums (delta >= 0), and
                    // sh - 16 in [0, 30]; the per-channel bias table takes the last 512 bytes of the B region
                    const bool codes32 = a.out_mode == FXPQ_OUT_CODES && a.py == 1 && a.sh >= 16 && a.sh <= 46;
                    const bool image32 = a.out_mode == FXPQ_OUT_F32 && a.K % 4 == 0;  // the fp32 image
                    if (a.px == 2 && a.pw == 2 && !a.has_scale && a.delta >= 0 && (codes32 || image32) &&
                        a.pw * a.R * (S2 / 2) * 64 * 32 + 512 <= tc_stages(64) * 64 * TC_BK * 2) {
                        const double taps = (double)a.R * S2 * 8;
                        const double hh = (double)limb_max(d.fmt_x, 0) * limb_max(d.fmt_w, 0) * taps;
                        const double hl = (double)limb_max(d.fmt_x, 0) * limb_max(d.fmt_w, 1) * taps;
                        const double lh = (double)limb_max(d.fmt_x, 1) * limb_max(d.fmt_w, 0) * taps;
                        const double ll = (double)limb_max(d.fmt_x, 1) * limb_max(d.fmt_w, 1) * taps;
                        const double bb = a.has_bias ? ldexp(1.0, d.fmt_b.bits - d.fmt_b.is_signed + a.delta) : 0.0;
                        const double Lb = 256.0 * (hl + lh) + ll + 65536.0;
                        const double Tb = hh + bb / 65536.0 + 1.0 + Lb / 65536.0 + 1.0;
                        const bool ok32 = Lb < ldexp(1.0, 31) && Tb < ldexp(1.0, 31) && !conv_path_is("tc_win64");
                        P.w32 = ok32 && codes32;
                        P.wf32 = ok32 && image32;
                    }
                }
            }
        }
        // 64-channel window mode (W64 instance) for one-plane stride-1 layers with at most 64 output
        // channels, kernels up to 3 x 3, a reduction of one exact group and one-plane codes out (VGG
        // conv1_2): 8 x 16 output patches, the weights resident (one 8 KiB swizzled block per tap), then
        // two window slots of S copies (shifted by 0 .. S - 1 pixels) of TH + R - 1 rows of 8 pixels
        if (P.patch == 0 && BN == 64 && a.K <= 64 && !acc64 && a.stride == 1 && a.Cp == 64 && a.px == 1 &&
            a.pw == 1 && P.n_groups == 1 && a.N > 0 && a.P > 0 && a.Q > 0 && a.R <= 3 && a.S <= 3 &&
            ((a.out_mode == FXPQ_OUT_CODES && a.py == 1 && (a.v32 || (a.sh >= 1 && a.sh <= 62))) ||
             (a.out_mode == FXPQ_OUT_F32 && a.K % 4 == 0)) &&
            !a.has_scale &&
            !conv_path_is("tc_rows") && !conv_path_is("tc_patch") && !conv_path_is("tc_nowin")) {
            const int WH = 16 + a.R - 1;
            const long long slot = (long long)a.S * WH * 1024;
            const long long wb = (long long)a.R * a.S * 8192;
            if (wb + 2 * slot <= TC_W64_SO) {
                const cuuint64_t xdims[4] = {(cuuint64_t)a.Cp, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.N};
                const cuuint64_t xstrides[3] = {(cuuint64_t)a.Cp * 2, (cuuint64_t)a.W * a.Cp * 2,
                                                (cuuint64_t)a.H * a.W * a.Cp * 2};
                const cuuint32_t xbox[4] = {64, 8, (cuuint32_t)WH, 1};
                const cuuint32_t es4[4] = {1, 1, 1, 1};
                CUtensorMap mx;
                if (enc(&mx, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<__half*>(a.x), xdims, xstrides, xbox, es4,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
                    P.tmap_x = mx;  // the weights keep the tiled map above (box {64, 64}: one tap)
                    P.patch = 4;
                    P.TW = 8;
                    P.TH = 16;
                    P.tiles_p = (a.P + 15) / 16;
                    P.tiles_q = (a.Q + 7) / 8;
                    P.WW = 8;
                    P.WH = WH;
                    P.win_bytes = (int)slot;
                    P.w64_slot0 = (int)wb;
                    P.w64_slot_stride = (int)slot;
                    P.nbuf = 2;
                }
            }
        }
        if (P.patch == 0 && rows_geom) {
            const cuuint64_t xdims[3] = {(cuuint64_t)P.RSC, (cuuint64_t)a.M, (cuuint64_t)a.px};
            const cuuint64_t xstrides[2] = {(cuuint64_t)P.RSC * 2, (cuuint64_t)a.x_ps * 2};
            const cuuint32_t xbox[3] = {(cuuint32_t)TC_BK, (cuuint32_t)TC_BM, 1};
            if (enc(&P.tmap_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<__half*>(a.x), xdims, xstrides, xbox, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS)
                P.rows_tma = 1;
        }
        // patch tiles for stride-1 layers whose taps are whole 64-channel blocks, or 8-channel inputs
        // (a k-block of 8 taps)
        const bool narrow = a.Cp == 8;
        if (P.patch == 0 && !P.rows_tma && a.stride == 1 && (P.cp64 || narrow) && a.P > 0 && a.Q > 0 && a.N > 0 &&
            !conv_path_is("tc_rows")) {
            int best_tw = 0, best_th = 0;
            long long best = 0;
            for (int tw = a.Q < TC_BM ? a.Q : TC_BM; tw >= 1; --tw) {
                const int th = TC_BM / tw < a.P ? TC_BM / tw : a.P;
                const long long cost = (long long)((a.P + th - 1) / th) * ((a.Q + tw - 1) / tw);
                if (best_tw == 0 || cost < best) best = cost, best_tw = tw, best_th = th;
            }
            // take patches unless they need more than twice as many tiles as 128-row tiles of N*P*Q:
            // one TMA box per k-block against 128 gathered rows pays for a good deal of idle MMA rows
            // (3x3 layers, 14x14 maps: 2 patches of 126 rows per image, 1.3x the row tiles, 1.7-2x
            // faster; 7x7 maps: 2.6x the row tiles, 6% slower)
            const long long row_tiles = (a.M + TC_BM - 1) / TC_BM;
            if ((double)a.N * best <= 2.0 * (double)row_tiles + 1e-9 || conv_path_is("tc_patch")) {
                const cuuint64_t xdims[5] = {(cuuint64_t)a.Cp, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.N,
                                             (cuuint64_t)a.px};
                const cuuint64_t xstrides[4] = {(cuuint64_t)a.Cp * 2, (cuuint64_t)a.W * a.Cp * 2,
                                                (cuuint64_t)a.H * a.W * a.Cp * 2, (cuuint64_t)a.x_ps * 2};
                const cuuint32_t xbox[5] = {(cuuint32_t)(narrow ? 8 : TC_BK), (cuuint32_t)best_tw,
                                            (cuuint32_t)best_th, 1, 1};
                const cuuint32_t es5[5] = {1, 1, 1, 1, 1};
                if (enc(&P.tmap_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 5, const_cast<__half*>(a.x), xdims, xstrides,
                        xbox, es5, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        narrow ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS) {
                    P.patch = narrow ? 2 : 1;
                    P.TW = best_tw;
                    P.TH = best_th;
                    P.tiles_p = (a.P + best_th - 1) / best_th;
                    P.tiles_q = (a.Q + best_tw - 1) / best_tw;
                }
            }
        }
        if (!P.rows_tma) P.pk = 0;
        if (P.w32 && !(a.out_mode == FXPQ_OUT_CODES && a.py == 1)) P.w32 = 0;
        if (P.wf32 && a.out_mode != FXPQ_OUT_F32) P.wf32 = 0;
        // one-plane codes: stage the tile in shared memory and write it with TMA stores (not with packed
        // weights, whose staging region holds the packed stages)
        P.fast_store = 0;
        if (a.out_mode == FXPQ_OUT_CODES && a.py == 1 && !P.pk) {
            CUresult r;
            if (P.patch) {
                const cuuint64_t ydims[4] = {(cuuint64_t)a.K, (cuuint64_t)a.Q, (cuuint64_t)a.P, (cuuint64_t)a.N};
                const cuuint64_t ystrides[3] = {(cuuint64_t)a.K * 2, (cuuint64_t)a.Q * a.K * 2,
                                                (cuuint64_t)a.P * a.Q * a.K * 2};
                const cuuint32_t ybox[4] = {64, (cuuint32_t)P.TW, (cuuint32_t)P.TH, 1};
                const cuuint32_t es4[4] = {1, 1, 1, 1};
                r = enc(&P.tmap_y, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, a.y, ydims, ystrides, ybox, es4,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
            } else {
                const cuuint64_t ydims[2] = {(cuuint64_t)a.K, (cuuint64_t)a.M};
                const cuuint64_t ystrides[1] = {(cuuint64_t)a.K * 2};
                const cuuint32_t ybox[2] = {64, (cuuint32_t)TC_BM};
                r = enc(&P.tmap_y, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, a.y, ydims, ystrides, ybox, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
            }
            P.fast_store = r == CUDA_SUCCESS;
        }
        if (!P.fast_store) P.w32 = 0;  // the 32-bit window epilogue writes through the staging tile
    }
    P.tiles_m = P.patch ? a.N * P.tiles_p * P.tiles_q : (int)((a.M + TC_BM - 1) / TC_BM);
    P.tiles_n = (a.K + BN - 1) / BN;
    P.n_tiles = P.tiles_m * P.tiles_n;
    if (P.n_tiles == 0) {
        launched = true;
        return FXPQ_OK;
    }
    // Split reduction for layers whose tiles cannot occupy the SMs (FC layers, small batches) and whose
    // reduction is long: ks units share every tile's k-blocks (share s of every exact group), and their
    // exact integer sums meet in the workspace.
    P.ksplit = 1;
    P.part = nullptr;
    P.gs[0] = 0;
    P.gs[1] = P.n_groups;
    // (64-column tiles, and 256-column TMA-row tiles, without a Scale layer: the instantiations that carry
    // the split)
    if (P.patch != 3 && P.patch != 4 && (BN == 64 || (BN == 256 && P.rows_tma && !acc64)) && !a.has_scale && ws &&
        P.n_tiles * 2 <= sms && !conv_path_is("tc_nosplit")) {
        const int ng = P.n_groups;
        int min_len = 1 << 30;
        for (int gi = 0; gi < ng; ++gi) min_len = std::min(min_len, P.g[gi].kb1 - P.g[gi].kb0);
        const size_t share = (size_t)a.M * a.K * (acc64 ? sizeof(long long) : sizeof(int));
        const int cap = std::min(sms / P.n_tiles, (int)std::min<size_t>(ws_bytes / share, TC_MAX_SPLIT));
        // long groups: each share takes a sub-range of every group (at least four k-blocks); many short
        // groups (two-limb layers): each share takes whole groups
        const int ks_sub = std::min(cap, std::min(min_len / 4, TC_MAX_GROUPS / ng));
        const int ks_whole = std::min(cap, ng);
        if (ks_sub >= 2 && ks_sub >= ks_whole) {
            TcGroup g0[TC_MAX_GROUPS];
            for (int gi = 0; gi < ng; ++gi) g0[gi] = P.g[gi];
            for (int s = 0; s < ks_sub; ++s) {
                for (int gi = 0; gi < ng; ++gi) {
                    const int len = g0[gi].kb1 - g0[gi].kb0;
                    TcGroup g = g0[gi];
                    g.kb0 = g0[gi].kb0 + (int)((long long)len * s / ks_sub);
                    g.kb1 = g0[gi].kb0 + (int)((long long)len * (s + 1) / ks_sub);
                    P.g[s * ng + gi] = g;
                }
                P.gs[s] = s * ng;
            }
            P.gs[ks_sub] = ks_sub * ng;
            P.ksplit = ks_sub;
        } else if (ks_whole >= 2) {
            for (int s = 0; s <= ks_whole; ++s) P.gs[s] = (int)((long long)ng * s / ks_whole);
            P.ksplit = ks_whole;
        }
        if (P.ksplit > 1) {
            P.part = ws;
            P.fast_store = 0;
        }
    }
    P.n_units = P.n_tiles * P.ksplit;
    {
        std::lock_guard<std::mutex> lk(g_tc_mu);
        if (!g_tc_attr_set) {
            if (cudaFuncSetAttribute(conv_tc_kernel<64, long long, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, long long, false, true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, int, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, int, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<64>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<128, int, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<128>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<256, int, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<256>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<256, int, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<256>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<256, int, false, true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<256, true>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<256, int, false, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)tc_smem_bytes<256, true>()) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, long long, false, false, false, true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)(tc_smem_bytes<64>() + 64 * TC_BM * 2)) != cudaSuccess ||
                cudaFuncSetAttribute(conv_tc_kernel<64, int, false, false, false, false, true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)tc_smem_w64()) != cudaSuccess)
                return FXPQ_ERR_CUDA;
            g_tc_attr_set = true;
        }
    }
    const int grid = P.n_units < sms ? P.n_units : sms;
    launched = true;
    if (a.has_scale) return launch_conv_tc_scaled(P, BN, acc64, grid, st);  // never split
    if (P.patch == 3 && (P.w32 || P.wf32))  // window mode, 32-bit two-limb epilogue: its own instance (never split)
        conv_tc_kernel<64, long long, false, false, false, true>
            <<<grid, tc_threads_win(), tc_smem_bytes<64>() + 64 * TC_BM * 2, st>>>(P);
    else if (P.patch == 4 && (P.fast_store || a.out_mode == FXPQ_OUT_F32))
        // 64-channel window mode: the instance with its own shared-memory layout and 16 epilogue warps
        conv_tc_kernel<64, int, false, false, false, false, true><<<grid, tc_threads_win(), tc_smem_w64(), st>>>(P);
    else if (P.patch == 4) {
        launched = false;  // no TMA store of the output: the CUDA-core kernel runs instead
        return FXPQ_OK;
    }
    else if (P.pk && P.ksplit > 1)
        conv_tc_kernel<256, int, false, true, true><<<grid, tc_threads_pk(256, true), tc_smem_bytes<256, true>(), st>>>(P);
    else if (P.pk)
        conv_tc_kernel<256, int, false, false, true><<<grid, tc_threads_pk(256, true), tc_smem_bytes<256, true>(), st>>>(P);
    else if (P.ksplit > 1 && BN == 256)
        conv_tc_kernel<256, int, false, true><<<grid, tc_threads(256), tc_smem_bytes<256>(), st>>>(P);
    else if (P.ksplit > 1 && acc64)
        conv_tc_kernel<64, long long, false, true><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (P.ksplit > 1)
        conv_tc_kernel<64, int, false, true><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (acc64)
        conv_tc_kernel<64, long long, false><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (BN == 64)
        conv_tc_kernel<64, int, false><<<grid, tc_threads(64), tc_smem_bytes<64>(), st>>>(P);
    else if (BN == 128)
        conv_tc_kernel<128, int, false><<<grid, tc_threads(128), tc_smem_bytes<128>(), st>>>(P);
    else
        conv_tc_kernel<256, int, false><<<grid, tc_threads(256), tc_smem_bytes<256>(), st>>>(P);
    launched = true;
    const fxpq_status s = after_launch("conv_tc");
    if (s != FXPQ_OK || P.ksplit == 1) return s;
    return launch_splitk_reduce(a, P.part, P.ksplit, acc64, st);
}

}  // namespace fxpq

// ------------------------------------------------------------------------------------------
// Failure detection: the kernels' bounded mbarrier wait, run on a barrier that nothing arrives on.
// ------------------------------------------------------------------------------------------
namespace {
__global__ void wait_selftest_kernel(long long limit, int* status) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    abort_flag = 0;
    const uint32_t b = fxpq::tc::smem_u32(&bar);
    fxpq::tc::mbar_init(b, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    // phase 0 of the barrier never completes: the wait runs out, latches the status and returns
    fxpq::tc::wait_bounded_for(b, 0, &abort_flag, status, limit);
}
}  // namespace

extern "C" fxpq_status fxpq_selftest_wait_timeout(int64_t limit_cycles, void* stream) {
    if (limit_cycles < 1 || limit_cycles > 100000000LL) return FXPQ_ERR_INVALID_ARG;
    wait_selftest_kernel<<<1, 1, 0, fxpq::as_stream(stream)>>>(limit_cycles, fxpq::status_ptr());
    return fxpq::after_launch("wait_selftest");
}
