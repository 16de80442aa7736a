#pragma once
// fxpq_conv_tc.cuh -- the C-Block contraction (Sec. IV-B) on the 5th-generation tensor cores.
//
// Implicit GEMM: rows = output pixels (N*P*Q), columns = output channels K, reduction over the
// flattened (r, s, c) taps of one code plane.  Operands are fp16 values that are exact integer
// codes (|code| <= 255 per limb), multiplied by tcgen05.mma .kind::f16 into fp32 TMEM
// accumulators.  fp32 accumulation is exact while every partial sum stays below 2^24, so the host
// splits the reduction into groups ("chunks") whose worst-case magnitude max|a| * max|w| * K_chunk
// is below 2^24; after each group the epilogue warps drain the accumulator, convert it to an
// integer (exact) and add it, shifted by the limb weight (0, 8 or 16 bits), into integer running
// sums.  The same grouping carries the two-limb split of 9..16-bit codes
// (v = 256 * v_hi + v_lo): one pass per (A limb, W limb) pair.
//
// CTA (one per SM, persistent over tiles): 9 warps.
//   warps 0-3  producers, into 128-byte swizzled K-major shared-memory stages.  The B tile
//              (BN channels x 64 taps) always comes by TMA.  The A tile takes one of two forms:
//              row tiles (128 consecutive output pixels): cp.async gather by 128 threads, with
//              zero fill for padding and ragged edges;
//              patch tiles (stride 1, Cp % 64 == 0): a TH x TW patch of output pixels of one
//              image, whose input window for one tap and 64 channels is a single 5-D TMA box
//              (the hardware zero-fills the padding); one thread issues both copies.
//   warp  4-7  epilogue: drain TMEM (tcgen05.ld), integer running sums, final bias / ReLU /
//              FxP-QLayer (shared with the CUDA-core kernel).
//   warp  8    TMEM allocation and the single MMA-issuing thread.
// Every wait is bounded: on expiry the kernel latches FXPQ_ERR_TIMEOUT, stops issuing work,
// drains its own copies and MMAs, frees TMEM and returns.
// The kernel is a template over the tile width, the integer type of the running sums and whether
// the layer carries a Scale layer (SC): fxpq_conv_tc.cu instantiates the SC = false kernels and the
// host side, fxpq_conv_tc_scale.cu the SC = true ones, so that the two compile in parallel and the
// Scale layer's epilogue costs the other layers nothing.
#include <cuda.h>  // CUtensorMap and its enums (the encoder is fetched through the runtime)
#include <climits>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "fxpq_common.cuh"
#include "fxpq_conv.cuh"

namespace fxpq {
namespace tc {


constexpr int TC_BM = 128;
constexpr int TC_BK = 64;  // fp16 elements per k-block row = 128 bytes (one swizzle atom row)
// Pipeline depth: 6 stages of 32 KB (BN <= 128); 4 of 48 KB for BN = 256, whose one-plane codes are
// stored through per-warp 2 KB slices (no TMA-store staging of the whole tile) so that the output
// staging keeps only 32 KB; 3 for the packed-weight instance, whose packed stages take the 64 KB
// staging region.  (The 256-column layers lose about a fifth of their speed from 3 stages to 2: the
// copies' latency, not the tensor pipe, bounds them at this depth.)
__host__ __device__ constexpr int tc_stages(int BN, bool PK = false) { return BN == 256 ? (PK ? 3 : 4) : 6; }
// Output staging bytes: BN / 64 boxes of 128 rows x 128 bytes for the TMA-store epilogue, 32 KB where
// the codes are stored directly (BN = 256 without packed weights).
__host__ __device__ constexpr int tc_out_bytes(int BN, bool PK = false) { return (BN == 256 && !PK) ? 32768 : BN * TC_BM * 2; }
// Row-tile producers arrive on a stage this many k-blocks after issuing its copies (cp.async groups
// in flight).  It must stay below the stage count: a producer waiting for a stage to be consumed
// must already have arrived on it.
__host__ __device__ constexpr int tc_lag(int BN, bool PK = false) { return tc_stages(BN, PK) - 1 < 3 ? tc_stages(BN, PK) - 1 : 3; }
// Warps: 4 producers, epilogue warps (four per 32-column chunk group: one per TMEM lane quadrant;
// BN / 8 of them up to 16, each then draining BN / 128 chunks), one MMA / TMEM-allocation warp.
__host__ __device__ constexpr int tc_epi_warps(int BN) { return BN / 8 < 16 ? BN / 8 : 16; }
__host__ __device__ constexpr int tc_threads(int BN) { return (5 + tc_epi_warps(BN)) * 32; }
// Packed weights (PK instances, BN = 256 only): the weights arrive as k-bit records (k <= 8) and these
// extra warps after the MMA warp, with producer warps 1-3, expand every k-block's records into the
// fp16 B stage.  The packed stages live in the output staging region, which PK layers do not use.
constexpr int TC_PK_WARPS = 5;
constexpr int TC_PK_CONVERTERS = 3 + TC_PK_WARPS;  // converter warps
__host__ __device__ constexpr int tc_threads_pk(int BN, bool pk) { return tc_threads(BN) + (pk ? 32 * TC_PK_WARPS : 0); }
// Window-mode instance (WIN, BN = 64, two-limb x and w, 32-bit epilogue): 16 epilogue warps of 16 columns
// each and two output staging tiles.
constexpr int TC_WIN_EPI_WARPS = 16;
// W64 instance (64-channel window mode) shared memory: resident weights (up to 9 taps of 8 KiB) and two
// window slots of up to 3 copies of 18 rows x 8 pixels x 128 bytes from the start, the two staging tiles
// at W64_SO.
constexpr int TC_W64_SO = 180 * 1024;
constexpr size_t tc_smem_w64() { return 1024 + TC_W64_SO + 2 * 64 * TC_BM * 2 + 256; }
__host__ __device__ constexpr int tc_threads_win() { return (5 + TC_WIN_EPI_WARPS) * 32; }
// Dynamic shared memory: barriers, the stages (A and B tiles), the output staging tile.
template <int BN, bool PK = false>
constexpr size_t tc_smem_bytes() {
    return 1024 + tc_stages(BN, PK) * (TC_BM * TC_BK * 2 + BN * TC_BK * 2) + tc_out_bytes(BN, PK) + 256;
}
static_assert(tc_smem_bytes<256>() <= 232448 && tc_smem_bytes<256, true>() <= 232448 && tc_smem_bytes<128>() <= 232448,
              "dynamic shared memory within the 227 KB a CTA may use");
constexpr int TC_MAX_GROUPS = 64;
constexpr int TC_MAX_SPLIT = 16;
constexpr long long TC_WAIT_CYCLES = 4000000000LL;  // ~2 s at 2 GHz
// TMA-issuing threads of patch tiles (lane 0 of warps 0 .. n-1).  Producer p issues the k-blocks of the
// stages s with s % n == p (n divides the stage count), so every use of a stage comes from one thread, in
// order, and its parity wait on the stage's `empty` barrier is never more than one phase ahead of it.
// (A parity wait two phases ahead reads as complete: with k-blocks dealt round-robin, more producers
// than stages could refill a stage before its data was consumed.)
__host__ __device__ constexpr int tc_producers(int BN, bool PK = false) {
    return tc_stages(BN, PK) <= 4 ? tc_stages(BN, PK) : 2;
}

struct TcGroup {
    int kb0, kb1;          // k-block range within a plane
    int a_plane, w_plane;  // limb planes (0 = hi or the only plane, 1 = lo)
    int shift;             // weight of this pass: 0, 8 or 16 bits
};

struct TcParams {
    CUtensorMap tmap_w;  // weights as [planes][K][R*S*Cp] fp16, box {64, BN, 1}, 128-byte swizzle
    CUtensorMap tmap_y;  // output codes: [M][K] box {64, 128} (linear tiles) or [N][P][Q][K] box {64, TW, TH, 1}
    CUtensorMap tmap_x;  // patch tiles: activations [planes][N][H][W][Cp], box {64, TW, TH, 1, 1}; window mode:
                         // [planes][N][H][W * 8], box {8 WW, WH, 1, 1} (a window row is one 16 WW-byte run)
    int fast_store;      // 1: one-plane codes staged in shared memory and written by TMA stores
    int nbuf;            // fp32 accumulator buffers in TMEM: 2, or 1 when BN = 256 needs running sums
    int patch;           // a tile is a TH x TW patch of one image and the A tile comes by TMA:
                         // 1: Cp % 64 == 0 (one 64-channel box per k-block, 128-byte swizzle);
                         // 2: Cp == 8 (one 8-channel box per tap, 8 taps per k-block, no swizzle);
                         // 3: Cp == 8, window mode (one input window per tile and limb plane, taps as
                         //    shifted descriptors, weights resident in shared memory)
                         // 4: Cp == 64, window mode of one-plane layers (W64 instance): the 8 x 16 patch's
                         //    input window, one 128-byte-swizzled TMA box per tile, weights resident,
                         //    every tap and 16-channel step one shifted swizzled MMA
    int rows_tma;        // 128-row tiles whose A tile is one 2-D TMA box of the activations seen as
                         // [planes][M][R*S*Cp] (1x1 stride-1 layers without padding, and kernels that
                         // cover the whole unpadded map: FC layers), box {64, 128, 1}, 128-byte
                         // swizzle, rows past M and taps past R*S*Cp zero filled
    int nacc;            // fp32 accumulators per TMEM buffer (window mode: one per limb pair)
    int WW, WH, S2;      // window mode: window width / height in pixels, taps per row rounded up to even
    int w32;             // window mode, two-limb x and w, one-plane codes out: the 32-bit epilogue (the
                         // host proved its bounds; see the epilogue), with m = sh - 16 in [0, 30]
    int wf32;            // the same window instance writing the fp32 image of v = 2^16 T + Lo
    int win_bytes;       // window mode: bytes of one window (128-byte aligned; patch 4: 16-byte aligned)
    int w64_slot0;       // patch 4: offset of window slot 0 (after the resident weights)
    int w64_slot_stride; // bytes between the two window slots (S copies of WH KiB)
    int TH, TW;          // patch shape (TH * TW = 128)
    int tiles_p, tiles_q;  // patches per image along P and Q
    ConvArgs a;
    int RSC;       // R * S * Cp: reduction length of one plane
    int tiles_m, tiles_n, n_tiles;
    int n_groups;
    // Split reduction: every tile's reduction is shared by ksplit work units, unit share s taking the
    // groups g[gs[s]] .. g[gs[s + 1] - 1] (sub-ranges of every exact group, or whole groups); a unit
    // writes its exact integer sums to part[s][M][K] (ACC) and a second kernel adds the shares and
    // applies the epilogue.  Without a split, gs = {0, n_groups}.
    int ksplit, n_units;
    int gs[TC_MAX_SPLIT + 1];
    void* part;
    int cp64;      // Cp % 64 == 0: a k-block never straddles a tap
    // Packed weights (pk = 1, one plane of wk <= 8 bits, wsigned): fxpq_pack_weights' tiles, words
    // [ceil(R*S*Cp / 64)][K_pad / 256][wk][256][2]: word (kb, t, b, o, h) bit i = bit b of code
    // 64 kb + 32 h + i of output channel 256 t + o.
    const uint32_t* wpack;
    int pk, wk, wsigned, K_pad;
    int* status;
    TcGroup g[TC_MAX_GROUPS];
};

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// The non-blocking probe, for the thread that issues the MMAs: a try_wait there stalls the issuing
// thread until its queued MMAs have drained (about 230 cycles per k-block of four 128-column MMAs, half
// the tensor rate), a test_wait costs about 45.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

// 2-D tiled TMA store from shared memory (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void tma_store_4d(const CUtensorMap* map, int x, int y, int z, int w, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%1, %2, %3, %4}], [%5];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y), "r"(z), "r"(w), "r"(src)
                 : "memory");
}

// 5-D tiled TMA load completing on mbarrier `bar` (coordinates innermost first; out-of-range
// positions, e.g. the convolution's padding, read as zero).
__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            int c4, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, "
        "%5, %6}], [%7];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(bar)
        : "memory");
}

// 4-D tiled TMA load (coordinates innermost first) completing on mbarrier `bar`.
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, "
        "%5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

// Output row (linear index into N*P*Q, or -1 when outside the map) of tile row i.
__device__ __forceinline__ long long tile_row(const TcParams& P, int tm, int i) {
    if (!P.patch) {
        const long long m = (long long)tm * 128 + i;
        return m < P.a.M ? m : -1;
    }
    if (i >= P.TH * P.TW) return -1;
    const int per_img = P.tiles_p * P.tiles_q;
    const int n = tm / per_img, r = tm - n * per_img;
    const int p = (r / P.tiles_q) * P.TH + i / P.TW, q = (r % P.tiles_q) * P.TW + i % P.TW;
    if (p >= P.a.P || q >= P.a.Q) return -1;
    return ((long long)n * P.a.P + p) * P.a.Q + q;
}

// 3-D tiled TMA load (coordinates innermost first) completing on mbarrier `bar`.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// 1-D bulk copy global -> shared completing on mbarrier `bar` (both addresses 16-byte aligned, bytes a
// multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Bit-plane bytes -> fp16 codes.  (lo, hi): an 8 x 8 bit matrix, byte b = plane b (bytes 0-3 in lo,
// 4-7 in hi), bit c = code c of eight consecutive codes.  Three delta swaps transpose it (Hacker's
// Delight, 7-3: byte c then holds code c's k bits).  Signed codes have bit k-1 flipped (`flip`), which
// maps them to u = code + 2^(k-1) in [0, 2^k); each byte then becomes the fp16 1024 + u (exponent
// byte 0x64, u in the mantissa) and one half2 subtraction of `off` = 1024 (+ 2^(k-1) if signed)
// leaves the code itself, exactly.  Returns the 16-byte chunk of the eight fp16 codes.
__device__ __forceinline__ uint4 planes_to_f16(uint32_t lo, uint32_t hi, uint32_t flip, uint32_t off) {
    uint32_t t;
    t = (lo ^ (lo >> 7)) & 0x00AA00AAu;
    lo ^= t ^ (t << 7);
    t = (hi ^ (hi >> 7)) & 0x00AA00AAu;
    hi ^= t ^ (t << 7);
    t = (lo ^ (lo >> 14)) & 0x0000CCCCu;
    lo ^= t ^ (t << 14);
    t = (hi ^ (hi >> 14)) & 0x0000CCCCu;
    hi ^= t ^ (t << 14);
    t = (lo ^ (hi << 4)) & 0xF0F0F0F0u;  // the 4 x 4 blocks across the two words
    lo ^= t;
    hi ^= t >> 4;
    lo ^= flip;
    hi ^= flip;
    const __half2 o2 = *reinterpret_cast<const __half2*>(&off);
    uint32_t h[4] = {__byte_perm(lo, 0x64646464u, 0x5140), __byte_perm(lo, 0x64646464u, 0x5342),
                     __byte_perm(hi, 0x64646464u, 0x5140), __byte_perm(hi, 0x64646464u, 0x5342)};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const __half2 v = __hsub2(*reinterpret_cast<const __half2*>(&h[q]), o2);
        h[q] = *reinterpret_cast<const uint32_t*>(&v);
    }
    return make_uint4(h[0], h[1], h[2], h[3]);
}

// 4 x 4 byte transpose: out[m] byte b = in[b] byte m.
__device__ __forceinline__ void byte_transpose4(const uint32_t (&in)[4], uint32_t (&out)[4]) {
    const uint32_t t0 = __byte_perm(in[0], in[1], 0x5140), t1 = __byte_perm(in[0], in[1], 0x7362);
    const uint32_t t2 = __byte_perm(in[2], in[3], 0x5140), t3 = __byte_perm(in[2], in[3], 0x7362);
    out[0] = __byte_perm(t0, t2, 0x5410);
    out[1] = __byte_perm(t0, t2, 0x7632);
    out[2] = __byte_perm(t1, t3, 0x5410);
    out[3] = __byte_perm(t1, t3, 0x7632);
}

// Expands one k-block's packed tile (`pk`: k bit planes of BN rows x 2 words, word (b, o, h) at
// 2 (b BN + o) + h, bit i = bit b of code 32 h + i of row o) into the fp16 B stage `sb` (BN rows of
// 128 bytes, 128-byte swizzle: chunk j of row o at 16 ((j ^ o) & 7)).  Thread tid of nthreads takes
// rows tid, tid + nthreads, ...: one 8-byte load per plane (consecutive rows: no bank conflicts), then
// eight chunks.
template <int BN>
__device__ __forceinline__ void pk_convert_stage(const uint32_t* pk, unsigned char* sb, int k, uint32_t flip,
                                                 uint32_t off, int tid, int nthreads) {
    for (int o = tid; o < BN; o += nthreads) {
        uint32_t w[2][8];
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            uint2 v = make_uint2(0u, 0u);
            if (b < k) v = *reinterpret_cast<const uint2*>(pk + 2 * (b * BN + o));
            w[0][b] = v.x;
            w[1][b] = v.y;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            uint32_t lo[4], hi[4];
            byte_transpose4({w[h][0], w[h][1], w[h][2], w[h][3]}, lo);
            byte_transpose4({w[h][4], w[h][5], w[h][6], w[h][7]}, hi);
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const int j = 4 * h + m;
                *reinterpret_cast<uint4*>(sb + o * 128 + ((j ^ (o & 7)) << 4)) = planes_to_f16(lo[m], hi[m], flip, off);
            }
        }
    }
}

// Bounded wait for the phase of `bar` with the given parity.  Returns false (and latches the
// timeout status, sets the CTA abort flag) if it gave up or another role already aborted.
// TEST: the first probe does not block (the MMA-issuing thread's fast path); the retries suspend in
// try_wait rather than spin, which would take issue slots from the epilogue warps.
template <bool TEST = false>
__device__ __forceinline__ bool wait_bounded_for(uint32_t bar, uint32_t parity, volatile int* abort, int* status,
                                                 long long limit) {
    if (TEST ? mbar_test_wait(bar, parity) : mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (clock64() - t0 > limit) {
            *abort = 1;
            latch_status(status, FXPQ_ERR_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort, int* status) {
    return wait_bounded_for(bar, parity, abort, status, TC_WAIT_CYCLES);
}
// the same for the MMA-issuing thread (a non-blocking first probe)
__device__ __forceinline__ bool wait_mma(uint32_t bar, uint32_t parity, volatile int* abort, int* status) {
    return wait_bounded_for<true>(bar, parity, abort, status, TC_WAIT_CYCLES);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
// Shared-memory matrix descriptor, K-major without swizzle: core matrices of 8 rows x 16 bytes;
// lbo = bytes between core matrices adjacent in K, sbo = bytes between 8-row groups.
__device__ __forceinline__ uint64_t make_sdesc_noswz(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1u << 46;  // descriptor version; layout type 0 = no swizzle
    return d;
}

__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);          // start address
    d |= (uint64_t)1u << 16;                          // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024u >> 4) << 32;                // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1u << 46;                          // descriptor version
    d |= (uint64_t)2u << 61;                          // SWIZZLE_128B
    return d;
}

// Instruction descriptor, kind::f16: fp16 A and B (K-major), fp32 accumulator, M x N.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N) {
    return (1u << 4)                        // D format F32
           | (0u << 7) | (0u << 10)         // A, B format F16
           | ((uint32_t)(N >> 3) << 17)     // N / 8
           | ((uint32_t)(M >> 4) << 24);    // M / 16
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// Loads / stores without their completion wait, so that several TMEM accesses share one round trip.
// After tmem_wait_ld(), reg_fence() on each loaded array orders every use of its registers after the
// wait (the empty asm redefines them).
__device__ __forceinline__ void tmem_ld16_nw(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void reg_fence(uint32_t (&r)[N]) {
#pragma unroll
    for (int i = 0; i < N; ++i) asm volatile("" : "+r"(r[i]));
}
__device__ __forceinline__ void tmem_st16_nw(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}
// Final epilogue of 32 consecutive output channels k0.. of row m (generic outputs: two-plane codes,
// int64 accumulators, fp32 calibration images): bias alignment, ReLU, FxP-QLayer.
template <typename ACC, bool SC>
__device__ __forceinline__ void epilogue_block32(const ConvArgs& a, long long m, int k0, const ACC (&acc)[32]) {
    if (a.out_mode == FXPQ_OUT_CODES) {
        __half* y = static_cast<__half*>(a.y);
        const long long base = m * a.K + k0;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int k = k0 + j;
            if (k < a.K) {
                const int32_t b = a.has_bias ? __ldg(a.bias + k) : 0;
                code_put(y, base + j, a.py, a.M * a.K, qlayer_code(a, cblock_value<SC>(a, k, (long long)acc[j], b)));
            }
        }
    } else if (a.out_mode == FXPQ_OUT_ACC64) {
        long long* y = static_cast<long long*>(a.y) + m * a.K + k0;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int k = k0 + j;
            if (k < a.K) y[j] = cblock_value<SC>(a, k, (long long)acc[j], a.has_bias ? __ldg(a.bias + k) : 0);
        }
    } else {
        float* y = static_cast<float*>(a.y) + m * a.K + k0;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int k = k0 + j;
            if (k < a.K)
                y[j] = __ll2float_rn(cblock_value<SC>(a, k, (long long)acc[j], a.has_bias ? __ldg(a.bias + k) : 0)) *
                       a.f32_scale;
        }
    }
}

// The same for fp32-image and int64 outputs through a 2 KiB shared-memory slice of the warp (`wbuf`): every
// round each lane puts 64 bytes of its row there (16-byte pieces rotated against bank conflicts), then the
// warp writes 16-byte pieces of whole row segments, eight rows per instruction, rather than 32 rows at one
// value per lane.  All 32 lanes take part; rows with m < 0 (outside the output) store nothing.  Needs K %
// 4 == 0 (fp32) or K % 2 == 0 (int64), so that a 16-byte piece is wholly inside or past K.
template <typename ACC, bool SC>
__device__ __forceinline__ void epilogue_block32_staged(const ConvArgs& a, long long m, int k0, const ACC (&acc)[32],
                                                        unsigned char* wbuf, int lane) {
    const bool f32 = a.out_mode == FXPQ_OUT_F32;
    const int per = f32 ? 16 : 8;  // values per round: 64 bytes of a row
#pragma unroll
    for (int c0 = 0; c0 < 32; c0 += 8) {
        if (c0 % per) continue;  // fp32 rounds start at 0 and 16
        uint32_t wv[16];
        if (f32) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int k = k0 + c0 + j;
                float v = 0.0f;
                if (m >= 0 && k < a.K && c0 + j < 32)
                    v = __ll2float_rn(cblock_value<SC>(a, k, (long long)acc[(c0 + j) & 31], a.has_bias ? __ldg(a.bias + k) : 0)) *
                        a.f32_scale;
                wv[j] = __float_as_uint(v);
            }
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int k = k0 + c0 + j;
                long long v = 0;
                if (m >= 0 && k < a.K) v = cblock_value<SC>(a, k, (long long)acc[c0 + j], a.has_bias ? __ldg(a.bias + k) : 0);
                wv[2 * j] = (uint32_t)(unsigned long long)v;
                wv[2 * j + 1] = (uint32_t)((unsigned long long)v >> 32);
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q)
            *reinterpret_cast<uint4*>(wbuf + lane * 64 + 16 * (q ^ ((lane >> 1) & 3))) =
                make_uint4(wv[4 * q], wv[4 * q + 1], wv[4 * q + 2], wv[4 * q + 3]);
        __syncwarp();
#pragma unroll
        for (int it = 0; it < 4; ++it) {
            const int r = (lane >> 2) + 8 * it, pc = lane & 3;
            const long long mr = __shfl_sync(0xffffffffu, m, r);
            const uint4 v = *reinterpret_cast<const uint4*>(wbuf + r * 64 + 16 * (pc ^ ((r >> 1) & 3)));
            const int kk = k0 + c0 + pc * (f32 ? 4 : 2);
            if (mr >= 0 && kk < a.K) {
                if (f32)
                    *reinterpret_cast<uint4*>(static_cast<float*>(a.y) + mr * a.K + kk) = v;
                else
                    *reinterpret_cast<uint4*>(static_cast<long long*>(a.y) + mr * a.K + kk) = v;
            }
        }
        __syncwarp();
    }
}

// Uniform constants of the 32-bit FxP-QLayer epilogue (the same arithmetic as qlayer_code32, with
// the bias alignment split into a left and a right shift so that it has no branches).
struct Epi32 {
    int bsl, bsr, fmask;  // bias term (b << bsl) >> bsr; fraction bits b & fmask (bias finer than acc)
    int sh, hm1;          // requantizing right shift and 2^(sh-1) - 1
    int floor;            // 0 with ReLU, INT_MIN without
    int lo, hi;
    int has_bias;
};

__host__ __device__ __forceinline__ Epi32 make_epi32(const ConvArgs& a) {
    Epi32 e;
    e.bsl = a.bsh > 0 ? a.bsh : 0;
    e.bsr = a.bsh < 0 ? -a.bsh : 0;
    e.fmask = (1 << e.bsr) - 1;
    e.sh = a.sh32;
    e.hm1 = (1 << (a.sh32 - 1)) - 1;
    e.floor = a.relu ? 0 : INT_MIN;
    e.lo = (int)a.lo;
    e.hi = (int)a.hi;
    e.has_bias = a.has_bias;
    return e;
}

// One code: N = acc + aligned bias; ReLU; N / 2^sh rounded half to even, then clipped.  With
// q = floor(N / 2^sh) and x = (q & 1) | phi, floor((N + 2^(sh-1) - 1 + x) / 2^sh) is q + 1 exactly
// when the remainder is above one half, or equal to it with q odd or phi set (phi: the bias had
// nonzero bits below the accumulator's scale, so the true value lies above the tie).  After a ReLU
// clamp N = 0 and the sum stays below 2^sh whatever phi is.  The host keeps |N| + 2^(sh-1) < 2^31.
__host__ __device__ __forceinline__ int epi32_code(const Epi32& e, int acc, int bterm, int phi) {
    const int N = max(acc + bterm, e.floor);
    const int x = ((N >> e.sh) & 1) | phi;
    return min(max((N + e.hm1 + x) >> e.sh, e.lo), e.hi);
}

// The same FxP-QLayer on 64-bit values (wide sums, two-limb layers, Scale layers), valid for
// 1 <= sh <= 62: the bias alignment is v = (acc << dr) + (B << dl) (one of dl, dr is zero), a Scale
// layer (SC) makes it ((v * aleph1) << dr2) + (aleph2 << dl2), and the code is
// round_half_even(v / 2^sh) = floor((v + 2^(sh-1) - 1 + ((v >> sh) & 1)) / 2^sh), clipped.  The host
// keeps |v| < 2^62 at every step, so neither the product nor the rounding sum can overflow.
struct Epi64 {
    int dl, dr, sh;
    long long hm1, floor;
    int lo, hi, has_bias, ok;  // ok: 1 <= sh <= 62 (otherwise the generic path runs)
    int dl2, dr2;
};

__host__ __device__ __forceinline__ Epi64 make_epi64(const ConvArgs& a) {
    Epi64 e;
    e.dl = a.delta > 0 ? a.delta : 0;
    e.dr = a.delta < 0 ? -a.delta : 0;
    e.sh = a.sh;
    e.ok = a.sh >= 1 && a.sh <= 62;
    e.hm1 = e.ok ? (1LL << (a.sh - 1)) - 1 : 0;
    e.floor = a.relu ? 0LL : LLONG_MIN;
    e.lo = (int)a.lo;
    e.hi = (int)a.hi;
    e.has_bias = a.has_bias;
    e.dl2 = a.delta2 > 0 ? a.delta2 : 0;
    e.dr2 = a.delta2 < 0 ? -a.delta2 : 0;
    return e;
}

// m, h: aleph1 and aleph2 codes of the channel (read only when SC)
template <bool SC>
__host__ __device__ __forceinline__ int epi64_code(const Epi64& e, long long acc, int32_t b, int32_t m, int32_t h) {
    long long v = (acc << e.dr) + ((long long)b << e.dl);
    if (SC) v = ((v * (long long)m) << e.dr2) + ((long long)h << e.dl2);
    v = max(v, e.floor);
    const long long c = (v + e.hm1 + ((v >> e.sh) & 1)) >> e.sh;
    return (int)min(max(c, (long long)e.lo), (long long)e.hi);
}

// aleph1 / aleph2 codes of channel k for the SC epilogue (0 past K)
__device__ __forceinline__ int32_t scale_code(const ConvArgs& a, int k) { return k < a.K ? __ldg(a.scale + k) : 0; }
__device__ __forceinline__ int32_t shift_code(const ConvArgs& a, int k) { return k < a.K ? __ldg(a.shift + k) : 0; }

// Two codes in [-512, 511] as a packed fp16 pair: 1536 + c has the bit pattern 0x6600 + c (the
// binade [1024, 2048) has unit spacing), and one packed subtraction of 1536 leaves c exactly.
__device__ __forceinline__ uint32_t pack_codes_f16(int c0, int c1) {
    // 0x6600 + c0 >= 0x6400 never borrows from the high half
    const uint32_t bits = (uint32_t)c1 * 65536u + (uint32_t)c0 + 0x66006600u;
    const __half2 h = __hsub2(*reinterpret_cast<const __half2*>(&bits), __halves2half2(__ushort_as_half(0x6600),
                                                                                        __ushort_as_half(0x6600)));
    return *reinterpret_cast<const uint32_t*>(&h);
}

// ------------------------------------------------------------------ kernel
// PK converter warp `cid` (of TC_PK_CONVERTERS): walks the same k-block sequence as the issuing thread;
// for each k-block waits until its A box and packed records have landed (pkfull), expands its share of
// the records into the B stage, makes the writes visible to the tensor cores' async proxy and arrives
// on the stage's full barrier (one arrival per warp).
template <int BN, bool SPLIT>
__device__ __forceinline__ void pk_convert_loop(const TcParams& P, int cid, int lane, const unsigned char* sP,
                                                unsigned char* sB, uint32_t pkfull0, uint32_t full0, volatile int* abort) {
    constexpr int STAGES = tc_stages(BN, true);
    constexpr int B_BYTES = BN * TC_BK * 2;
    const int k = P.wk;
    const uint32_t flip = P.wsigned ? 0x01010101u * (1u << (k - 1)) : 0u;
    const uint32_t o1 = 0x6400u + (P.wsigned ? (1u << (k - 1)) : 0u);  // fp16 bits of 1024 (+ 2^(k-1))
    const uint32_t off = o1 | (o1 << 16);
    uint32_t it = 0;
    for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles); ut += gridDim.x) {
        const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
        (void)t;
        (void)sp;
        for (int gi = SPLIT ? P.gs[sp] : 0; gi < (SPLIT ? P.gs[sp + 1] : P.n_groups); ++gi) {
            for (int kb = P.g[gi].kb0; kb < P.g[gi].kb1; ++kb, ++it) {
                const uint32_t stage = it % STAGES, phase = (it / STAGES) & 1;
                if (!wait_bounded(pkfull0 + 8 * stage, phase, abort, P.status)) return;
                pk_convert_stage<BN>(reinterpret_cast<const uint32_t*>(sP + stage * (BN * 64)), sB + stage * B_BYTES, k,
                                     flip, off, cid * 32 + lane, TC_PK_CONVERTERS * 32);
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(full0 + 8 * stage);
            }
        }
    }
}

// SPLIT: the instantiation that runs split reductions (P.ksplit >= 1, unit share ranges P.gs); without it
// the unit loop is the tile loop and every tile takes all P.n_groups groups.
// PK: the instantiation that reads packed k-bit weights (P.pk = 1; BN = 256, TMA A tiles, no output
// staging): one thread issues every copy and TC_PK_CONVERTERS warps expand the weights.
// WIN: the window-mode instance of the 32-bit two-limb epilogue (P.patch == 3, P.w32): 16 epilogue warps and
// two staging tiles; only window mode's roles are compiled into it.
// W64: the same for the 64-channel window mode (P.patch == 4) with one-plane codes out.
template <int BN, typename ACC, bool SC, bool SPLIT = false, bool PK = false, bool WIN = false, bool W64 = false>
__global__ void __launch_bounds__((WIN || W64) ? tc_threads_win() : tc_threads_pk(BN, PK), 1)
    conv_tc_kernel(const __grid_constant__ TcParams P) {
    constexpr int TC_STAGES = tc_stages(BN, PK);
    constexpr int TC_LAG = tc_lag(BN, PK);
    // 256-column tiles without packed weights store their one-plane codes with plain stores through
    // each warp's 2 KB slice of the staging region rather than by TMA stores of a whole staged tile
    constexpr bool DIRECT = BN == 256 && !PK;
    static_assert(TC_LAG >= 1 && TC_LAG < TC_STAGES, "producer lag must be below the stage count");
    static_assert(!PK || (BN == 256 && sizeof(ACC) == 4 && !SC), "packed weights: 256-column int32 tiles only");
    static_assert(!PK || TC_STAGES * BN * 64 <= tc_out_bytes(BN, PK), "packed stages must fit the staging region");
    // PK: one issuing thread (producer warp 0), so its stage waits are in order by construction
    constexpr int TC_PRODUCERS = PK ? 1 : tc_producers(BN, PK);
    static_assert(TC_STAGES % TC_PRODUCERS == 0 && TC_PRODUCERS <= 4,
                  "each stage must have one producer thread among warps 0..3");
    static_assert(!WIN || (BN == 64 && sizeof(ACC) == 8 && !SC && !SPLIT && !PK), "window instance: BN = 64, int64");
    static_assert(!W64 || (BN == 64 && sizeof(ACC) == 4 && !SC && !SPLIT && !PK && !WIN), "W64 instance: BN = 64, int32");
    constexpr bool WEPI = WIN || W64;  // the window instances' epilogue (16 warps, two staging tiles)
    constexpr int EPI_WARPS = WEPI ? TC_WIN_EPI_WARPS : tc_epi_warps(BN);
    constexpr int EPI_THREADS = 32 * EPI_WARPS;
    static_assert(WEPI || tc_out_bytes(BN, PK) >= EPI_WARPS * 2048, "the staged fp32 / int64 epilogue takes 2 KB per warp");
    constexpr int MMA_WARP = 4 + EPI_WARPS;
    constexpr int CPW = WEPI ? 1 : (BN / 32) / (EPI_WARPS / 4);  // 32-column chunks per epilogue warp
    constexpr int A_BYTES = TC_BM * TC_BK * 2;  // 16 KB
    constexpr int B_BYTES = BN * TC_BK * 2;
    constexpr uint32_t IDESC = make_idesc(TC_BM, BN);
    // fp32 accumulator buffers + integer running sums, rounded up to a power of two (BN = 256: two
    // buffers without running sums, or one buffer with them)
    // (the int64 instance also serves window mode: two buffers of up to four limb-pair accumulators)
    constexpr uint32_t USED_COLS = (BN == 256 || sizeof(ACC) == 8) ? 512u : 2 * BN + BN * (uint32_t)(sizeof(ACC) / 4);
    constexpr uint32_t TMEM_COLS = USED_COLS <= 256 ? 256u : 512u;
    extern __shared__ unsigned char smem_raw[];
    unsigned char* base = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    unsigned char* sA = base;
    unsigned char* sB = base + TC_STAGES * A_BYTES;
    unsigned char* sO = W64 ? base + TC_W64_SO : sB + TC_STAGES * B_BYTES;  // output staging: BN/64 halves of
                                                                         // [128 rows][64 codes]
    uint64_t* bars = reinterpret_cast<uint64_t*>(sO + (WEPI ? 2 * BN * TC_BM * 2 : tc_out_bytes(BN, PK)));  // WEPI: two staging tiles
    // bars: full[STAGES], empty[STAGES], accfull[2], accempty[2], done
    volatile int* abort = reinterpret_cast<volatile int*>(bars + 2 * TC_STAGES + 5);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * TC_STAGES + 6);
    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + TC_STAGES);
    const uint32_t accfull0 = smem_u32(bars + 2 * TC_STAGES), accempty0 = smem_u32(bars + 2 * TC_STAGES + 2);
    const uint32_t done_bar = smem_u32(bars + 2 * TC_STAGES + 4);
    const uint32_t stg_full = smem_u32(bars + 2 * TC_STAGES + 7);  // staging written by every epilogue warp
    const uint32_t stg_free = smem_u32(bars + 2 * TC_STAGES + 8);  // staging read by the previous TMA store
    const uint32_t wbar = smem_u32(bars + 2 * TC_STAGES + 9);      // window mode: resident weights loaded
    const uint32_t stg_full2 = smem_u32(bars + 2 * TC_STAGES + 10);  // WIN: the second staging tile
    const uint32_t stg_free2 = smem_u32(bars + 2 * TC_STAGES + 11);
    // PK: pkfull[s] completes when stage s's A box and packed weight records have landed; the
    // converters then fill the B stage and arrive on full[s]
    const uint32_t pkfull0 = smem_u32(bars + 2 * TC_STAGES + 10);
    unsigned char* sP = sO;  // PK: packed stages of BN * 64 bytes (k <= 8 words per 32 codes)

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const ConvArgs& a = P.a;

    if (threadIdx.x == 0) {
        for (int s = 0; s < TC_STAGES; ++s) {
            // patch tiles: one expect_tx arrival for both TMAs; row tiles: one arrival per producer
            // warp + the weight TMA's expect_tx
            mbar_init(full0 + 8 * s, PK ? TC_PK_CONVERTERS : (P.patch || P.rows_tma) ? 1 : 4 + 1);
            mbar_init(empty0 + 8 * s, 1);
            if (PK) mbar_init(pkfull0 + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accfull0 + 8 * b, 1);
            mbar_init(accempty0 + 8 * b, EPI_WARPS);  // one arrival per epilogue warp
        }
        mbar_init(done_bar, 1);
        mbar_init(stg_full, EPI_WARPS);
        mbar_init(stg_free, 1);
        if (WEPI) {
            mbar_init(stg_full2, EPI_WARPS);
            mbar_init(stg_free2, 1);
        }
        mbar_init(wbar, 1);
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == MMA_WARP) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(TMEM_COLS));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    // window mode, 32-bit epilogue: per output channel the aligned bias B' = b 2^delta split as
    // (B' >> 16, B' & 0xFFFF), in the last 512 bytes of the B region (the resident weights stay below)
    int2* wtab = reinterpret_cast<int2*>(sB + TC_STAGES * B_BYTES - 512);
    if (BN == 64 && sizeof(ACC) == 8 && !SC && P.patch == 3 && (P.w32 || P.wf32) && warp == 1) {
        for (int k = lane; k < 64; k += 32) {
            const long long bb = (a.has_bias && k < a.K) ? ((long long)__ldg(a.bias + k) << (a.delta > 0 ? a.delta : 0)) : 0;
            wtab[k] = make_int2((int)(bb >> 16), (int)(bb & 0xFFFF));
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (!WIN && warp < 4 && P.patch == 4) {
        // ============================================================ producer, 64-channel window mode
        // The weights, one 128-byte-swizzled box {64 ch, 64 out ch} per tap (8 KiB, the layout of a B
        // stage), are loaded once to the start of shared memory.  Per tile and tap column s, the input
        // window of the 16 x 8 patch shifted by s pixels, TH + R - 1 rows of 8 pixels of 64 channels (one
        // swizzle pattern per row, padding zero filled), is one box into window slot (tile count mod 2):
        // every tap's A operand then starts on a pattern boundary.
        if (threadIdx.x == 0) {
            mbar_arrive_expect_tx(wbar, (uint32_t)(a.R * a.S) * 8192u);
            for (int t = 0; t < a.R * a.S; ++t)
                tma_load_3d(smem_u32(sA) + (uint32_t)t * 8192u, &P.tmap_w, t * TC_BK, 0, 0, wbar);
            const uint32_t copyb = (uint32_t)P.WH * 1024u;
            const int per_img = P.tiles_p * P.tiles_q;
            uint32_t it = 0, stage = 0, phase = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < P.n_tiles && ok; t += gridDim.x) {
                const int n_img = t / per_img, r = t - n_img * per_img;
                const int hp0 = (r / P.tiles_q) * P.TH - a.pad, wq0 = (r % P.tiles_q) * P.TW - a.pad;
                if (!wait_bounded(empty0 + 8 * stage, phase ^ 1, abort, P.status)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = full0 + 8 * stage;
                mbar_arrive_expect_tx(fb, (uint32_t)a.S * copyb);
                const uint32_t dst = smem_u32(sA) + (uint32_t)P.w64_slot0 + stage * (uint32_t)P.w64_slot_stride;
                for (int q = 0; q < a.S; ++q) tma_load_4d(dst + (uint32_t)q * copyb, &P.tmap_x, 0, wq0 + q, hp0, n_img, fb);
                ++it;
                if (++stage == 2) {
                    stage = 0;
                    phase ^= 1;
                }
            }
            const uint32_t from = it >= 2 ? it - 2 : 0;
            for (uint32_t j = from; j < it; ++j) {
                const long long t0 = clock64();
                while (!mbar_try_wait(full0 + 8 * (j % 2), (j / 2) & 1) && clock64() - t0 < TC_WAIT_CYCLES) {
                }
            }
            const long long t0 = clock64();
            while (!mbar_try_wait(wbar, 0) && clock64() - t0 < TC_WAIT_CYCLES) {
            }
        }
    } else if (!W64 && warp < 4 && P.patch == 3) {
        // ============================================================ producer, window mode
        // Stride 1, Cp == 8: the weights are loaded once into the B region, per kernel row r and tap
        // pair sp a block of the two taps, each tap the BN output channels of every limb plane in turn
        // (rows [W_hi | W_lo] of one B operand of N = pw BN: one MMA forms both limb sums of an x limb;
        // one box {8 ch, BN out ch} per tap and plane, taps past S zero filled); per tile, one box per
        // x limb plane holds the input window of TH + R - 1 rows by TW + S2 - 1 pixels (padding zero
        // filled).
        if (threadIdx.x == 0) {
            const int np = P.S2 / 2;
            const uint32_t tapb = (uint32_t)(BN * 16);  // one tap of one plane
            mbar_arrive_expect_tx(wbar, (uint32_t)(a.pw * a.R * np * 2) * tapb);
            for (int r = 0; r < a.R; ++r)
                for (int t = 0; t < 2 * np; ++t)
                    for (int iw = 0; iw < a.pw; ++iw)
                        tma_load_5d(smem_u32(sB) + (uint32_t)(((r * np + t / 2) * 2 + (t & 1)) * a.pw + iw) * tapb,
                                    &P.tmap_w, 0, 0, t, r, iw, wbar);
            const uint32_t win_tx = (uint32_t)(P.WW * P.WH * 16);
            const int per_img = P.tiles_p * P.tiles_q;
            uint32_t it = 0, stage = 0, phase = 0;
            bool ok = true;
            for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
                const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
                (void)sp;
                const int tm = t / P.tiles_n;
                const int n_img = tm / per_img, r = tm - n_img * per_img;
                const int hp0 = (r / P.tiles_q) * P.TH - a.pad, wq0 = (r % P.tiles_q) * P.TW - a.pad;
                if (!wait_bounded(empty0 + 8 * stage, phase ^ 1, abort, P.status)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = full0 + 8 * stage;
                mbar_arrive_expect_tx(fb, (uint32_t)a.px * win_tx);
                // (pixels and channels of a row are one inner dimension: x = 8 * pixel, a multiple of 8)
                for (int ia = 0; ia < a.px; ++ia)
                    tma_load_4d(smem_u32(sA + stage * A_BYTES) + (uint32_t)(ia * P.win_bytes), &P.tmap_x, 8 * wq0, hp0,
                                n_img, ia, fb);
                ++it;
                if (++stage == TC_STAGES) {
                    stage = 0;
                    phase ^= 1;
                }
            }
            // bounded wait until the copies of the last stages and the weights have landed
            const uint32_t from = it >= TC_STAGES ? it - TC_STAGES : 0;
            for (uint32_t j = from; j < it; ++j) {
                const long long t0 = clock64();
                while (!mbar_try_wait(full0 + 8 * (j % TC_STAGES), (j / TC_STAGES) & 1) &&
                       clock64() - t0 < TC_WAIT_CYCLES) {
                }
            }
            const long long t0 = clock64();
            while (!mbar_try_wait(wbar, 0) && clock64() - t0 < TC_WAIT_CYCLES) {
            }
        }
    } else if (!WEPI && warp < 4 && (P.patch || P.rows_tma)) {
        // ============================================================ producer, patch tiles
        // Stride 1 and Cp % 64 == 0: the A tile of tap (r, s) and channels c0..c0+63 is the box
        // {64, TW, TH} of the input at (c0, q0 + s - pad, p0 + r - pad); the padding reads as zeros.
        // Cp == 8: a k-block is 8 taps of 8 channels; tap tl's box {8, TW, TH} lands at byte
        // 2048 tl of the stage (a 16-byte K column of the no-swizzle layout), and taps past R*S
        // are boxes wholly outside the tensor (zero filled).
        if (lane == 0 && warp < TC_PRODUCERS) {
            // k-block it goes to producer (it % TC_STAGES) % TC_PRODUCERS: one thread's latency per k-block
            // (barrier wait, two TMA instructions) would bound the stage rate
            const int me = warp;
            const bool narrow = P.patch == 2;
            const uint32_t a_bytes = P.rows_tma ? (uint32_t)(TC_BM * 128) : (uint32_t)(P.TH * P.TW * (narrow ? 8 * 16 : 128));
            const int per_img = P.rows_tma ? 1 : P.tiles_p * P.tiles_q;
            uint32_t it = 0;
            bool ok = true;
            for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
                const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
                (void)sp;
                const int tm = t / P.tiles_n, tn = t % P.tiles_n;
                const int n_img = tm / per_img, r = tm - n_img * per_img;
                const int tq = P.rows_tma ? 1 : P.tiles_q;
                const int hp0 = (r / tq) * P.TH - a.pad, wq0 = (r % tq) * P.TW - a.pad;
                for (int gi = SPLIT ? P.gs[sp] : 0; gi < (SPLIT ? P.gs[sp + 1] : P.n_groups) && ok; ++gi) {
                    const TcGroup g = P.g[gi];
                    // tap (rr, ss) and channel offset cc of the group's first k-block, then stepped by
                    // TC_BK channels (Cp % 64 == 0: a k-block never straddles a tap)
                    const int tp0 = g.kb0 * TC_BK / a.Cp;
                    int cc = g.kb0 * TC_BK - tp0 * a.Cp;
                    int rr = tp0 / a.S, ss = tp0 - rr * a.S;
                    for (int kb = g.kb0; kb < g.kb1; ++kb, ++it) {
                        if ((int)((it % TC_STAGES) % TC_PRODUCERS) == me) {
                            const uint32_t stage = it % TC_STAGES, phase = (it / TC_STAGES) & 1;
                            if (!wait_bounded(empty0 + 8 * stage, phase ^ 1, abort, P.status)) {
                                ok = false;
                                break;
                            }
                            const uint32_t fb = PK ? pkfull0 + 8 * stage : full0 + 8 * stage;
                            const uint32_t pk_bytes = PK ? (uint32_t)(BN * 8 * P.wk) : 0u;
                            mbar_arrive_expect_tx(fb, a_bytes + (PK ? pk_bytes : (uint32_t)B_BYTES));
                            if (narrow) {
                                for (int tl = 0; tl < 8; ++tl) {
                                    const int tap = kb * 8 + tl;
                                    const bool in = tap < a.R * a.S;
                                    const int r8 = in ? tap / a.S : 0, s8 = in ? tap - (tap / a.S) * a.S : 0;
                                    tma_load_5d(smem_u32(sA + stage * A_BYTES + tl * 2048), &P.tmap_x, in ? 0 : 8,
                                                wq0 + s8, hp0 + r8, n_img, g.a_plane, fb);
                                }
                            } else if (P.rows_tma) {
                                tma_load_3d(smem_u32(sA + stage * A_BYTES), &P.tmap_x, kb * TC_BK, tm * TC_BM, g.a_plane,
                                            fb);
                            } else {
                                tma_load_5d(smem_u32(sA + stage * A_BYTES), &P.tmap_x, cc, wq0 + ss, hp0 + rr, n_img,
                                            g.a_plane, fb);
                            }
                            if (PK)
                                bulk_load(smem_u32(sP + stage * (BN * 64)),
                                          P.wpack + ((size_t)kb * P.K_pad + (size_t)tn * BN) * 2 * P.wk, pk_bytes, fb);
                            else
                                tma_load_3d(smem_u32(sB + stage * B_BYTES), &P.tmap_w, kb * TC_BK, tn * BN, g.w_plane,
                                            fb);
                        }
                        if (!narrow) {
                            cc += TC_BK;
                            if (cc >= a.Cp) {
                                cc = 0;
                                if (++ss == a.S) {
                                    ss = 0;
                                    ++rr;
                                }
                            }
                        }
                    }
                }
            }
            // bounded wait until the copies of the last stages have landed (PK: on pkfull, which only
            // the copies complete)
            const uint32_t drain0 = PK ? pkfull0 : full0;
            const uint32_t from = it >= TC_STAGES ? it - TC_STAGES : 0;
            for (uint32_t j = from; j < it; ++j) {
                const long long t0 = clock64();
                while (!mbar_try_wait(drain0 + 8 * (j % TC_STAGES), (j / TC_STAGES) & 1) &&
                       clock64() - t0 < TC_WAIT_CYCLES) {
                }
            }
        }
        if (PK && warp >= 1) pk_convert_loop<BN, SPLIT>(P, warp - 1, lane, sP, sB, pkfull0, full0, abort);
    } else if (!WEPI && warp < 4) {
        // ============================================================ producers, row tiles
        // Thread t copies 16-byte chunk c = t % 8 of rows t/8, t/8 + 16, ...: eight consecutive
        // threads cover one 128-byte row, so every warp instruction reads four whole rows.
        const int c = threadIdx.x & 7;
        const int r0 = threadIdx.x >> 3;  // 0..15
        constexpr int AR = TC_BM / 16;    // A rows per thread
        const __half* xb = a.x;
        uint32_t it = 0;
        bool ok = true;
        for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
            const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
            (void)sp;
            const int tm = t / P.tiles_n, tn = t % P.tiles_n;
            long long rowoff[AR];  // element offset of the (r, s) = (0, 0) tap of each row (may be negative)
            int p0[AR], q0[AR];
#pragma unroll
            for (int i = 0; i < AR; ++i) {
                const long long m = (long long)tm * TC_BM + r0 + 16 * i;
                const long long mm = m < a.M ? m : 0;
                const int n_img = (int)(mm / ((long long)a.P * a.Q));
                const int pq = (int)(mm - (long long)n_img * a.P * a.Q);
                p0[i] = (pq / a.Q) * a.stride - a.pad;
                q0[i] = (pq % a.Q) * a.stride - a.pad;
                if (m >= a.M) p0[i] = -(1 << 20);  // rows past the end read zeros
                rowoff[i] = (((long long)n_img * a.H + p0[i]) * a.W + q0[i]) * a.Cp;
            }
            for (int gi = SPLIT ? P.gs[sp] : 0; gi < (SPLIT ? P.gs[sp + 1] : P.n_groups) && ok; ++gi) {
                const TcGroup g = P.g[gi];
                const __half* xp = xb + (long long)g.a_plane * a.x_ps;
                for (int kb = g.kb0; kb < g.kb1; ++kb) {
                    const int stage = it % TC_STAGES;
                    const uint32_t ph = (it / TC_STAGES) & 1;
                    if (!wait_bounded(empty0 + 8 * stage, ph ^ 1, abort, P.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dA = smem_u32(sA + stage * A_BYTES);
                    if (threadIdx.x == 0) {  // the weight tile: one TMA, zero-filled past K and R*S*Cp
                        mbar_arrive_expect_tx(full0 + 8 * stage, (uint32_t)B_BYTES);
                        tma_load_3d(smem_u32(sB + stage * B_BYTES), &P.tmap_w, kb * TC_BK, tn * BN, g.w_plane,
                                    full0 + 8 * stage);
                    }
                    const int f = kb * TC_BK + 8 * c;  // this thread's chunk of the flattened (r, s, c) index
                    const bool fvalid = f < P.RSC;
                    const int tp = f / a.Cp;
                    const int cc = f - tp * a.Cp;
                    const int rr = tp / a.S, ss = tp - rr * a.S;
                    const long long toff = ((long long)rr * a.W + ss) * a.Cp + cc;
#pragma unroll
                    for (int i = 0; i < AR; ++i) {
                        const int row = r0 + 16 * i;
                        const int h = p0[i] + rr, w = q0[i] + ss;
                        const bool v = fvalid && (unsigned)h < (unsigned)a.H && (unsigned)w < (unsigned)a.W;
                        const __half* src = v ? xp + rowoff[i] + toff : xb;
                        cp_async16(dA + row * 128 + (uint32_t)((c ^ (row & 7)) << 4), src, v ? 16u : 0u);
                    }
                    cp_async_commit();
                    if (it >= TC_LAG) {
                        // this warp's copies of stage it - TC_LAG have landed: one arrival for the warp
                        cp_async_wait<TC_LAG>();
                        fence_proxy_async();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(full0 + 8 * ((it - TC_LAG) % TC_STAGES));
                    }
                    ++it;
                }
            }
        }
        cp_async_wait<0>();
        fence_proxy_async();
        __syncwarp();
        const uint32_t first = it >= TC_LAG ? it - TC_LAG : 0;
        if (lane == 0)
            for (uint32_t j = first; j < it; ++j) mbar_arrive(full0 + 8 * (j % TC_STAGES));
        if (threadIdx.x == 0) {
            // Every weight TMA this thread issued has landed once its stage's phase completes (the MMA
            // thread already waited for them unless the kernel aborted): bounded wait on the last ones.
            const uint32_t from = it >= TC_STAGES ? it - TC_STAGES : 0;
            for (uint32_t j = from; j < it; ++j) {
                const long long t0 = clock64();
                while (!mbar_try_wait(full0 + 8 * (j % TC_STAGES), (j / TC_STAGES) & 1) &&
                       clock64() - t0 < TC_WAIT_CYCLES) {
                }
            }
        }
    } else if (WEPI && warp < MMA_WARP) {
        // ============================================================ epilogue, window instances
        // Warp w drains TMEM lanes 32 (w % 4) .. + 31 and the 16 columns 16 cw .., cw = (w - 4) / 4: WIN of
        // the four limb accumulators, with the 32-bit arithmetic of the generic window epilogue below;
        // W64 of the one int32-exact accumulator, with the FxP-QLayer of the generic epilogue.  Tile u
        // goes through staging tile u % 2, whose previous store must have read it (at most the other
        // tile's store is then in flight).
        const int quad = warp & 3, cw = (warp - 4) >> 2;
        const int row = quad * 32 + lane;
        const bool leader = threadIdx.x == 128;  // waits for and issues the TMA stores
        const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
        const int m = a.sh - 16;
        const int half = m > 0 ? 1 << (m - 1) : 0;
        const int mmask = (int)((1u << m) - 1u);
        const int lo = (int)a.lo, hi = (int)a.hi;
        const int per_img = P.tiles_p * P.tiles_q;
        const bool f32out = a.out_mode == FXPQ_OUT_F32;  // the fp32 image (calibration) instead of codes
        // W64, 32-bit codes: a thread's 16 output channels are the same in every tile, so their aligned
        // bias terms and the flags of bias bits below the accumulator's scale are formed once
        const Epi32 e32w = make_epi32(a);
        int btw[16];
        uint32_t phiw = 0u;
        if (W64) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int k = cw * 16 + j;
                const int32_t b = (a.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                btw[j] = (b << e32w.bsl) >> e32w.bsr;
                phiw |= ((b & e32w.fmask) != 0 ? 1u : 0u) << j;
            }
        }
        bool ok = true;
        uint32_t u = 0;
        for (int t = blockIdx.x; t < P.n_tiles && ok; t += gridDim.x, ++u) {
            const uint32_t buf = u & 1;
            if (!wait_bounded(accfull0 + 8 * buf, (u >> 1) & 1, abort, P.status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t w[16];  // codes: 8 words of fp16 pairs; fp32 image: 16 values
            if (W64) {
                uint32_t f[16];
                tmem_ld16_nw(lane_base + buf * (uint32_t)BN + (uint32_t)(cw * 16), f);
                tmem_wait_ld();
                reg_fence(f);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(accempty0 + 8 * buf);
                if (f32out) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int k = cw * 16 + j;
                        const int acc = __float2int_rn(__uint_as_float(f[j]));
                        const int32_t b = (a.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                        w[j] = __float_as_uint(__ll2float_rn(cblock_value<false>(a, k, (long long)acc, b)) * a.f32_scale);
                    }
                }
                if (!f32out && a.v32) {
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        int c2[2];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int jj = 2 * j + h;
                            c2[h] = epi32_code(e32w, __float2int_rn(__uint_as_float(f[jj])), btw[jj], (int)((phiw >> jj) & 1u));
                        }
                        w[j] = pack_codes_f16(c2[0], c2[1]);
                    }
                } else if (!f32out) {
                    const Epi64 e64 = make_epi64(a);
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        int c2[2];
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            const int k = cw * 16 + 2 * j + h;
                            const int acc = __float2int_rn(__uint_as_float(f[2 * j + h]));
                            const int32_t b = (a.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                            c2[h] = epi64_code<false>(e64, (long long)acc, b, 0, 0);
                        }
                        w[j] = pack_codes_f16(c2[0], c2[1]);
                    }
                }
            }
            uint32_t fhh[16], fhl[16], flh[16], fll[16];
            if (WIN) {
                const uint32_t abase = lane_base + buf * (uint32_t)(4 * BN) + (uint32_t)(cw * 16);
                tmem_ld16_nw(abase, fhh);
                tmem_ld16_nw(abase + (uint32_t)BN, fhl);
                tmem_ld16_nw(abase + (uint32_t)(2 * BN), flh);
                tmem_ld16_nw(abase + (uint32_t)(3 * BN), fll);
                tmem_wait_ld();
                reg_fence(fhh);
                reg_fence(fhl);
                reg_fence(flh);
                reg_fence(fll);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(accempty0 + 8 * buf);
            }
            if (WIN && f32out) {
                // the fp32 nearest-even image of v = 2^16 T + Lo (ReLU: 0 when T < 0), scaled by 2^-s
#pragma unroll
                for (int jj = 0; jj < 16; ++jj) {
                    const int2 bt = wtab[cw * 16 + jj];
                    const int mid = __float2int_rn(__uint_as_float(fhl[jj])) + __float2int_rn(__uint_as_float(flh[jj]));
                    const int L = mid * 256 + __float2int_rn(__uint_as_float(fll[jj])) + bt.y;
                    const int T = __float2int_rn(__uint_as_float(fhh[jj])) + bt.x + (L >> 16);
                    const long long v = (a.relu && T < 0) ? 0LL : ((long long)T << 16) + (L & 0xFFFF);
                    w[jj] = __float_as_uint(__ll2float_rn(v) * a.f32_scale);
                }
            }
#pragma unroll
            for (int j = 0; j < ((WIN && !f32out) ? 8 : 0); ++j) {
                int c2[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int jj = 2 * j + h;
                    const int2 bt = wtab[cw * 16 + jj];
                    const int mid = __float2int_rn(__uint_as_float(fhl[jj])) + __float2int_rn(__uint_as_float(flh[jj]));
                    const int L = mid * 256 + __float2int_rn(__uint_as_float(fll[jj])) + bt.y;
                    const int T = __float2int_rn(__uint_as_float(fhh[jj])) + bt.x + (L >> 16);
                    const int Lo = L & 0xFFFF;
                    int q, up;
                    if (m > 0) {
                        q = T >> m;
                        const int rem = T & mmask;
                        up = (rem > half) | ((rem == half) & ((Lo != 0) | (q & 1)));
                    } else {
                        q = T;
                        up = (Lo > 0x8000) | ((Lo == 0x8000) & (q & 1));
                    }
                    const int cc = (a.relu && T < 0) ? 0 : q + up;
                    c2[h] = min(max(cc, lo), hi);
                }
                w[j] = pack_codes_f16(c2[0], c2[1]);
            }
            if (f32out) {
                // fp32 image out: this row's 16 values are 64 contiguous bytes of the output row
                const long long mrow = tile_row(P, t, row);
                if (mrow >= 0) {
                    float* yp = static_cast<float*>(a.y) + mrow * a.K + cw * 16;
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        if (cw * 16 + 4 * q < a.K)
                            *reinterpret_cast<uint4*>(yp + 4 * q) = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
                }
                continue;
            }
            const uint32_t sb = u & 1, n = u >> 1;  // staging tile and its use count
            const uint32_t sfull = sb ? stg_full2 : stg_full, sfree = sb ? stg_free2 : stg_free;
            if (n > 0) {
                if (leader) {
                    bulk_wait_read1();  // the store of tile u - 2 (this staging tile) has read it
                    mbar_arrive(sfree);
                }
                if (!wait_bounded(sfree, (n - 1) & 1, abort, P.status)) {
                    ok = false;
                    break;
                }
            }
            unsigned char* sbuf = sO + sb * (TC_BM * 128);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const int chunk = cw * 2 + q;
                *reinterpret_cast<uint4*>(sbuf + row * 128 + ((chunk ^ (row & 7)) << 4)) =
                    make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(sfull);
            if (leader) {
                if (!wait_bounded(sfull, n & 1, abort, P.status)) {
                    ok = false;
                    break;
                }
                const int n_img = t / per_img, r = t - n_img * per_img;
                tma_store_4d(&P.tmap_y, 0, (r % P.tiles_q) * P.TW, (r / P.tiles_q) * P.TH, n_img, smem_u32(sbuf));
                bulk_commit();
            }
        }
        if (leader) bulk_wait0();  // every output store has completed
    } else if (warp < MMA_WARP) {
        // ============================================================ epilogue
        // Warp w drains TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31 (the quadrant a warp may access) and
        // the 32-column chunks cw * CPW .. cw * CPW + CPW - 1, cw = (w - 4) / 4, of every accumulator.
        const int quad = warp & 3;
        const int cw = (warp - 4) >> 2;
        const int row = quad * 32 + lane;
        const bool leader = threadIdx.x == 128;  // waits for and issues the tile's TMA stores
        const int nbuf = P.nbuf;
        uint32_t gcount = 0;
        bool ok = true;
        // Integer running sums of a tile live in TMEM after the accumulator buffers: columns
        // [nbuf BN, nbuf BN + BN * words), words = 1 (int32) or 2 (int64 as lo / hi column blocks).
        const uint32_t lane_base = tmem + ((uint32_t)(quad * 32) << 16);
        const uint32_t run_base = (uint32_t)(nbuf * BN);
        uint32_t u = 0;  // tiles written through the staging buffer so far
        for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
            const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
            (void)sp;
            const int tm = t / P.tiles_n, tn = t % P.tiles_n;
            const long long m = tile_row(P, tm, row);  // -1: row outside the output
            const int g_lo = SPLIT ? P.gs[sp] : 0, g_hi = SPLIT ? P.gs[sp + 1] : P.n_groups;
            for (int gi = g_lo; gi < g_hi; ++gi) {
                const int shift = P.g[gi].shift;
                const bool first = gi == g_lo, last = gi == g_hi - 1;
                const uint32_t buf = nbuf == 2 ? (gcount & 1) : 0;
                const uint32_t par = nbuf == 2 ? ((gcount >> 1) & 1) : (gcount & 1);
                if (!wait_bounded(accfull0 + 8 * buf, par, abort, P.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (!DIRECT && last && P.fast_store && u > 0) {
                    // the previous tile's TMA store must have read the staging buffer
                    if (leader) {
                        bulk_wait_read0();
                        mbar_arrive(stg_free);
                    }
                    if (!wait_bounded(stg_free, (u - 1) & 1, abort, P.status)) {
                        ok = false;
                        break;
                    }
                }
#pragma unroll 1
                for (int c = 0; c < CPW; ++c) {
                    const int cb = cw * CPW + c;
                    const int k0 = tn * BN + cb * 32;
                    const uint32_t run_col = run_base + cb * 32;
                    if (BN == 64 && sizeof(ACC) == 8 && !SC && P.patch == 3 && P.w32) {
                        // window mode, two-limb x and w, 32-bit arithmetic.  With the limb sums S_hh,
                        // S_mid = S_hl + S_lh, S_ll and the aligned bias B' = 2^16 Bh + Bl (0 <= Bl < 2^16):
                        //   v = 2^16 S_hh + 2^8 S_mid + S_ll + B' = 2^16 T + Lo,
                        //   L = 2^8 S_mid + S_ll + Bl,  T = S_hh + Bh + (L >> 16),  Lo = L & 0xFFFF,
                        // (the host keeps |L| and |T| below 2^31).  With sh = 16 + m, floor(v / 2^sh) =
                        // T >> m and the remainder is 2^16 (T mod 2^m) + Lo, so round half to even needs
                        // T mod 2^m against 2^(m-1), and Lo only to tell a tie (Lo = 0) from above it.
                        // ReLU: v < 0 exactly when T < 0.
                        const int m = a.sh - 16;
                        const int half = m > 0 ? 1 << (m - 1) : 0;
                        const int mmask = (int)((1u << m) - 1u);
                        const int lo = (int)a.lo, hi = (int)a.hi;
                        const uint32_t abase = lane_base + buf * (uint32_t)(4 * BN) + cb * 32;
                        uint32_t w[16];
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            uint32_t fhh[16], fhl[16], flh[16], fll[16];
                            tmem_ld16_nw(abase + 16 * hf, fhh);
                            tmem_ld16_nw(abase + (uint32_t)BN + 16 * hf, fhl);
                            tmem_ld16_nw(abase + (uint32_t)(2 * BN) + 16 * hf, flh);
                            tmem_ld16_nw(abase + (uint32_t)(3 * BN) + 16 * hf, fll);
                            tmem_wait_ld();
                            reg_fence(fhh);
                            reg_fence(fhl);
                            reg_fence(flh);
                            reg_fence(fll);
                            if (hf == 1 && c == CPW - 1) {
                                tc_fence_before();
                                __syncwarp();
                                if (lane == 0) mbar_arrive(accempty0 + 8 * buf);
                            }
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                int c2[2];
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    const int jj = 2 * j + h;
                                    const int2 bt = wtab[cb * 32 + 16 * hf + jj];
                                    const int mid = __float2int_rn(__uint_as_float(fhl[jj])) +
                                                    __float2int_rn(__uint_as_float(flh[jj]));
                                    const int L = mid * 256 + __float2int_rn(__uint_as_float(fll[jj])) + bt.y;
                                    const int T = __float2int_rn(__uint_as_float(fhh[jj])) + bt.x + (L >> 16);
                                    const int Lo = L & 0xFFFF;
                                    int q, up;
                                    if (m > 0) {
                                        q = T >> m;
                                        const int rem = T & mmask;
                                        up = (rem > half) | ((rem == half) & ((Lo != 0) | (q & 1)));
                                    } else {
                                        q = T;
                                        up = (Lo > 0x8000) | ((Lo == 0x8000) & (q & 1));
                                    }
                                    int cc = (a.relu && T < 0) ? 0 : q + up;
                                    c2[h] = min(max(cc, lo), hi);
                                }
                                w[8 * hf + j] = pack_codes_f16(c2[0], c2[1]);
                            }
                        }
                        unsigned char* half_buf = sO + (cb >> 1) * (TC_BM * 128);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int chunk = (cb & 1) * 4 + q;
                            *reinterpret_cast<uint4*>(half_buf + row * 128 + ((chunk ^ (row & 7)) << 4)) =
                                make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
                        }
                        continue;
                    }
                    if (sizeof(ACC) == 8 && P.patch == 3 && P.nacc == 4 && P.fast_store && a.sh >= 1 && a.sh <= 62) {
                        // window mode, two-limb x and w, one-plane codes out: each 16-column half goes
                        // from the four limb accumulators to packed codes before the next is loaded
                        // (keeps the live 64-bit values to 16)
                        const Epi64 e64 = make_epi64(a);
                        const int k0 = tn * BN + cb * 32;
                        const uint32_t abase = lane_base + buf * (uint32_t)(P.nacc * BN) + cb * 32;
                        uint32_t w[16];
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            uint32_t fhh[16], fhl[16], flh[16], fll[16];
                            tmem_ld16_nw(abase + 16 * hf, fhh);
                            tmem_ld16_nw(abase + (uint32_t)BN + 16 * hf, fhl);
                            tmem_ld16_nw(abase + (uint32_t)(2 * BN) + 16 * hf, flh);
                            tmem_ld16_nw(abase + (uint32_t)(3 * BN) + 16 * hf, fll);
                            tmem_wait_ld();
                            reg_fence(fhh);
                            reg_fence(fhl);
                            reg_fence(flh);
                            reg_fence(fll);
                            if (hf == 1 && c == CPW - 1) {
                                tc_fence_before();
                                __syncwarp();
                                if (lane == 0) mbar_arrive(accempty0 + 8 * buf);
                            }
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                int c2[2];
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    const int jj = 2 * j + h;
                                    const int k = k0 + 16 * hf + jj;
                                    const long long v = ((long long)__float2int_rn(__uint_as_float(fhh[jj])) << 16) +
                                                        ((long long)(__float2int_rn(__uint_as_float(fhl[jj])) +
                                                                     __float2int_rn(__uint_as_float(flh[jj])))
                                                         << 8) +
                                                        (long long)__float2int_rn(__uint_as_float(fll[jj]));
                                    const int32_t b = (e64.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                                    c2[h] = epi64_code<SC>(e64, v, b, SC ? scale_code(a, k) : 0,
                                                           SC ? shift_code(a, k) : 0);
                                }
                                w[8 * hf + j] = pack_codes_f16(c2[0], c2[1]);
                            }
                        }
                        unsigned char* half_buf = sO + (cb >> 1) * (TC_BM * 128);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int chunk = (cb & 1) * 4 + q;
                            *reinterpret_cast<uint4*>(half_buf + row * 128 + ((chunk ^ (row & 7)) << 4)) =
                                make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
                        }
                        continue;
                    }
                    // One TMEM round trip per load batch: the fp32 group sums and, after the first group,
                    // the integer running sums are loaded together; the running-sum stores share one
                    // completion wait.
                    ACC acc[32];
                    if (sizeof(ACC) == 8 && P.patch == 3) {
                        // window mode: one accumulator per limb pair (ia, iw), combined with its weight
                        // 2^(8 ((px-1-ia) + (pw-1-iw))); each is an exact integer below 2^24
                        const uint32_t abase = lane_base + buf * (uint32_t)(P.nacc * BN) + cb * 32;
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            if (P.nacc == 4) {
                                // two-limb x and w: the four accumulators share one load round trip;
                                // v = 2^16 S_hh + 2^8 (S_hl + S_lh) + S_ll, the middle pair summed in 32 bits
                                uint32_t fhh[16], fhl[16], flh[16], fll[16];
                                tmem_ld16_nw(abase + 16 * hf, fhh);
                                tmem_ld16_nw(abase + (uint32_t)BN + 16 * hf, fhl);
                                tmem_ld16_nw(abase + (uint32_t)(2 * BN) + 16 * hf, flh);
                                tmem_ld16_nw(abase + (uint32_t)(3 * BN) + 16 * hf, fll);
                                tmem_wait_ld();
                                reg_fence(fhh);
                                reg_fence(fhl);
                                reg_fence(flh);
                                reg_fence(fll);
#pragma unroll
                                for (int j = 0; j < 16; ++j) {
                                    const int hh = __float2int_rn(__uint_as_float(fhh[j]));
                                    const int mid = __float2int_rn(__uint_as_float(fhl[j])) +
                                                    __float2int_rn(__uint_as_float(flh[j]));
                                    const int ll = __float2int_rn(__uint_as_float(fll[j]));
                                    acc[16 * hf + j] = ((ACC)hh << 16) + ((ACC)mid << 8) + (ACC)ll;
                                }
                            } else {
#pragma unroll
                                for (int j = 0; j < 16; ++j) acc[16 * hf + j] = 0;
                                for (int ia = 0; ia < a.px; ++ia)
                                    for (int iw = 0; iw < a.pw; ++iw) {
                                        uint32_t f16[16];
                                        tmem_ld16_nw(abase + (uint32_t)((ia * a.pw + iw) * BN) + 16 * hf, f16);
                                        tmem_wait_ld();
                                        reg_fence(f16);
                                        const int sh = 8 * ((a.px - 1 - ia) + (a.pw - 1 - iw));
#pragma unroll
                                        for (int j = 0; j < 16; ++j)
                                            acc[16 * hf + j] += ((ACC)__float2int_rn(__uint_as_float(f16[j]))) << sh;
                                    }
                            }
                        }
                    } else if (sizeof(ACC) == 8) {
                        // int64 running sums in 16-column halves (lo and hi words in separate column blocks)
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            uint32_t f16[16], lo[16], hi[16];
                            tmem_ld16_nw(lane_base + buf * BN + cb * 32 + 16 * hf, f16);
                            if (!first) {
                                tmem_ld16_nw(lane_base + run_col + 16 * hf, lo);
                                tmem_ld16_nw(lane_base + run_col + BN + 16 * hf, hi);
                            }
                            tmem_wait_ld();
                            reg_fence(f16);
                            if (!first) {
                                reg_fence(lo);
                                reg_fence(hi);
                            }
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                ACC v = ((ACC)__float2int_rn(__uint_as_float(f16[j]))) << shift;
                                if (!first) v += (ACC)(((unsigned long long)hi[j] << 32) | lo[j]);
                                acc[16 * hf + j] = v;
                            }
                            if (!last) {
#pragma unroll
                                for (int j = 0; j < 16; ++j) {
                                    lo[j] = (uint32_t)(unsigned long long)acc[16 * hf + j];
                                    hi[j] = (uint32_t)((unsigned long long)acc[16 * hf + j] >> 32);
                                }
                                tmem_st16_nw(lane_base + run_col + 16 * hf, lo);
                                tmem_st16_nw(lane_base + run_col + BN + 16 * hf, hi);
                            }
                        }
                        if (!last) tmem_wait_st();
                    } else {
                        // int32 running sums, 16-column halves (keeps the live registers low)
#pragma unroll
                        for (int hf = 0; hf < 2; ++hf) {
                            uint32_t f16[16], run[16];
                            tmem_ld16_nw(lane_base + buf * BN + cb * 32 + 16 * hf, f16);
                            if (!first) tmem_ld16_nw(lane_base + run_col + 16 * hf, run);
                            tmem_wait_ld();
                            reg_fence(f16);
                            if (!first) reg_fence(run);
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                ACC v = ((ACC)__float2int_rn(__uint_as_float(f16[j]))) << shift;
                                if (!first) v += (ACC)(int)run[j];
                                acc[16 * hf + j] = v;
                            }
                            if (!last) {
#pragma unroll
                                for (int j = 0; j < 16; ++j) run[j] = (uint32_t)(unsigned long long)acc[16 * hf + j];
                                tmem_st16_nw(lane_base + run_col + 16 * hf, run);
                            }
                        }
                        if (!last) tmem_wait_st();
                    }
                    if (c == CPW - 1) {
                        // every chunk of this warp is out of the accumulator buffer: free it for the
                        // next group's MMAs before the final arithmetic (one arrival per warp: same-address
                        // arrivals of every thread serialise)
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(accempty0 + 8 * buf);
                    }
                    if (!last) continue;
                    if (SPLIT && P.ksplit > 1) {
                        // one share of the reduction: its exact integer sums go to the partial buffer
                        if (m >= 0) {
                            ACC* dst = static_cast<ACC*>(P.part) + ((long long)sp * a.M + m) * a.K + k0;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (k0 + j < a.K) dst[j] = acc[j];
                        }
                        continue;
                    }
                    if (P.fast_store) {
                        // 32 one-plane codes -> 4 swizzled 16-byte chunks of this row in the staging buffer
                        // (the epilogue constants are rebuilt here from the parameters rather than kept
                        // live across the tile loop)
                        uint32_t w[16];
                        const Epi32 e32 = make_epi32(a);
                        const Epi64 e64 = make_epi64(a);
                        if (sizeof(ACC) == 4 && !SC && a.v32) {
                            // the chunk's 32 biases by 16-byte loads where they are whole and aligned
                            const bool bvec = e32.has_bias && k0 + 32 <= a.K &&
                                              (reinterpret_cast<uintptr_t>(a.bias) & 15u) == 0;
#pragma unroll
                            for (int j4 = 0; j4 < 8; ++j4) {
                                int bb[4];
                                if (bvec) {
                                    const int4 v4 = __ldg(reinterpret_cast<const int4*>(a.bias + k0) + j4);
                                    bb[0] = v4.x;
                                    bb[1] = v4.y;
                                    bb[2] = v4.z;
                                    bb[3] = v4.w;
                                } else {
#pragma unroll
                                    for (int e = 0; e < 4; ++e) {
                                        const int k = k0 + 4 * j4 + e;
                                        bb[e] = (e32.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                                    }
                                }
                                int c4[4];
#pragma unroll
                                for (int e = 0; e < 4; ++e)
                                    c4[e] = epi32_code(e32, (int)acc[4 * j4 + e], (bb[e] << e32.bsl) >> e32.bsr,
                                                       min(bb[e] & e32.fmask, 1));
                                w[2 * j4] = pack_codes_f16(c4[0], c4[1]);
                                w[2 * j4 + 1] = pack_codes_f16(c4[2], c4[3]);
                            }
                        } else if (e64.ok) {
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                int c2[2];
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    const int k = k0 + 2 * j + h;
                                    const int32_t b = (e64.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                                    c2[h] = epi64_code<SC>(e64, (long long)acc[2 * j + h], b,
                                                           SC ? scale_code(a, k) : 0, SC ? shift_code(a, k) : 0);
                                }
                                w[j] = pack_codes_f16(c2[0], c2[1]);
                            }
                        } else {
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                int c2[2];
#pragma unroll
                                for (int h = 0; h < 2; ++h) {
                                    const int k = k0 + 2 * j + h;
                                    const int32_t b = (a.has_bias && k < a.K) ? __ldg(a.bias + k) : 0;
                                    c2[h] = qlayer_code(a, cblock_value<SC>(a, k, (long long)acc[2 * j + h], b));
                                }
                                w[j] = pack_codes_f16(c2[0], c2[1]);
                            }
                        }
                        if (DIRECT) {
                            // through the warp's 2 KB slice of the staging region: each lane puts its row's
                            // 64 bytes there (16-byte pieces rotated against bank conflicts), then every
                            // store instruction writes whole 64-byte row segments of eight rows.  One-plane
                            // codes have K % 8 == 0, so a 16-byte piece lies wholly inside or past K.
                            unsigned char* wbuf = sO + (warp - 4) * 2048;
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                *reinterpret_cast<uint4*>(wbuf + lane * 64 + 16 * (q ^ ((lane >> 1) & 3))) =
                                    make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
                            __syncwarp();
#pragma unroll
                            for (int it = 0; it < 4; ++it) {
                                const int r = (lane >> 2) + 8 * it, pc = lane & 3;
                                const long long mr = __shfl_sync(0xffffffffu, m, r);
                                const uint4 v = *reinterpret_cast<const uint4*>(wbuf + r * 64 + 16 * (pc ^ ((r >> 1) & 3)));
                                const int kk = k0 + pc * 8;
                                if (mr >= 0 && kk < a.K)
                                    *reinterpret_cast<uint4*>(static_cast<__half*>(a.y) + mr * a.K + kk) = v;
                            }
                            __syncwarp();
                            continue;
                        }
                        unsigned char* half_buf = sO + (cb >> 1) * (TC_BM * 128);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const int chunk = (cb & 1) * 4 + q;
                            *reinterpret_cast<uint4*>(half_buf + row * 128 + ((chunk ^ (row & 7)) << 4)) =
                                make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
                        }
                    } else if (!PK && (a.out_mode == FXPQ_OUT_F32 ? a.K % 4 == 0 : (a.out_mode == FXPQ_OUT_ACC64 && a.K % 2 == 0))) {
                        // fp32 / int64 outputs through the warp's 2 KiB of the (unused) staging tile
                        epilogue_block32_staged<ACC, SC>(a, m, k0, acc, sO + (warp - 4) * 2048, lane);
                    } else if (m >= 0) {
                        epilogue_block32<ACC, SC>(a, m, k0, acc);
                    }
                }
                ++gcount;
                if (!DIRECT && last && P.fast_store) {
                    // make the staging writes visible to the async proxy, then one thread stores the tile
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(stg_full);
                    if (leader) {
                        if (!wait_bounded(stg_full, u & 1, abort, P.status)) {
                            ok = false;
                            break;
                        }
                        if (P.patch) {
                            const int per_img = P.tiles_p * P.tiles_q;
                            const int n_img = tm / per_img, r = tm - n_img * per_img;
                            for (int hb = 0; hb < BN / 64; ++hb)
                                tma_store_4d(&P.tmap_y, tn * BN + hb * 64, (r % P.tiles_q) * P.TW,
                                             (r / P.tiles_q) * P.TH, n_img, smem_u32(sO + hb * (TC_BM * 128)));
                        } else {
                            for (int hb = 0; hb < BN / 64; ++hb)
                                tma_store_2d(&P.tmap_y, tn * BN + hb * 64, tm * TC_BM,
                                             smem_u32(sO + hb * (TC_BM * 128)));
                        }
                        bulk_commit();
                    }
                    ++u;
                }
            }
        }
        if (leader) bulk_wait0();  // every output store has completed
    } else if (PK && warp > MMA_WARP) {
        // ============================================================ packed-weight converters
        pk_convert_loop<BN, SPLIT>(P, 3 + (warp - MMA_WARP - 1), lane, sP, sB, pkfull0, full0, abort);
    } else if (!WIN && lane == 0 && P.patch == 4) {
        // ============================================================ MMA issue, 64-channel window mode
        // Per tile, tap (r, s) and 16-channel step kk: one MMA.  A is window copy s from row r: rows 128
        // bytes apart, the 8-row groups (patch rows, TW = 8) one pattern (1 KiB) apart; B the resident tap
        // block (a B stage's layout).  One barrier round per tile.
        const uint32_t copyb = (uint32_t)P.WH * 1024u;
        uint32_t stage = 0, phase = 0, gcount = 0;
        bool ok = wait_mma(wbar, 0, abort, P.status);
        tc_fence_after();
        for (int t = blockIdx.x; t < P.n_tiles && ok; t += gridDim.x) {
            const uint32_t buf = gcount & 1;
            if (!wait_mma(accempty0 + 8 * buf, ((gcount >> 1) & 1) ^ 1, abort, P.status) ||
                !wait_mma(full0 + 8 * stage, phase, abort, P.status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t wa = smem_u32(sA) + (uint32_t)P.w64_slot0 + stage * (uint32_t)P.w64_slot_stride;
            const uint32_t d = tmem + buf * BN;
            uint32_t accum = 0;
            for (int r = 0; r < a.R; ++r)
                for (int q = 0; q < a.S; ++q) {
                    const uint64_t ad = make_sdesc(wa + (uint32_t)q * copyb + (uint32_t)r * 1024u);
                    const uint64_t bd = make_sdesc(smem_u32(sA) + (uint32_t)(r * a.S + q) * 8192u);
#pragma unroll
                    for (int kk = 0; kk < TC_BK / 16; ++kk) {
                        tc_mma(d, ad + 2 * kk, bd + 2 * kk, IDESC, accum);
                        accum = 1;
                    }
                }
            tc_commit(empty0 + 8 * stage);
            if (++stage == 2) {
                stage = 0;
                phase ^= 1;
            }
            tc_commit(accfull0 + 8 * buf);
            ++gcount;
        }
        // every MMA issued by this thread has completed once `done` fires
        tc_commit(done_bar);
        const long long t0 = clock64();
        while (!mbar_try_wait(done_bar, 0) && clock64() - t0 < TC_WAIT_CYCLES) {
        }
    } else if (!W64 && lane == 0 && P.patch == 3) {
        // ============================================================ MMA issue, window mode
        // Per tile and limb pair (ia, iw): R * S2/2 MMAs of K = 16 (two taps of 8 channels).  The A
        // operand of taps (r, 2sp), (r, 2sp + 1) is the window shifted by (r, 2sp) pixels: K-major
        // without swizzle, the two K core matrices one pixel (16 bytes) apart, the 8-row groups (the
        // patch rows, TW = 8) one window row apart.  B is the resident box (iw, r, sp).
        const int np = P.S2 / 2;
        const uint32_t tapb = (uint32_t)(BN * 16);
        // N = pw BN: the B operand of tap pair (r, sp) holds [W_hi | W_lo] (one plane: N = BN); its K
        // core matrices (the two taps) are pw BN 16 bytes apart, its 8-row groups 128 bytes apart
        const uint32_t idesc_w = a.pw == 2 ? make_idesc(TC_BM, 2 * BN) : IDESC;
        uint64_t bdesc[8];
        uint32_t aoff[8];  // A start of tap pair (r, sp) in the window, in 16-byte units
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int r = i / np, sp = i - r * np;
            bdesc[i] = make_sdesc_noswz(smem_u32(sB) + (uint32_t)(i * 2 * a.pw) * tapb, (uint32_t)a.pw * tapb, 128);
            aoff[i] = (uint32_t)((r * P.WW + 2 * sp) * 16) >> 4;
        }
        uint32_t stage = 0, phase = 0, gcount = 0;
        bool ok = wait_mma(wbar, 0, abort, P.status);
        tc_fence_after();
        for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
            const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
            (void)sp;
            const uint32_t buf = gcount & 1;
            if (!wait_mma(accempty0 + 8 * buf, ((gcount >> 1) & 1) ^ 1, abort, P.status) ||
                !wait_mma(full0 + 8 * stage, phase, abort, P.status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t d0 = tmem + buf * (uint32_t)(P.nacc * BN);
            const uint32_t wa = smem_u32(sA + stage * A_BYTES);
            for (int ia = 0; ia < a.px; ++ia) {
                // accumulators (ia, iw) at columns (ia pw + iw) BN: one MMA of N = pw BN fills the pw of them
                const uint32_t d = d0 + (uint32_t)(ia * a.pw * BN);
                const uint64_t ad0 = make_sdesc_noswz(wa + (uint32_t)(ia * P.win_bytes), 16, (uint32_t)(P.WW * 16));
                const int nt = a.R * np;  // <= 8
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    if (i < nt) tc_mma(d, ad0 + (uint64_t)aoff[i], bdesc[i], idesc_w, i > 0 ? 1u : 0u);
            }
            tc_commit(empty0 + 8 * stage);
            if (++stage == TC_STAGES) {
                stage = 0;
                phase ^= 1;
            }
            tc_commit(accfull0 + 8 * buf);
            ++gcount;
        }
        // every MMA issued by this thread has completed once `done` fires
        tc_commit(done_bar);
        const long long t0 = clock64();
        while (!mbar_try_wait(done_bar, 0) && clock64() - t0 < TC_WAIT_CYCLES) {
        }
    } else if (!WEPI && lane == 0) {
        // ============================================================ MMA issue (one thread of MMA_WARP)
        // Descriptors of stage 0; a stage or a 16-element k step moves the start-address field
        // (address >> 4, 14 bits) without carry since shared addresses stay below 256 KB.
        // 8-channel patch tiles: no-swizzle A, one 16-element k step = two taps = 4096 bytes
        const bool narrow_a = P.patch == 2;
        const uint64_t adesc0 = narrow_a ? make_sdesc_noswz(smem_u32(sA), 2048, 128) : make_sdesc(smem_u32(sA));
        const uint32_t a_kstep = narrow_a ? 4096u >> 4 : 2u;
        const uint64_t bdesc0 = make_sdesc(smem_u32(sB));
        uint32_t stage = 0, phase = 0, gcount = 0;
        bool ok = true;
        for (int ut = blockIdx.x; ut < (SPLIT ? P.n_units : P.n_tiles) && ok; ut += gridDim.x) {
            const int t = SPLIT ? ut / P.ksplit : ut, sp = SPLIT ? ut - t * P.ksplit : 0;
            (void)sp;
            for (int gi = SPLIT ? P.gs[sp] : 0; gi < (SPLIT ? P.gs[sp + 1] : P.n_groups) && ok; ++gi) {
                const TcGroup g = P.g[gi];
                const uint32_t buf = P.nbuf == 2 ? (gcount & 1) : 0;
                const uint32_t par = P.nbuf == 2 ? ((gcount >> 1) & 1) : (gcount & 1);
                if (!wait_mma(accempty0 + 8 * buf, par ^ 1, abort, P.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem + buf * BN;
                uint32_t accum = 0;
                for (int kb = g.kb0; kb < g.kb1; ++kb) {
                    if (!wait_mma(full0 + 8 * stage, phase, abort, P.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = adesc0 + (uint64_t)((stage * A_BYTES) >> 4);
                    const uint64_t bd = bdesc0 + (uint64_t)((stage * B_BYTES) >> 4);
#pragma unroll
                    for (int kk = 0; kk < TC_BK / 16; ++kk) {
                        tc_mma(d, ad + a_kstep * kk, bd + 2 * kk, IDESC, accum);
                        accum = 1;
                    }
                    tc_commit(empty0 + 8 * stage);
                    if (++stage == TC_STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                tc_commit(accfull0 + 8 * buf);
                ++gcount;
            }
        }
        // every MMA issued by this thread has completed once `done` fires
        tc_commit(done_bar);
        const long long t0 = clock64();
        while (!mbar_try_wait(done_bar, 0) && clock64() - t0 < TC_WAIT_CYCLES) {
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == MMA_WARP) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS));
    }
}

}  // namespace tc

// Launches the SC = true kernel for tile width BN (acc64: the 64-bit running-sum variant, BN = 64).
fxpq_status launch_conv_tc_scaled(const tc::TcParams& P, int BN, bool acc64, int grid, cudaStream_t st);

}  // namespace fxpq
