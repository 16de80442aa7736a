// Host-side check of the C-Block epilogue arithmetic (Sec. IV-B: bias alignment, optional Scale
// layer, ReLU, FxP-QLayer).  For each case read from stdin it plans the layer with the library's own
// host planner (plan_conv: integer bounds and the choice of the 32-bit path) and evaluates, on the CPU,
// the same inline functions the kernels use:
//   generic  qlayer_code(cblock_value)        (CUDA-core kernel, split-reduction epilogue)
//   code32   qlayer_code32                    (CUDA-core kernel, 32-bit path)
//   epi32    epi32_code, with the tensor-core kernel's bias-term expression
//   epi64    epi64_code<SC>                   (tensor-core kernel, 64-bit path)
// tests/test_epilogue_host.py compiles it against the library's objects and compares every printed
// code with the oracle's C-Block and FxP-QLayer.
//
// Input, one case per line (integers):
//   xb xs xfl  wb ws wfl  bb bs bfl  yb ys yfl  relu has_bias C w_l1  acc bias
//   has_scale  sb ss sfl  hb hs hfl  m h
// Output, one line per case:
//   status v32 sh generic code32 epi32 epi64   (NA = -2147483648 where a path does not apply)
#include <climits>
#include <cstdio>

#include "fxpq_conv_tc.cuh"

using namespace fxpq;
using namespace fxpq::tc;

int main() {
    long long v[27];
    const long long NA = INT_MIN;
    while (true) {
        int got = 0;
        for (int i = 0; i < 27; ++i) got += scanf("%lld", &v[i]) == 1;
        if (got != 27) break;
        fxpq_conv_desc d = {};
        d.N = 1, d.H = 1, d.W = 1, d.C = (int)v[14], d.Cp = (int)((v[14] + 7) / 8 * 8);
        d.K = 8, d.R = 1, d.S = 1, d.stride = 1, d.pad = 0;
        d.relu = (int)v[12];
        d.out_mode = FXPQ_OUT_CODES;
        d.fmt_x = fxpq_fmt{(int)v[0], (int)v[1], (int)v[2]};
        d.fmt_w = fxpq_fmt{(int)v[3], (int)v[4], (int)v[5]};
        d.fmt_b = fxpq_fmt{(int)v[6], (int)v[7], (int)v[8]};
        d.fmt_y = fxpq_fmt{(int)v[9], (int)v[10], (int)v[11]};
        d.w_l1 = v[15];
        const bool has_bias = v[13] != 0, has_scale = v[18] != 0;
        // never dereferenced: plan_conv only checks them for null and alignment
        static __align__(16) int32_t dummy[16];
        if (has_scale) {
            d.fmt_scale = fxpq_fmt{(int)v[19], (int)v[20], (int)v[21]};
            d.fmt_shift = fxpq_fmt{(int)v[22], (int)v[23], (int)v[24]};
            d.d_scale = dummy;
            d.d_shift = dummy;
        }
        const long long acc = v[16];
        const int32_t b = has_bias ? (int32_t)v[17] : 0;
        const int32_t m = (int32_t)v[25], h = (int32_t)v[26];
        ConvArgs a{};
        int32_t s_out = 0;
        bool need64 = false;
        const fxpq_status st = plan_conv(d, dummy, dummy, has_bias ? dummy : nullptr, dummy, a, &s_out, need64);
        long long generic = NA, code32 = NA, epi32 = NA, epi64 = NA;
        if (st == FXPQ_OK) {
            if (!has_scale) generic = qlayer_code(a, cblock_value<false>(a, 0, acc, b));
            if (a.v32) {
                code32 = qlayer_code32(a, (int)acc, b);
                const Epi32 e = make_epi32(a);
                const int32_t bk = e.has_bias ? b : 0;
                epi32 = epi32_code(e, (int)acc, (bk << e.bsl) >> e.bsr, (bk & e.fmask) != 0 ? 1 : 0);
            }
            const Epi64 e = make_epi64(a);
            if (e.ok) {
                const int32_t bk = e.has_bias ? b : 0;
                epi64 = has_scale ? epi64_code<true>(e, acc, bk, m, h) : epi64_code<false>(e, acc, bk, 0, 0);
            }
        }
        printf("%d %d %d %lld %lld %lld %lld\n", (int)st, a.v32, a.sh, generic, code32, epi32, epi64);
    }
    return 0;
}
