// fxpq_common.cuh -- internal helpers shared by the libfxpq.so translation units.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "fxpq.h"

namespace fxpq {

// ---------------------------------------------------------------- host-side bookkeeping
// Device address of the latched status word (one per device; defined in fxpq_host.cu).
int* status_ptr();
// Count one kernel launch (for benchmarks) and check the launch error.
fxpq_status after_launch(const char* what);
void note_launch();

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

inline bool fmt_ok(const fxpq_fmt& f, int max_bits = 16) {
    return f.bits >= 2 && f.bits <= max_bits && (f.is_signed == 0 || f.is_signed == 1) && f.fl >= -32 &&
           f.fl <= 40;
}
// Formats of standalone code tensors may also be 1-bit: the levels {0, 1} (S = 0) or the binary
// quantizer (S = 1, Eq. fp_1_bit_quantization).
inline bool fmt_ok1(const fxpq_fmt& f, int max_bits = 16) {
    return f.bits == 1 ? (f.is_signed == 0 || f.is_signed == 1) && f.fl >= -32 && f.fl <= 40 : fmt_ok(f, max_bits);
}
inline int planes_of(const fxpq_fmt& f) { return f.bits > 8 ? 2 : 1; }
inline int64_t qmin_of(const fxpq_fmt& f) { return f.is_signed ? -(int64_t(1) << (f.bits - 1)) : 0; }
inline int64_t qmax_of(const fxpq_fmt& f) { return (int64_t(1) << (f.bits - f.is_signed)) - 1; }
inline bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ---------------------------------------------------------------- device helpers
__device__ __forceinline__ void latch_status(int* st, int code) {
    if (st) atomicCAS(st, 0, code);
}

// Round half to even of v / 2^sh for sh >= 1 (exact, int64): the FxP-QLayer's shift.  (Host-callable
// like the rest of the epilogue arithmetic, so that the CPU tests can run it.)
__host__ __device__ __forceinline__ long long rne_shift(long long v, int sh) {
    long long q = v >> sh;  // floor (arithmetic shift)
    unsigned long long rem = (unsigned long long)(v - (q << sh));
    unsigned long long half = 1ull << (sh - 1);
    q += (rem > half) || (rem == half && (q & 1));
    return q;
}

// value * 2^(fl_out - s) rounded half-even, clipped to [lo, hi]  (sh = s - fl_out)
__host__ __device__ __forceinline__ long long requant_value(long long v, int sh, long long lo, long long hi) {
    long long q;
    if (sh > 0)
        q = rne_shift(v, sh);
    else
        q = v << (-sh);
    return q < lo ? lo : (q > hi ? hi : q);
}

// Code <-> fp16 limb planes: code = 256*hi + lo with lo in [0,255].
__device__ __forceinline__ void split_limbs(int code, __half& hi, __half& lo) {
    int h = code >> 8;  // floor division
    int l = code - (h << 8);
    hi = __int2half_rn(h);
    lo = __int2half_rn(l);
}

// fp16 code tensors are plane-major: a k > 8 tensor stores its hi plane (a whole tensor) and then
// its lo plane, plane_stride elements later.  idx indexes one plane.
__device__ __forceinline__ int code_get(const __half* __restrict__ t, long long idx, int planes, long long plane_stride) {
    if (planes == 1) return __half2int_rn(t[idx]);
    return (__half2int_rn(t[idx]) << 8) + __half2int_rn(t[plane_stride + idx]);
}

__device__ __forceinline__ void code_put(__half* __restrict__ t, long long idx, int planes, long long plane_stride,
                                         int code) {
    if (planes == 1) {
        t[idx] = __int2half_rn(code);
    } else {
        __half h, l;
        split_limbs(code, h, l);
        t[idx] = h;
        t[plane_stride + idx] = l;
    }
}

}  // namespace fxpq
