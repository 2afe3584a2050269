// Numerics shared by the kernels that normalise logits over a vocabulary: base-2 exponentials of
// scaled logits, log-sum-exp and argmax merges, exact fixed-point probability masses and warp scans.
#pragma once

#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

namespace bp {

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// 2^(a - b) for scaled log-values, 0 when a is -inf
__device__ __forceinline__ float ex2d(float a, float b) { return a == -INFINITY ? 0.f : ex2(__fsub_rn(a, b)); }

// Probability mass in 2^-52 units: segment, slice and row sums are exact integer additions
// (a row's masses add up to about 1, i.e. about 2^52 units, far from the 2^64 limit).  Built
// from the float's fields with integer shifts (truncating below 2^-52): the float -> 64-bit
// integer conversion instruction runs on the slow FP64 pipe of this GPU.
__device__ __forceinline__ unsigned long long to_fix(float x) {
    const unsigned bits = __float_as_uint(x);
    const int e = (int)((bits >> 23) & 0xffu);  // x = mant * 2^(e - 150) for normal x >= 0
    if (e == 0 || (bits >> 31)) return 0ull;      // zero, denormal (< 2^-126) or negative
    const unsigned long long mant = (unsigned long long)((bits & 0x7fffffu) | 0x800000u);
    const int sh = e - 98;                         // x * 2^52 = mant * 2^(e - 98)
    if (sh >= 0) return sh < 40 ? mant << sh : ~0ull;  // x >= 2^12 is out of range: saturate
    return sh > -24 ? mant >> (-sh) : 0ull;
}

__device__ __forceinline__ float warp_incl_scan_f(float v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}
__device__ __forceinline__ unsigned long long warp_incl_scan(unsigned long long v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}
// merge two (scaled max, sum) pairs of a log-sum-exp
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
    const float M = fmaxf(m, m2);
    s = s * ex2d(m, M) + s2 * ex2d(m2, M);
    m = M;
}
// argmax with the lowest index winning ties
__device__ __forceinline__ void amax_merge(float& v, int& i, float v2, int i2) {
    if (v2 > v || (v2 == v && i2 < i)) {
        v = v2;
        i = i2;
    }
}

// Lane `lane` of a warp holding the values v[0..31] (per lane) ends with the warp-wide sum of
// value `lane`: a butterfly that halves the values it carries at every step (31 shuffles).
__device__ __forceinline__ float reduce_scatter32(float (&v)[32], int lane) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int q = 0; q < o; ++q) {
            const float send = up ? v[q] : v[q + o];
            const float keep = up ? v[q + o] : v[q];
            v[q] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    return v[0];
}

}  // namespace bp
