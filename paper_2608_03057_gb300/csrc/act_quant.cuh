// Per-token activation quantization (App. A.1.2) of one row: its scale and offset, and
// the fp16 codes of eight bf16 inputs (the quantizer's single-pass row kernel).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {

// Quantization range of a group: [lo, hi] -> (alpha, z) in the fp32 order
// alpha = (hi - lo) / denom, z = -lo / alpha; a constant group gets alpha = 1
// and z = half (symmetric range) or -lo.
__device__ inline void scale_of_range(float lo, float hi, float denom, float half, int mode, float* alpha,
                                      float* z) {
    float range = __fsub_rn(hi, lo);
    if (range == 0.0f) {
        *alpha = 1.0f;
        *z = (mode == TASQ_SYMRANGE) ? half : -lo;
    } else {
        *alpha = __fdiv_rn(range, denom);
        *z = __fdiv_rn(-lo, *alpha);
    }
}

// Scale of a row whose values span [lo, hi], at n bits: the symmetric range
// [-max|x|, max|x|] (TASQ_SYMRANGE) or [lo, hi] itself (TASQ_ASYM); ralpha = RN(1/alpha).
struct RowScale {
    float alpha, ralpha, z;
};
__device__ inline RowScale row_scale(float lo, float hi, int n_bits, int mode) {
    if (mode == TASQ_SYMRANGE) {
        hi = fmaxf(fabsf(lo), fabsf(hi));
        lo = -hi;
    }
    const int half = 1 << (n_bits - 1), qmax = (1 << n_bits) - 1;
    RowScale r;
    scale_of_range(lo, hi, float(qmax), float(half), mode, &r.alpha, &r.z);
    r.ralpha = __frcp_rn(r.alpha);
    return r;
}

// fp16 codes s = Q - half of the eight bf16 values of one 16-byte chunk, with
// Q = clamp(rint(x / alpha + z), 0, qmax) and x / alpha the correctly rounded quotient
// (div_rn_by: one Markstein correction from RN(1/alpha)).  Element pairs run on packed
// fp32 operations, each lane rounded exactly as the scalar one (the remainder
// fma(-q, a, x) is taken as fma(q, -a, x)).  RN(u + 1.5 * 2^23 + 0x6400) is the integer
// rint(u) + that constant, whose low 16 bits are the fp16 pattern 0x6400 + rint(u), i.e.
// the value 1024 + Q for 0 <= Q <= 255; one packed fp16 subtraction of 1024 + half then
// leaves s, clamped (packed) to [-half, half - 1].  For a finite row whose alpha is a
// normal float, u stays within (-0.5, qmax + 0.5), and any u in [-25600, 39935] clamps to
// the same code as clamping u before rounding.
__device__ __forceinline__ uint4 codes8_f16_of_bf16(const uint4& d, const RowScale& rs, int half) {
    const float2 ra2 = make_float2(rs.ralpha, rs.ralpha), na2 = make_float2(-rs.alpha, -rs.alpha);
    const float2 z2 = make_float2(rs.z, rs.z);
    const float2 magic2 = make_float2(12608512.0f, 12608512.0f);  // 1.5 * 2^23 + 0x6400
    const uint32_t w[4] = {d.x, d.y, d.z, d.w};
    uint32_t vb[8];
#pragma unroll
    for (int j = 0; j < 8; j += 2) {
        const float2 x2 = make_float2(__uint_as_float(w[j >> 1] << 16), __uint_as_float(w[j >> 1] & 0xFFFF0000u));
        const float2 q2 = ptx::fmul2(x2, ra2);
        const float2 r2 = ptx::ffma2(q2, na2, x2);
        const float2 u2 = ptx::fadd2(ptx::ffma2(r2, ra2, q2), z2);
        const float2 v2 = ptx::fadd2(u2, magic2);
        vb[j] = __float_as_uint(v2.x);
        vb[j + 1] = __float_as_uint(v2.y);
    }
    const uint32_t off = 0x6400u + uint32_t(half);
    const __half2 bias2 = __halves2half2(__ushort_as_half(uint16_t(off)), __ushort_as_half(uint16_t(off)));
    const __half2 lo2 = __float2half2_rn(float(-half)), hi2 = __float2half2_rn(float(half - 1));
    auto sub2 = [&](uint32_t v0, uint32_t v1) -> uint32_t {
        uint32_t p = __byte_perm(v0, v1, 0x5410);
        __half2 r = __hsub2(*reinterpret_cast<__half2*>(&p), bias2);
        r = __hmax2(__hmin2(r, hi2), lo2);
        return *reinterpret_cast<uint32_t*>(&r);
    };
    return make_uint4(sub2(vb[0], vb[1]), sub2(vb[2], vb[3]), sub2(vb[4], vb[5]), sub2(vb[6], vb[7]));
}

}  // namespace tasq
