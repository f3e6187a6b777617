// Quantizers (App. A.1), weight packing (App. F.1) and the failure-detection
// self test.  All kernels here are bandwidth-bound: 16-byte vector loads and
// stores, warp-shuffle reductions, one warp per row.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdio>
#include <mutex>

#include "act_quant.cuh"
#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {
namespace {

constexpr int kRowWarps = 8;  // rows per 256-thread block
// Rows per block of the single-pass per-token kernel: small blocks spread the
// one wave of rows evenly over the SMs (blocks, not warps, are what get placed).
constexpr int kRegRowWarps = 2;
// L2 prefetch of the input ahead of the dependency wait: the first kPrefetchBlocks
// blocks take one slice each, for inputs up to half of the 129 MB L2
constexpr int kPrefetchBlocks = 128;
constexpr uint64_t kPrefetchMaxBytes = 64ull << 20;

// Eight consecutive input floats (as fp32) from a 16-byte (bf16) or two
// 16-byte (fp32) chunks.  `i` counts 8-element groups along the row.
__device__ inline void load8(const void* row, int dtype, int64_t i, float v[8]) {
    if (dtype == TASQ_F32) {
        const float4* p = reinterpret_cast<const float4*>(row) + 2 * i;
        float4 a = __ldg(p), b = __ldg(p + 1);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    } else {
        uint4 r = __ldg(reinterpret_cast<const uint4*>(row) + i);
        uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[2 * j] = __uint_as_float(w[j] << 16);
            v[2 * j + 1] = __uint_as_float(w[j] & 0xFFFF0000u);
        }
    }
}

__device__ inline float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ inline float warp_min(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ inline int warp_sum(int v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Activation code: Q = clamp(rint(x / alpha + z), 0, qmax), s = Q - half.
// ralpha = RN(1 / alpha); x / alpha is still rounded exactly as IEEE division.
__device__ inline int act_code(float x, float alpha, float ralpha, float z, int qmax, int half) {
    const float u = __fadd_rn(div_rn_by(x, alpha, ralpha), z);
    // u lies in [-1, qmax + 1] up to rounding for x inside the quantization range;
    // clamp first so the bit trick's |u| <= 2^22 precondition always holds
    const int q = rint_small(fminf(fmaxf(u, -2.0f), float(qmax) + 2.0f));
    return min(max(q, 0), qmax) - half;
}

// Codes s[0..7] of 8-element group i: int8, or fp16 (and, for TASQ_CODES_F16_E5M2,
// the same codes as e5m2 bytes at out8).
__device__ inline void store8_codes(void* out, int code_fmt, int64_t i, const int s[8], void* out8 = nullptr) {
    if (code_fmt == TASQ_CODES_S8) {
        uint2 pk;
        pk.x = (s[0] & 0xFF) | ((s[1] & 0xFF) << 8) | ((s[2] & 0xFF) << 16) | ((uint32_t)(s[3] & 0xFF) << 24);
        pk.y = (s[4] & 0xFF) | ((s[5] & 0xFF) << 8) | ((s[6] & 0xFF) << 16) | ((uint32_t)(s[7] & 0xFF) << 24);
        reinterpret_cast<uint2*>(out)[i] = pk;
    } else {
        uint4 pk;
        uint32_t h[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) h[j] = __half_as_ushort(__int2half_rn(s[j]));
        pk.x = h[0] | (h[1] << 16);
        pk.y = h[2] | (h[3] << 16);
        pk.z = h[4] | (h[5] << 16);
        pk.w = h[6] | (h[7] << 16);
        reinterpret_cast<uint4*>(out)[i] = pk;
        if (code_fmt == TASQ_CODES_F16_E5M2)
            reinterpret_cast<uint2*>(out8)[i] = make_uint2(ptx::e5m2x4(pk.x, pk.y), ptx::e5m2x4(pk.z, pk.w));
    }
}

// ---------------------------------------------------------------- weights --
// mode TASQ_SYMRANGE: range [-max|w|, max|w|] (z = 128); TASQ_ASYM: the channel's
// [min, max] and a real zero point, zcw_out[n] = 128 - z.
__global__ void __launch_bounds__(256) quant_weights_kernel(const void* __restrict__ w, int dtype, int N, int K,
                                                            int mode, int8_t* __restrict__ sw, float* __restrict__ cw,
                                                            float* __restrict__ zcw_out,
                                                            float* __restrict__ alpha_out) {
    int lane = threadIdx.x & 31;
    int n = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (n >= N) return;
    const char* row = reinterpret_cast<const char*>(w) + int64_t(n) * K * (dtype == TASQ_F32 ? 4 : 2);
    int groups = K / 8;
    float amax = 0.0f, lo = INFINITY, hi = -INFINITY;
    for (int i = lane; i < groups; i += 32) {
        float v[8];
        load8(row, dtype, i, v);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            amax = fmaxf(amax, fabsf(v[j]));
            lo = fminf(lo, v[j]);
            hi = fmaxf(hi, v[j]);
        }
    }
    if (mode == TASQ_ASYM) {
        lo = warp_min(lo);
        hi = warp_max(hi);
    } else {
        amax = warp_max(amax);
        lo = -amax;
        hi = amax;
    }
    float alpha, z;
    scale_of_range(lo, hi, 256.0f, 128.0f, mode, &alpha, &z);
    int8_t* srow = sw + int64_t(n) * K;
    for (int i = lane; i < groups; i += 32) {
        float v[8];
        load8(row, dtype, i, v);
        uint32_t pk[2] = {0u, 0u};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            float u = __fadd_rn(__fdiv_rn(v[j], alpha), z);
            int q = __float2int_rd(u);  // floor
            q = min(max(q, 0), 255) - 128;
            pk[j >> 2] |= uint32_t(q & 0xFF) << (8 * (j & 3));
        }
        reinterpret_cast<uint2*>(srow)[i] = make_uint2(pk[0], pk[1]);
    }
    if (lane == 0) {
        cw[n] = __fmul_rn(alpha, __fdiv_rn(256.0f, 255.0f));
        if (zcw_out) zcw_out[n] = __fsub_rn(128.0f, z);
        if (alpha_out) alpha_out[n] = alpha;
    }
}

// ------------------------------------------------------ activations, token --
__global__ void __launch_bounds__(256) quant_act_token_kernel(const void* __restrict__ x, int dtype, int M, int K,
                                                              int n_bits, int mode, void* __restrict__ codes,
                                                              int code_fmt, float* __restrict__ alpha_out,
                                                              float* __restrict__ zc_out,
                                                              int32_t* __restrict__ code_sums) {
    int lane = threadIdx.x & 31;
    int m = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (m >= M) return;
    const char* row = reinterpret_cast<const char*>(x) + int64_t(m) * K * (dtype == TASQ_F32 ? 4 : 2);
    int groups = K / 8;
    float lo = INFINITY, hi = -INFINITY;
    for (int i = lane; i < groups; i += 32) {
        float v[8];
        load8(row, dtype, i, v);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            lo = fminf(lo, v[j]);
            hi = fmaxf(hi, v[j]);
        }
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    if (mode == TASQ_SYMRANGE) {
        hi = fmaxf(fabsf(lo), fabsf(hi));
        lo = -hi;
    }
    const int half = 1 << (n_bits - 1), qmax = (1 << n_bits) - 1;
    float alpha, z;
    scale_of_range(lo, hi, float(qmax), float(half), mode, &alpha, &z);
    const float ralpha = __frcp_rn(alpha);
    char* out = reinterpret_cast<char*>(codes) + int64_t(m) * K * (code_fmt == TASQ_CODES_S8 ? 1 : 2);
    // TASQ_CODES_F16_E5M2: the e5m2 copy follows the M x K fp16 codes
    char* out8 = reinterpret_cast<char*>(codes) + int64_t(M) * K * 2 + int64_t(m) * K;
    int csum = 0;
    for (int i = lane; i < groups; i += 32) {
        float v[8];
        load8(row, dtype, i, v);
        int s[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            s[j] = act_code(v[j], alpha, ralpha, z, qmax, half);
            csum += s[j];
        }
        store8_codes(out, code_fmt, i, s, out8);
    }
    if (code_sums) csum = warp_sum(csum);
    if (lane == 0) {
        alpha_out[m] = alpha;
        zc_out[m] = __fsub_rn(float(half), z);
        if (code_sums) code_sums[m] = csum;
    }
}

// Single-pass per-token quantization: one warp per row, the whole row held in
// registers as NPL 16-byte chunks per lane (chunk c of the row is lane c % 32,
// slot c / 32), so every load is issued before the min/max reduction.  SUMS:
// also write the row's code sum (asymmetric weights need it).
template <int NPL, int DTYPE, int CODES, bool SUMS>
__global__ void __launch_bounds__(kRegRowWarps * 32) quant_act_rowreg_kernel(const void* __restrict__ x, int M, int K, int n_bits,
                                                               int mode, void* __restrict__ codes,
                                                               float* __restrict__ alpha_out,
                                                               float* __restrict__ zc_out,
                                                               int32_t* __restrict__ code_sums) {
    constexpr int EPC = DTYPE == TASQ_F32 ? 4 : 8;  // elements per 16-byte chunk
    const int lane = threadIdx.x & 31;
    const int m = blockIdx.x * kRegRowWarps + (threadIdx.x >> 5);
    // Launched with programmatic dependent launch, so the first blocks may run beside
    // the previous kernel's last CTAs.  They pull the whole input into L2 meanwhile,
    // one slice each: L2 is the GPU's point of coherence, so if the previous kernel
    // writes x after this, its stores update the lines and the loads below (issued
    // after the wait) see them.  Nothing else is read or written before the wait
    // (the previous kernel may still read the code buffer).
    if (threadIdx.x == 0 && blockIdx.x < kPrefetchBlocks) {
        const uint64_t total = uint64_t(M) * uint64_t(K) * (DTYPE == TASQ_F32 ? 4u : 2u);  // K % 8 == 0: 16-byte rows
        const uint64_t slice = ((total + kPrefetchBlocks - 1) / kPrefetchBlocks + 15) & ~uint64_t(15);
        const uint64_t lo = uint64_t(blockIdx.x) * slice;
        if (lo < total && total <= kPrefetchMaxBytes) {
            const uint64_t n = total - lo < slice ? total - lo : slice;
            ptx::prefetch_l2_bulk(reinterpret_cast<const char*>(x) + lo, uint32_t(n));
        }
    }
    ptx::grid_dependency_wait();
    // let the next kernel's CTAs start their prologue on SMs this grid vacates;
    // they still wait for this grid's completion before reading its output
    ptx::grid_launch_dependents();
    if (m >= M) return;
    const int chunks = K / EPC;
    const uint4* row = reinterpret_cast<const uint4*>(x) + int64_t(m) * chunks;
    uint4 d[NPL];
#pragma unroll
    for (int k = 0; k < NPL; ++k) {
        const int c = lane + 32 * k;
        d[k] = c < chunks ? __ldg(row + c) : make_uint4(0, 0, 0, 0);
    }
    auto elem = [&](const uint4& v, int j) -> float {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        if (DTYPE == TASQ_F32) return __uint_as_float(w[j]);
        return __uint_as_float((j & 1) ? (w[j >> 1] & 0xFFFF0000u) : (w[j >> 1] << 16));
    };
    float lo = INFINITY, hi = -INFINITY;
    if constexpr (DTYPE == TASQ_BF16) {
        // bf16 pairs compared as bf16 (exact), one instruction per two elements
        __nv_bfloat162 mn = __float2bfloat162_rn(INFINITY), mx = __float2bfloat162_rn(-INFINITY);
#pragma unroll
        for (int k = 0; k < NPL; ++k) {
            if (lane + 32 * k < chunks) {
                const uint32_t w[4] = {d[k].x, d[k].y, d[k].z, d[k].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const __nv_bfloat162 p = *reinterpret_cast<const __nv_bfloat162*>(&w[j]);
                    mn = __hmin2(mn, p);
                    mx = __hmax2(mx, p);
                }
            }
        }
        lo = fminf(__low2float(mn), __high2float(mn));
        hi = fmaxf(__low2float(mx), __high2float(mx));
    } else {
#pragma unroll
        for (int k = 0; k < NPL; ++k) {
            if (lane + 32 * k < chunks) {
#pragma unroll
                for (int j = 0; j < EPC; ++j) {
                    const float f = elem(d[k], j);
                    lo = fminf(lo, f);
                    hi = fmaxf(hi, f);
                }
            }
        }
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    const RowScale rs = row_scale(lo, hi, n_bits, mode);
    const float alpha = rs.alpha, z = rs.z, ralpha = rs.ralpha;
    const int half = 1 << (n_bits - 1), qmax = (1 << n_bits) - 1;
    const float qmaxf = float(qmax);
    const float2 ra2 = make_float2(ralpha, ralpha), na2 = make_float2(-alpha, -alpha), z2 = make_float2(z, z);
    // 1.5 * 2^23 + 0x6400: RN(u + this) is the integer rint(u) + this, whose fp32 bits
    // end in the 16 bits 0x6400 + rint(u) (for 0 <= rint(u) <= 255)
    const float2 magic2 = make_float2(12608512.0f, 12608512.0f);
    char* out = reinterpret_cast<char*>(codes) + int64_t(m) * K * (CODES == TASQ_CODES_S8 ? 1 : 2);
    // TASQ_CODES_F16_E5M2: the e5m2 copy follows the M x K fp16 codes
    char* out8 = reinterpret_cast<char*>(codes) + int64_t(M) * K * 2 + int64_t(m) * K;
    int csum = 0;  // sum of this lane's codes Q - half (kept only when code_sums is set)
#pragma unroll
    for (int k = 0; k < NPL; ++k) {
        const int c = lane + 32 * k;
        if (c >= chunks) continue;
        if constexpr (DTYPE == TASQ_BF16 && CODES != TASQ_CODES_S8 && !SUMS) {
            const uint4 pk = codes8_f16_of_bf16(d[k], rs, half);
            reinterpret_cast<uint4*>(out)[c] = pk;
            if constexpr (CODES == TASQ_CODES_F16_E5M2)
                reinterpret_cast<uint2*>(out8)[c] = make_uint2(ptx::e5m2x4(pk.x, pk.y), ptx::e5m2x4(pk.z, pk.w));
        } else {
            // vb[j]: fp32 bits of Q + 1.5 * 2^23 + 0x6400 with Q = clamp(rint(x / alpha + z),
            // 0, qmax), so the low 16 bits are 0x6400 + Q (clamping u to the integer bounds
            // before rounding gives the same Q as rounding first); x / alpha as div_rn_by.  Element pairs: every packed
            // f32x2 operation rounds each lane exactly as the scalar one (the divide's
            // remainder fma(-q, a, x) is taken as fma(q, -a, x)).
            uint32_t vb[EPC];
    #pragma unroll
            for (int j = 0; j < EPC; j += 2) {
                const float2 x2 = make_float2(elem(d[k], j), elem(d[k], j + 1));
                const float2 q2 = ptx::fmul2(x2, ra2);
                const float2 r2 = ptx::ffma2(q2, na2, x2);
                const float2 u2 = ptx::fadd2(ptx::ffma2(r2, ra2, q2), z2);
                // For a finite row whose alpha is a normal float, u stays within (-0.5,
                // qmax + 0.5) (alpha and z come from the row's own range; the error is a few
                // ulps of qmax), so the clamp never binds and fp16 codes are clamped once,
                // packed, after the subtraction below instead (which also keeps codes in
                // range for inputs outside that class).  Integer codes and code sums take Q
                // from the bits here, so they clamp u first.
                float2 c2 = u2;
                if constexpr (CODES == TASQ_CODES_S8 || SUMS)
                    c2 = make_float2(fminf(fmaxf(u2.x, 0.0f), qmaxf), fminf(fmaxf(u2.y, 0.0f), qmaxf));
                const float2 v2 = ptx::fadd2(c2, magic2);
                vb[j] = __float_as_uint(v2.x);
                vb[j + 1] = __float_as_uint(v2.y);
            }
            int q[EPC];
    #pragma unroll
            for (int j = 0; j < EPC; ++j) q[j] = int(vb[j] & 0xFFFFu) - (0x6400 + half);
            if constexpr (SUMS) {
    #pragma unroll
                for (int j = 0; j < EPC; ++j) csum += q[j];
            }
            if (CODES == TASQ_CODES_S8) {
                if (EPC == 8) {
                    uint2 pk;
                    pk.x = (q[0] & 0xFF) | ((q[1] & 0xFF) << 8) | ((q[2] & 0xFF) << 16) | ((uint32_t)(q[3] & 0xFF) << 24);
                    pk.y = (q[4 % EPC] & 0xFF) | ((q[5 % EPC] & 0xFF) << 8) | ((q[6 % EPC] & 0xFF) << 16) |
                           ((uint32_t)(q[7 % EPC] & 0xFF) << 24);
                    reinterpret_cast<uint2*>(out)[c] = pk;
                } else {
                    reinterpret_cast<uint32_t*>(out)[c] =
                        (q[0] & 0xFF) | ((q[1] & 0xFF) << 8) | ((q[2 % EPC] & 0xFF) << 16) | ((uint32_t)(q[3 % EPC] & 0xFF) << 24);
                }
            } else {
                // fp16 of a small integer s: the bits 0x6400 + (s + half) hold 1024 + s + half
                // exactly; one packed subtraction of 1024 + half leaves s
                const uint32_t off = 0x6400u + uint32_t(half);
                const __half2 bias2 = __halves2half2(__ushort_as_half(uint16_t(off)), __ushort_as_half(uint16_t(off)));
                // the low halves of two vb words, 0x6400 + Q each, are the fp16 values
                // 1024 + Q; one packed subtraction of 1024 + half leaves the codes s = Q - half
                const __half2 lo2 = __float2half2_rn(float(-half)), hi2 = __float2half2_rn(float(half - 1));
                auto sub2 = [&](uint32_t v0, uint32_t v1) -> uint32_t {
                    uint32_t w = __byte_perm(v0, v1, 0x5410);
                    __half2 r = __hsub2(*reinterpret_cast<__half2*>(&w), bias2);
                    if constexpr (!SUMS) r = __hmax2(__hmin2(r, hi2), lo2);
                    return *reinterpret_cast<uint32_t*>(&r);
                };
                const uint32_t* h = vb;
                if (EPC == 8) {
                    uint4 pk;
                    pk.x = sub2(h[0], h[1]);
                    pk.y = sub2(h[2], h[3]);
                    pk.z = sub2(h[4 % EPC], h[5 % EPC]);
                    pk.w = sub2(h[6 % EPC], h[7 % EPC]);
                    reinterpret_cast<uint4*>(out)[c] = pk;
                    if constexpr (CODES == TASQ_CODES_F16_E5M2)
                        reinterpret_cast<uint2*>(out8)[c] = make_uint2(ptx::e5m2x4(pk.x, pk.y), ptx::e5m2x4(pk.z, pk.w));
                } else {
                    const uint2 pk = make_uint2(sub2(h[0], h[1]), sub2(h[2 % EPC], h[3 % EPC]));
                    reinterpret_cast<uint2*>(out)[c] = pk;
                    if constexpr (CODES == TASQ_CODES_F16_E5M2) reinterpret_cast<uint32_t*>(out8)[c] = ptx::e5m2x4(pk.x, pk.y);
                }
            }
        }
    }
    if constexpr (SUMS) csum = warp_sum(csum);
    if (lane == 0) {
        alpha_out[m] = alpha;
        zc_out[m] = __fsub_rn(float(half), z);
        if constexpr (SUMS) code_sums[m] = csum;
    }
}

template <int NPL, int DTYPE>
cudaError_t launch_rowreg(const void* x, int M, int K, int n_bits, int mode, void* codes, int code_fmt, float* alpha,
                          float* zc, int32_t* sums, cudaStream_t st) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3((M + kRegRowWarps - 1) / kRegRowWarps);
    cfg.blockDim = dim3(kRegRowWarps * 32);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    auto kernel = code_fmt == TASQ_CODES_S8
                      ? (sums ? quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_S8, true>
                              : quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_S8, false>)
                  : code_fmt == TASQ_CODES_F16
                      ? (sums ? quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_F16, true>
                              : quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_F16, false>)
                      : (sums ? quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_F16_E5M2, true>
                              : quant_act_rowreg_kernel<NPL, DTYPE, TASQ_CODES_F16_E5M2, false>);
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, x, M, K, n_bits, mode, codes, alpha, zc, sums);
    return e == cudaSuccess ? cudaGetLastError() : e;
}

template <int DTYPE>
bool dispatch_rowreg(int chunks_per_lane, const void* x, int M, int K, int n_bits, int mode, void* codes, int code_fmt,
                     float* alpha, float* zc, int32_t* sums, cudaStream_t st, cudaError_t* e) {
    if (chunks_per_lane <= 2) *e = launch_rowreg<2, DTYPE>(x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, sums, st);
    else if (chunks_per_lane <= 5) *e = launch_rowreg<5, DTYPE>(x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, sums, st);
    else if (chunks_per_lane <= 9) *e = launch_rowreg<9, DTYPE>(x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, sums, st);
    else if (chunks_per_lane <= 18)
        *e = launch_rowreg<18, DTYPE>(x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, sums, st);
    else if (chunks_per_lane <= 24)
        *e = launch_rowreg<24, DTYPE>(x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, sums, st);
    else return false;
    return true;
}

// ----------------------------------------------------- activations, tensor --
// Order-preserving map of a float onto an unsigned key.
__device__ inline uint32_t order_key(float f) {
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ inline float key_value(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// scratch[0] = ~key(min), scratch[1] = key(max); both start at 0.
__global__ void __launch_bounds__(256) tensor_range_kernel(const void* __restrict__ x, int dtype, int64_t groups,
                                                           unsigned int* scratch) {
    float lo = INFINITY, hi = -INFINITY;
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < groups; i += int64_t(gridDim.x) * blockDim.x) {
        float v[8];
        load8(x, dtype, i, v);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            lo = fminf(lo, v[j]);
            hi = fmaxf(hi, v[j]);
        }
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    __shared__ float slo[8], shi[8];
    int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        slo[warp] = lo;
        shi[warp] = hi;
    }
    ptx::cta_sync();
    if (threadIdx.x == 0) {
        for (int i = 1; i < int(blockDim.x >> 5); ++i) {
            lo = fminf(lo, slo[i]);
            hi = fmaxf(hi, shi[i]);
        }
        if (lo <= hi) {
            atomicMax(&scratch[0], ~order_key(lo));
            atomicMax(&scratch[1], order_key(hi));
        }
    }
}

__global__ void __launch_bounds__(256) quant_act_tensor_kernel(const void* __restrict__ x, int dtype, int64_t groups,
                                                               int n_bits, int mode, void* __restrict__ codes,
                                                               int code_fmt, float* __restrict__ alpha_out,
                                                               float* __restrict__ zc_out,
                                                               const unsigned int* __restrict__ scratch) {
    float lo = key_value(~scratch[0]);
    float hi = key_value(scratch[1]);
    if (mode == TASQ_SYMRANGE) {
        hi = fmaxf(fabsf(lo), fabsf(hi));
        lo = -hi;
    }
    const int half = 1 << (n_bits - 1), qmax = (1 << n_bits) - 1;
    float alpha, z;
    scale_of_range(lo, hi, float(qmax), float(half), mode, &alpha, &z);
    const float ralpha = __frcp_rn(alpha);
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < groups; i += int64_t(gridDim.x) * blockDim.x) {
        float v[8];
        load8(x, dtype, i, v);
        int s[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) s[j] = act_code(v[j], alpha, ralpha, z, qmax, half);
        store8_codes(codes, code_fmt, i, s, reinterpret_cast<char*>(codes) + groups * 16);
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        alpha_out[0] = alpha;
        zc_out[0] = __fsub_rn(float(half), z);
    }
}

// --------------------------------------------------------- code row sums --
// One warp per row of codes [M][K] (K % 16 == 0): sums[m] = sum_k codes[m][k].
__global__ void __launch_bounds__(256) code_row_sums_kernel(const void* __restrict__ codes, int code_fmt, int M, int K,
                                                            int32_t* __restrict__ sums) {
    const int lane = threadIdx.x & 31;
    const int m = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (m >= M) return;
    int s = 0;
    if (code_fmt == TASQ_CODES_S8) {
        const char4* row = reinterpret_cast<const char4*>(codes) + int64_t(m) * (K / 4);
        for (int i = lane; i < K / 4; i += 32) {
            const char4 v = row[i];
            s += v.x + v.y + v.z + v.w;
        }
    } else {
        const __half2* row = reinterpret_cast<const __half2*>(codes) + int64_t(m) * (K / 2);
        for (int i = lane; i < K / 2; i += 32) {
            const float2 v = __half22float2(row[i]);
            s += int(v.x) + int(v.y);
        }
    }
    s = warp_sum(s);
    if (lane == 0) sums[m] = s;
}

// -------------------------------------------------------------------- pack --
__global__ void pack_header_kernel(int kind, int N, int K, int has_zp, PackedHeader* hdr) {
    PackedHeader h = packed_layout(kind, N, K);
    h.has_zp = has_zp;
    for (int b = 0; b <= kBMax; ++b) h.chunk_kb[b] = (b >= kBMin) ? 0x7FFFFFFF : 0;
    *hdr = h;
}

// One block per output channel: row sums and per-tap sums for every b, and
// the channel's longest certified chunk (in 64-wide K blocks) for every b.
__global__ void __launch_bounds__(256) pack_sums_kernel(const int8_t* __restrict__ sw, int kind, int N, int K, int Cin,
                                                        char* packed) {
    extern __shared__ int smem_sums[];  // [kNumB][KB] block abs sums
    const PackedHeader lay = packed_layout(kind, N, K);
    PackedHeader* hdr = reinterpret_cast<PackedHeader*>(packed);
    int32_t* rs = reinterpret_cast<int32_t*>(packed + lay.off_rs);
    int32_t* ts = reinterpret_cast<int32_t*>(packed + lay.off_ts);
    const int n = blockIdx.x;
    const int KB = (K + kCertKBlock - 1) / kCertKBlock;
    const int8_t* row = sw + int64_t(n) * K;
    __shared__ int red[kNumB][9];
    if (threadIdx.x < kNumB * 9) red[threadIdx.x / 9][threadIdx.x % 9] = 0;
    for (int i = threadIdx.x; i < kNumB * KB; i += blockDim.x) smem_sums[i] = 0;
    ptx::cta_sync();
    // per-thread partials: [b][tap] signed sums; block abs sums via shared atomics
    int part[kNumB][9];
#pragma unroll
    for (int bi = 0; bi < kNumB; ++bi)
#pragma unroll
        for (int t = 0; t < 9; ++t) part[bi][t] = 0;
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
        int v = row[k];
        int tap = (kind == TASQ_CONV3X3) ? k / Cin : 0;
        int kb = k / kCertKBlock;
#pragma unroll
        for (int bi = 0; bi < kNumB; ++bi) {
            int m = mask_code(v, bi + kBMin);
#pragma unroll
            for (int t = 0; t < 9; ++t)
                if (t == tap) part[bi][t] += m;
            atomicAdd(&smem_sums[bi * KB + kb], abs(m));
        }
    }
#pragma unroll
    for (int bi = 0; bi < kNumB; ++bi)
#pragma unroll
        for (int t = 0; t < 9; ++t) {
            int s = part[bi][t];
#pragma unroll
            for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
            if ((threadIdx.x & 31) == 0 && s) atomicAdd(&red[bi][t], s);
        }
    ptx::cta_sync();
    if (threadIdx.x < kNumB) {
        int bi = threadIdx.x;
        int tot = 0;
        for (int t = 0; t < 9; ++t) tot += red[bi][t];
        rs[bi * N + n] = tot;
        if (kind == TASQ_CONV3X3)
            for (int t = 0; t < 9; ++t) ts[(int64_t(bi) * N + n) * 9 + t] = red[bi][t];
    }
    // Longest chunk length C (in K blocks) such that EVERY window of C
    // consecutive blocks stays within the bound.  Windows (not only aligned
    // chunks) make the property monotone in C, so the minimum over channels is
    // valid for every channel.  C = (shortest window whose sum exceeds the
    // bound) - 1, found by two pointers over the non-negative block sums.
    ptx::cta_sync();
    if (threadIdx.x < kNumB) {
        const int bi = threadIdx.x;
        const int* S = smem_sums + bi * KB;
        int shortest = KB + 1;
        int64_t sum = 0;
        int l = 0;
        for (int r = 0; r < KB; ++r) {
            sum += S[r];
            while (sum > kCertLimit) {
                shortest = min(shortest, r - l + 1);
                sum -= S[l++];
            }
        }
        atomicMin(&hdr->chunk_kb[bi + kBMin], max(1, shortest - 1));
    }
}

// ------------------------------------------------------------- self test --
__global__ void selftest_timeout_kernel(int* status, unsigned long long timeout_ns) {
    __shared__ __align__(8) unsigned long long bar;
    if (threadIdx.x == 0) {
        uint32_t a = (uint32_t)__cvta_generic_to_shared(&bar);
        asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(1));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        unsigned long long t0;
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
        uint32_t done = 0;
        while (!done) {
            asm volatile(
                "{\n.reg .pred p;\n"
                "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                "selp.u32 %0, 1, 0, p;\n}\n"
                : "=r"(done)
                : "r"(a), "r"(0u)
                : "memory");
            if (done) break;
            unsigned long long t;
            asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
            if (t - t0 > timeout_ns) {
                set_status(status, TASQ_ERR_DEVICE_TIMEOUT);
                break;
            }
        }
    }
}

// Counts x / a pairs where the activation quantizer's quotient differs from
// IEEE division (bit patterns compared).  Each thread takes dividends and runs
// them against every divisor (the divisors are read by all lanes at once).
__global__ void __launch_bounds__(256) selftest_quotients_kernel(const float* __restrict__ x, int nx,
                                                                 const float* __restrict__ a, int na,
                                                                 unsigned long long* mismatches) {
    unsigned long long bad = 0;
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < nx; i += int64_t(gridDim.x) * blockDim.x) {
        const float xv = x[i];
        for (int j = 0; j < na; ++j) {
            const float av = a[j];
            const float ra = __frcp_rn(av);
            bad += __float_as_uint(div_rn_by(xv, av, ra)) != __float_as_uint(__fdiv_rn(xv, av));
        }
    }
    for (int o = 16; o; o >>= 1) bad += __shfl_xor_sync(0xffffffffu, bad, o);
    if ((threadIdx.x & 31) == 0 && bad) atomicAdd(mismatches, bad);
}

}  // namespace

cudaError_t launch_selftest_quotients(const float* x, int nx, const float* a, int na, unsigned long long* mismatches,
                                      cudaStream_t st) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int want = (nx + 255) / 256;
    selftest_quotients_kernel<<<want < 8 * sms ? want : 8 * sms, 256, 0, st>>>(x, nx, a, na, mismatches);
    return cudaGetLastError();
}

cudaError_t launch_quant_weights(const void* w, int dtype, int N, int K, int mode, int8_t* sw, float* cw,
                                 float* zcw, float* alpha, cudaStream_t st) {
    if (N == 0) return cudaSuccess;
    quant_weights_kernel<<<(N + kRowWarps - 1) / kRowWarps, 256, 0, st>>>(w, dtype, N, K, mode, sw, cw, zcw, alpha);
    return cudaGetLastError();
}

cudaError_t launch_quant_act_token(const void* x, int dtype, int M, int K, int n_bits, int mode, void* codes,
                                   int code_fmt, float* alpha, float* zc, int32_t* code_sums, cudaStream_t st) {
    if (M == 0) return cudaSuccess;
    // rows that fit in registers: one pass over HBM
    const int chunks = K * (dtype == TASQ_F32 ? 4 : 2) / 16;
    const int per_lane = (chunks + 31) / 32;
    cudaError_t e = cudaSuccess;
    if (dtype == TASQ_F32
            ? dispatch_rowreg<TASQ_F32>(per_lane, x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, code_sums, st, &e)
            : dispatch_rowreg<TASQ_BF16>(per_lane, x, M, K, n_bits, mode, codes, code_fmt, alpha, zc, code_sums, st, &e))
        return e;
    // longer rows: two passes (the second mostly from L2)
    quant_act_token_kernel<<<(M + kRowWarps - 1) / kRowWarps, 256, 0, st>>>(x, dtype, M, K, n_bits, mode, codes,
                                                                            code_fmt, alpha, zc, code_sums);
    return cudaGetLastError();
}

cudaError_t launch_quant_act_tensor(const void* x, int dtype, int64_t count, int n_bits, int mode, void* codes,
                                    int code_fmt, float* alpha, float* zc, unsigned int* scratch, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(scratch, 0, 16, st);
    if (e != cudaSuccess) return e;
    int64_t groups = count / 8;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int64_t want = (groups + 255) / 256;
    int grid = int(want < 4 * sms ? (want > 0 ? want : 1) : 4 * sms);
    tensor_range_kernel<<<grid, 256, 0, st>>>(x, dtype, groups, scratch);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    quant_act_tensor_kernel<<<grid, 256, 0, st>>>(x, dtype, groups, n_bits, mode, codes, code_fmt, alpha, zc,
                                                  scratch);
    return cudaGetLastError();
}

cudaError_t launch_code_row_sums(const void* codes, int code_fmt, int M, int K, int32_t* sums, cudaStream_t st) {
    if (M == 0) return cudaSuccess;
    code_row_sums_kernel<<<(M + kRowWarps - 1) / kRowWarps, 256, 0, st>>>(codes, code_fmt, M, K, sums);
    return cudaGetLastError();
}

cudaError_t launch_pack(int kind, const int8_t* sw, const float* cw, const float* zcw, const float* bias, int N, int K,
                        int Cin, void* packed, cudaStream_t st) {
    const PackedHeader lay = packed_layout(kind, N, K);
    char* p = reinterpret_cast<char*>(packed);
    cudaError_t e = cudaMemsetAsync(p, 0, lay.total, st);
    if (e != cudaSuccess) return e;
    pack_header_kernel<<<1, 1, 0, st>>>(kind, N, K, zcw ? 1 : 0, reinterpret_cast<PackedHeader*>(p));
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (N == 0) return cudaSuccess;
    if ((e = cudaMemcpyAsync(p + lay.off_w, sw, size_t(N) * K, cudaMemcpyDeviceToDevice, st)) != cudaSuccess) return e;
    if ((e = cudaMemcpyAsync(p + lay.off_cw, cw, size_t(N) * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess) return e;
    if (bias && (e = cudaMemcpyAsync(p + lay.off_bias, bias, size_t(N) * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
        return e;
    if (zcw && (e = cudaMemcpyAsync(p + lay.off_zcw, zcw, size_t(N) * 4, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
        return e;
    int KB = (K + kCertKBlock - 1) / kCertKBlock;
    size_t smem = size_t(kNumB) * KB * sizeof(int);
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(pack_sums_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
    }
    pack_sums_kernel<<<N, 256, smem, st>>>(sw, kind, N, K, Cin, p);
    return cudaGetLastError();
}

cudaError_t launch_selftest_timeout(int* status, unsigned long long timeout_ns, cudaStream_t st) {
    selftest_timeout_kernel<<<1, 32, 0, st>>>(status, timeout_ns);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Per-tensor activation quantization that allocates nothing.
//
// For callers that cannot allocate device memory at run time (an inference
// plugin whose host framework forbids allocation inside enqueue, a process
// whose memory is planned once up front, code that must not create a
// context-owned buffer), the reduction scratch of per-tensor quantization
// lives in a file-scope device array instead of context memory.  Each block
// of the first kernel writes the (min, max) of its own slice into its slot;
// the second kernel folds the slots in a fixed order, so the result does not
// depend on timing and no slot needs clearing between calls.  The array is
// 16 KB and stays resident on every GPU that loads the library, until exit.
// ---------------------------------------------------------------------------
namespace {

constexpr int kNoAllocMaxBlocks = 2048;
constexpr int64_t kNoAllocSlice = 32768;  // elements reduced per block
static __device__ __align__(256) float2 g_noalloc_ranges[kNoAllocMaxBlocks];

__global__ void __launch_bounds__(256) noalloc_range_kernel(const void* __restrict__ x, int dtype, int64_t count,
                                                            float2* ranges) {
    const int64_t g0 = blockIdx.x * (kNoAllocSlice / 8);
    const int64_t g1 = min(count / 8, g0 + kNoAllocSlice / 8);
    float lo = INFINITY, hi = -INFINITY;
    for (int64_t i = g0 + threadIdx.x; i < g1; i += blockDim.x) {
        float v[8];
        load8(x, dtype, i, v);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            lo = fminf(lo, v[j]);
            hi = fmaxf(hi, v[j]);
        }
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    __shared__ float slo[8], shi[8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        slo[warp] = lo;
        shi[warp] = hi;
    }
    ptx::cta_sync();
    if (threadIdx.x == 0) {
        for (int i = 1; i < int(blockDim.x >> 5); ++i) {
            lo = fminf(lo, slo[i]);
            hi = fmaxf(hi, shi[i]);
        }
        ranges[blockIdx.x] = make_float2(lo, hi);
    }
}

__global__ void __launch_bounds__(256) noalloc_quant_kernel(const void* __restrict__ x, int dtype, int64_t count,
                                                            int nranges, int n_bits, int mode, void* __restrict__ codes,
                                                            int code_fmt, float* __restrict__ alpha_out,
                                                            float* __restrict__ zc_out,
                                                            const float2* __restrict__ ranges) {
    __shared__ float s_lo, s_hi;
    if (threadIdx.x < 32) {
        float lo = INFINITY, hi = -INFINITY;
        for (int i = threadIdx.x; i < nranges; i += 32) {
            const float2 r = ranges[i];
            lo = fminf(lo, r.x);
            hi = fmaxf(hi, r.y);
        }
        lo = warp_min(lo);
        hi = warp_max(hi);
        if (threadIdx.x == 0) {
            s_lo = lo;
            s_hi = hi;
        }
    }
    ptx::cta_sync();
    float lo = s_lo, hi = s_hi;
    if (mode == TASQ_SYMRANGE) {
        hi = fmaxf(fabsf(lo), fabsf(hi));
        lo = -hi;
    }
    const int half = 1 << (n_bits - 1), qmax = (1 << n_bits) - 1;
    float alpha, z;
    scale_of_range(lo, hi, float(qmax), float(half), mode, &alpha, &z);
    const float ralpha = __frcp_rn(alpha);
    const int64_t groups = count / 8;
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < groups; i += int64_t(gridDim.x) * blockDim.x) {
        float v[8];
        load8(x, dtype, i, v);
        int sv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) sv[j] = act_code(v[j], alpha, ralpha, z, qmax, half);
        store8_codes(codes, code_fmt, i, sv);
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        alpha_out[0] = alpha;
        zc_out[0] = __fsub_rn(float(half), z);
    }
}

// Device address of g_noalloc_ranges, looked up once per device (the host-side
// name is only a stand-in for the device array).
std::mutex g_noalloc_mu;
void* g_noalloc_addr[64] = {};

int noalloc_fail(int code, const char* msg) {
    set_noctx_error(msg);
    return code;
}

}  // namespace

}  // namespace tasq

extern "C" __attribute__((visibility("default"))) int tasq_quant_act_tensor_noalloc(
    const void* d_x, int dtype, int M, int K, int n_bits, int mode, void* d_codes, int code_fmt, float* d_alpha,
    float* d_zc, tasq_stream stream) {
    using namespace tasq;
    if (dtype != TASQ_F32 && dtype != TASQ_BF16) return noalloc_fail(TASQ_ERR_INVALID_ARG, "dtype must be F32 or BF16");
    if (mode != TASQ_SYMRANGE && mode != TASQ_ASYM) return noalloc_fail(TASQ_ERR_INVALID_ARG, "mode must be SYMRANGE or ASYM");
    if (code_fmt != TASQ_CODES_S8 && code_fmt != TASQ_CODES_F16)
        return noalloc_fail(TASQ_ERR_INVALID_ARG, "code_fmt must be CODES_S8 or CODES_F16");
    if (n_bits < 2 || n_bits > 8) return noalloc_fail(TASQ_ERR_INVALID_ARG, "n_bits must be in 2..8");
    if (M < 0 || K <= 0) return noalloc_fail(TASQ_ERR_INVALID_ARG, "need M >= 0 and K > 0");
    if (K % 16) return noalloc_fail(TASQ_ERR_UNSUPPORTED, "K must be a multiple of 16");
    const int64_t count = int64_t(M) * K;
    if (count > int64_t(kNoAllocMaxBlocks) * kNoAllocSlice) {
        char msg[160];
        snprintf(msg, sizeof msg, "tensor of %lld elements exceeds the %lld-element limit of quantization without allocation",
                 (long long)count, (long long)(int64_t(kNoAllocMaxBlocks) * kNoAllocSlice));
        return noalloc_fail(TASQ_ERR_UNSUPPORTED, msg);
    }
    if (M == 0) return TASQ_OK;
    if (!d_x || !d_codes || !d_alpha || !d_zc) return noalloc_fail(TASQ_ERR_INVALID_ARG, "NULL pointer");
    if ((reinterpret_cast<uintptr_t>(d_x) | reinterpret_cast<uintptr_t>(d_codes)) & 15u)
        return noalloc_fail(TASQ_ERR_UNSUPPORTED, "d_x and d_codes must be 16-byte aligned");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return noalloc_fail(TASQ_ERR_CUDA, cudaGetErrorString(e));
    if (dev < 0 || dev >= 64) return noalloc_fail(TASQ_ERR_UNSUPPORTED, "device index above 63");
    void* ranges = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_noalloc_mu);
        if (!g_noalloc_addr[dev]) {
            e = cudaGetSymbolAddress(&g_noalloc_addr[dev], g_noalloc_ranges);
            if (e != cudaSuccess) {
                g_noalloc_addr[dev] = nullptr;
                return noalloc_fail(TASQ_ERR_CUDA, cudaGetErrorString(e));
            }
        }
        ranges = g_noalloc_addr[dev];
    }
    const int nranges = int((count + kNoAllocSlice - 1) / kNoAllocSlice);
    cudaStream_t st = (cudaStream_t)stream;
    noalloc_range_kernel<<<nranges, 256, 0, st>>>(d_x, dtype, count, reinterpret_cast<float2*>(ranges));
    if ((e = cudaGetLastError()) != cudaSuccess) return noalloc_fail(TASQ_ERR_CUDA, cudaGetErrorString(e));
    int sms = 148;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (count / 8 + 255) / 256;
    const int grid = int(want < 4 * sms ? want : 4 * sms);
    noalloc_quant_kernel<<<grid, 256, 0, st>>>(d_x, dtype, count, nranges, n_bits, mode, d_codes, code_fmt, d_alpha,
                                               d_zc, reinterpret_cast<const float2*>(ranges));
    if ((e = cudaGetLastError()) != cudaSuccess) return noalloc_fail(TASQ_ERR_CUDA, cudaGetErrorString(e));
    return TASQ_OK;
}

