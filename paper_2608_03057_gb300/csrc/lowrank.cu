// 16-bit low-rank branch of an SVD-split linear layer (SVDQuant's branch, which
// the paper's SVDQuant+TASQ pipelines keep beside the masked int8 weights: rank
// 32 for the 4-bit setting, 16 for the 6-bit one).  The layer computes
// y = Q(x) Q_b(R)^T + (x l2^T) l1^T; this file is the down-projection.  The
// masked contraction (tasq_masked_gemm_lr) adds the up-projection inside its
// integer accumulator, in the accumulator's units: (u / alpha) . (l1 / c_w)^T,
// as one more K block of fp16 MMAs, so this kernel writes u' = fp16(u / alpha[m])
// into a [M][64] fp16 block (one 128-byte swizzle atom per row; columns >= rank
// zero), u = bf16(x) l2^T accumulated in fp32.
//
// One CTA of sixteen warps per 16 rows of x; warp w takes the K steps
// [w S / 16, (w + 1) S / 16) of S = K / 16 on mma.m16n8k16 (bf16 operands, fp32
// accumulators): per batch of four steps it loads the x and l2 tiles with
// coalesced 16-byte loads, stores them to its shared-memory tiles and reads the
// MMA fragments back with ldmatrix; the sixteen partial sums meet in shared
// memory, added in warp order.  (The steps past s1 of the last batch reload step
// s0, in bounds, and issue no MMA.)  Launched as a programmatic dependent of the
// layer's quantization: only the final division by alpha waits for it.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {

PFN_cuTensorMapEncodeTiled_v12000 get_encode();  // gemm_tc.cu

namespace {

// Eight bf16 of x[row][k..k+7] (16 bytes); zeros past M
template <int DTYPE>
__device__ __forceinline__ uint4 x_oct(const void* x, int M, int K, int row, int k) {
    if (row >= M) return make_uint4(0u, 0u, 0u, 0u);
    if constexpr (DTYPE == TASQ_BF16) {
        return __ldg(reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(x) + int64_t(row) * K + k));
    } else {
        const float4* p = reinterpret_cast<const float4*>(static_cast<const float*>(x) + int64_t(row) * K + k);
        const float4 v0 = __ldg(p), v1 = __ldg(p + 1);
        const __nv_bfloat162 h0 = __floats2bfloat162_rn(v0.x, v0.y), h1 = __floats2bfloat162_rn(v0.z, v0.w);
        const __nv_bfloat162 h2 = __floats2bfloat162_rn(v1.x, v1.y), h3 = __floats2bfloat162_rn(v1.z, v1.w);
        return make_uint4(*reinterpret_cast<const uint32_t*>(&h0), *reinterpret_cast<const uint32_t*>(&h1),
                          *reinterpret_cast<const uint32_t*>(&h2), *reinterpret_cast<const uint32_t*>(&h3));
    }
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

constexpr int kDownWarps = 16;
constexpr int kDownBatch = 2;  // K steps per batch of loads

// Per warp and batch: x [kDownBatch][16 rows][16 k] and l2 [kDownBatch][R ranks][16 k]
// bf16 tiles, rows of 32 bytes with the two 16-byte halves swapped on odd rows
// (4 row groups of the same bank pattern -> conflict-free 8-row ldmatrix phases).
// A warp's partial sums [16][R] fp32 take its own tiles' place after its last batch.
template <int R>
struct DownWarpTiles {
    uint16_t xs[kDownBatch][16][16];
    uint16_t ls[kDownBatch][R][16];
};
template <int R>
struct DownSmem {
    DownWarpTiles<R> w[kDownWarps];
};
static_assert(sizeof(float) * 16 * 16 <= sizeof(DownWarpTiles<16>) && sizeof(float) * 16 * 32 <= sizeof(DownWarpTiles<32>),
              "partial sums fit a warp's tiles");

__device__ __forceinline__ uint32_t tile_off(int row, int half) { return uint32_t(row * 32 + ((half ^ (row >> 2 & 1)) << 4)); }

template <int DTYPE, int R>
__global__ void __launch_bounds__(kDownWarps * 32, 2)
    lowrank_down_kernel(const void* __restrict__ x, int M, int K, const uint16_t* __restrict__ l2,
                        const float* __restrict__ alpha, int per_tensor, uint16_t* __restrict__ u) {
    constexpr int NT = R / 8;  // 8-wide rank tiles
    extern __shared__ __align__(16) uint8_t smem_raw[];
    DownSmem<R>& sm = *reinterpret_cast<DownSmem<R>*>(smem_raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    const int m0 = blockIdx.x * 16;
    const int S = K / 16;
    const int s0 = (warp * S) / kDownWarps, s1 = ((warp + 1) * S) / kDownWarps;
    float d[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) d[nt][i] = 0.f;
    const uint32_t xs0 = ptx::smem_u32(&sm.w[warp].xs[0][0][0]), ls0 = ptx::smem_u32(&sm.w[warp].ls[0][0][0]);
    for (int st = s0; st < s1; st += kDownBatch) {
        // coalesced 16-byte loads of the batch: lane -> x row lane / 2, half lane % 2;
        // l2: the R x 32-byte tile in LP 16-byte pieces per lane (piece i of lane l is
        // 16-byte piece l + 32 i of the tile: row (l + 32 i) / 2, half l % 2)
        constexpr int LP = R / 16;
        uint4 xv[kDownBatch], lv[kDownBatch][LP];
#pragma unroll
        for (int q = 0; q < kDownBatch; ++q) {
            const int k0 = (st + q < s1 ? st + q : s0) * 16;
            xv[q] = x_oct<DTYPE>(x, M, K, m0 + (lane >> 1), k0 + (lane & 1) * 8);
#pragma unroll
            for (int i = 0; i < LP; ++i) {
                const int pc = lane + 32 * i;
                lv[q][i] = __ldg(reinterpret_cast<const uint4*>(l2 + int64_t(pc >> 1) * K + k0 + (pc & 1) * 8));
            }
        }
        __syncwarp();  // the previous batch's ldmatrix reads are done
#pragma unroll
        for (int q = 0; q < kDownBatch; ++q) {
            *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(&sm.w[warp].xs[q][0][0]) + tile_off(lane >> 1, lane & 1)) = xv[q];
#pragma unroll
            for (int i = 0; i < LP; ++i) {
                const int pc = lane + 32 * i;
                *reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(&sm.w[warp].ls[q][0][0]) + tile_off(pc >> 1, pc & 1)) =
                    lv[q][i];
            }
        }
        __syncwarp();
#pragma unroll
        for (int q = 0; q < kDownBatch; ++q) {
            if (st + q >= s1) break;
            // A (16 x 16, rows = x rows): matrices (rows 0-7 | 8-15) x (k 0-7 | 8-15)
            uint32_t a[4];
            ldmatrix_x4(xs0 + uint32_t(q * 16 * 32) + tile_off(lane & 15, lane >> 4), a);
#pragma unroll
            for (int np = 0; np < NT / 2; ++np) {
                // B of two rank tiles: matrices (ranks 16np + 0-7 | 8-15) x (k 0-7 | 8-15)
                uint32_t b[4];
                const int rank = np * 16 + (lane & 7) + ((lane >> 4) << 3);
                ldmatrix_x4(ls0 + uint32_t(q * R * 32) + tile_off(rank, (lane >> 3) & 1), b);
                ptx::mma_bf16_16816(d[2 * np], a, b[0], b[1]);
                ptx::mma_bf16_16816(d[2 * np + 1], a, b[2], b[3]);
            }
        }
    }
    __syncwarp();  // this warp's ldmatrix reads of its x tiles are done
    // the contraction that reads u' may start its set-up; alpha comes from the
    // previous kernel (the layer's quantization), whose launch this one overlaps
    ptx::grid_launch_dependents();
    ptx::grid_dependency_wait();
    auto red = [&](int w) { return reinterpret_cast<float(*)[R]>(&sm.w[w].xs[0][0][0]); };
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        red(warp)[g][nt * 8 + 2 * t] = d[nt][0];
        red(warp)[g][nt * 8 + 2 * t + 1] = d[nt][1];
        red(warp)[g + 8][nt * 8 + 2 * t] = d[nt][2];
        red(warp)[g + 8][nt * 8 + 2 * t + 1] = d[nt][3];
    }
    ptx::cta_sync();
    // u' rows of 64 fp16: the rank columns, then zeros
    for (int i = threadIdx.x; i < 16 * 64; i += blockDim.x) {
        const int row = i >> 6, col = i & 63, m = m0 + row;
        if (m >= M) continue;
        float v = 0.f;
        if (col < R) {
            v = red(0)[row][col];
#pragma unroll
            for (int w = 1; w < kDownWarps; ++w) v = __fadd_rn(v, red(w)[row][col]);
            v = __fdiv_rn(v, alpha[per_tensor ? 0 : m]);
        }
        u[int64_t(m) * 64 + col] = __half_as_ushort(__float2half_rn(v));
    }
}

// ---------------------------------------------------------------------------
// The same down-projection on the 5th-generation tensor cores, for bf16 x: a CTA
// of four warps per 128 rows computes D[128 rows][R] = x_tile . l2^T in tensor
// memory, tcgen05.mma kind::f16 with bf16 A (x, [128][64] per stage) and B (l2,
// [R][64] per stage), both K-major in the 128-byte swizzle, brought in by TMA
// through a ring of kTcStages stages (one thread loads, one thread issues the
// four K = 16 MMAs per stage).  Each warp then reads its 32 rows of D and writes
// u' = fp16(D / alpha).  Every wait is bounded: on a timeout the kernel records
// TASQ_ERR_DEVICE_TIMEOUT and skips its output.
constexpr int kTcStages = 4;
constexpr int kTcRows = 128;

template <int R>
struct DownTcSmem {
    alignas(1024) uint8_t xs[kTcStages][kTcRows * 128];
    alignas(1024) uint8_t ls[kTcStages][R * 128];
    uint64_t full[kTcStages], empty[kTcStages], done;
    uint32_t tmem;
    int abort;
};

__device__ __forceinline__ bool bounded_wait(uint32_t bar, uint32_t parity, unsigned long long timeout_ns,
                                             int* abort, bool ignore_abort = false) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if ((it & 63) == 0) {
            if (!ignore_abort && *(volatile int*)abort) return false;
            if (ptx::globaltimer() - t0 > timeout_ns) {
                *(volatile int*)abort = 1;
                return false;
            }
        }
    }
}

template <int R>
__global__ void __launch_bounds__(128)
    lowrank_down_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_l2, int M,
                           int K, const float* __restrict__ alpha, int per_tensor, uint16_t* __restrict__ u,
                           int* status, unsigned long long timeout_ns) {
    extern __shared__ uint8_t smem_raw[];
    DownTcSmem<R>* s =
        reinterpret_cast<DownTcSmem<R>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * kTcRows;
    const int KB = (K + 63) / 64;
    constexpr uint32_t kStageBytes = kTcRows * 128 + R * 128;
    // D: fp32, bf16 A and B (format code 1 in both fields), M = 128, N = R
    constexpr uint32_t idesc = ptx::idesc_f16_f32(kTcRows, R) | (1u << 7) | (1u << 10);
    if (warp == 0) {
        ptx::tmem_alloc(ptx::smem_u32(&s->tmem), 32);
        ptx::tmem_relinquish();
        ptx::tc_fence_before();
    }
    if (threadIdx.x == 32) {
        for (int i = 0; i < kTcStages; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->full[i]), 1);
            ptx::mbar_init(ptx::smem_u32(&s->empty[i]), 1);
        }
        ptx::mbar_init(ptx::smem_u32(&s->done), 1);
        s->abort = 0;
        ptx::fence_mbar_init();
        ptx::prefetch_tmap(&tm_x);
        ptx::prefetch_tmap(&tm_l2);
    }
    ptx::cta_sync();
    ptx::tc_fence_after();
    const uint32_t tmem = s->tmem;
    bool ok = true;
    int issued = 0;  // producer: stages loaded
    if (threadIdx.x == 0) {
        // producer: x is the layer's input and l2 a weight, both written before the
        // quantization this launch overlaps
        for (int kb = 0; kb < KB && ok; ++kb, ++issued) {
            const int st = kb % kTcStages;
            if (kb >= kTcStages &&
                !bounded_wait(ptx::smem_u32(&s->empty[st]), ((kb / kTcStages) - 1) & 1, timeout_ns, &s->abort)) {
                ok = false;
                break;
            }
            const uint32_t fb = ptx::smem_u32(&s->full[st]);
            ptx::mbar_arrive_expect_tx(fb, kStageBytes);
            ptx::tma_load_2d(ptx::smem_u32(s->xs[st]), &tm_x, fb, kb * 64, m0);
            ptx::tma_load_2d(ptx::smem_u32(s->ls[st]), &tm_l2, fb, kb * 64, 0);
        }
    } else if (threadIdx.x == 32) {
        // MMA issuer
        for (int kb = 0; kb < KB && ok; ++kb) {
            const int st = kb % kTcStages;
            if (!bounded_wait(ptx::smem_u32(&s->full[st]), (kb / kTcStages) & 1, timeout_ns, &s->abort)) {
                ok = false;
                break;
            }
            ptx::tc_fence_after();
            const uint64_t adesc = ptx::sw128_kmajor_desc(ptx::smem_u32(s->xs[st]));
            const uint64_t bdesc = ptx::sw128_kmajor_desc(ptx::smem_u32(s->ls[st]));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)  // K steps of 16 bf16 = 32 bytes along the rows
                asm volatile(
                    "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
                    "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem),
                    "l"(adesc + uint64_t(2 * kk)), "l"(bdesc + uint64_t(2 * kk)), "r"(idesc),
                    "r"((kb | kk) ? 1u : 0u));
            ptx::mma_commit(ptx::smem_u32(&s->empty[st]));
        }
        ptx::mma_commit(ptx::smem_u32(&s->done));
    }
    __syncwarp();
    // the contraction that reads u' may start its set-up; alpha comes from the
    // previous kernel (the layer's quantization)
    ptx::grid_launch_dependents();
    ptx::grid_dependency_wait();
    const bool got = bounded_wait(ptx::smem_u32(&s->done), 0, timeout_ns, &s->abort);
    ptx::tc_fence_after();
    if (got && !*(volatile int*)&s->abort) {
        uint32_t v[32];
        if constexpr (R == 32) {
            ptx::tmem_ld32(tmem + (uint32_t(warp * 32) << 16), v);
        } else {
            ptx::tmem_ld16(tmem + (uint32_t(warp * 32) << 16), *reinterpret_cast<uint32_t(*)[16]>(&v[0]));
        }
        ptx::tmem_wait_ld();
        const int m = m0 + warp * 32 + lane;
        if (m < M) {
            const float al = alpha[per_tensor ? 0 : m];
            uint32_t h[32];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float a0 = 2 * j < R ? __fdiv_rn(__uint_as_float(v[2 * j]), al) : 0.f;
                const float a1 = 2 * j + 1 < R ? __fdiv_rn(__uint_as_float(v[2 * j + 1]), al) : 0.f;
                const __half2 hh = __floats2half2_rn(a0, a1);
                h[j] = *reinterpret_cast<const uint32_t*>(&hh);
            }
#pragma unroll
            for (int j = 16; j < 32; ++j) h[j] = 0u;
            uint4* dst = reinterpret_cast<uint4*>(u + int64_t(m) * 64);
#pragma unroll
            for (int q = 0; q < 8; ++q) dst[q] = make_uint4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]);
        }
    }
    if (threadIdx.x == 0) {
        // copies still in flight land before the CTA may exit (only after an abort can
        // the MMA issuer have left a loaded stage unread)
        for (int kb = issued - kTcStages < 0 ? 0 : issued - kTcStages; kb < issued; ++kb)
            bounded_wait(ptx::smem_u32(&s->full[kb % kTcStages]), (kb / kTcStages) & 1, timeout_ns, &s->abort, true);
        if (*(volatile int*)&s->abort) set_status(status, TASQ_ERR_DEVICE_TIMEOUT);
    }
    ptx::tc_fence_before();
    ptx::cta_sync();
    if (warp == 0) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 32);
    }
}

}  // namespace

namespace {

// The tensor-core kernel for bf16 x (16-byte aligned x and l2); false when its
// tensor maps cannot be encoded.
template <int R>
bool launch_down_tc(const void* x, int M, int K, const uint16_t* l2, const float* alpha, int per_tensor, uint16_t* u,
                    int* status, unsigned long long timeout_ns, cudaStream_t st, cudaError_t* err) {
    auto encode = get_encode();
    if (!encode) return false;
    CUtensorMap tm_x, tm_l2;
    cuuint64_t dx[2] = {cuuint64_t(K), cuuint64_t(M)}, dl[2] = {cuuint64_t(K), cuuint64_t(R)};
    cuuint64_t sx[1] = {cuuint64_t(K) * 2}, sl[1] = {cuuint64_t(K) * 2};
    cuuint32_t bx[2] = {64, kTcRows}, bl[2] = {64, R}, es[2] = {1, 1};
    if (encode(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dx, sx, bx, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS ||
        encode(&tm_l2, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t*>(l2), dl, sl, bl, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return false;
    const int smem = int(sizeof(DownTcSmem<R>)) + 1024;
    cudaError_t e = cudaFuncSetAttribute(lowrank_down_tc_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) {
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3(unsigned((M + kTcRows - 1) / kTcRows));
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, lowrank_down_tc_kernel<R>, tm_x, tm_l2, M, K, alpha, per_tensor, u, status,
                               timeout_ns);
        if (e == cudaSuccess) e = cudaGetLastError();
    }
    *err = e;
    return true;
}

}  // namespace

cudaError_t launch_lowrank_down(const void* x, int dtype, int M, int K, const uint16_t* l2, int rank,
                                const float* alpha, int per_tensor, uint16_t* u, int* status,
                                unsigned long long timeout_ns, cudaStream_t st) {
    if (dtype == TASQ_BF16 && ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(l2)) & 15u) == 0) {
        cudaError_t e = cudaSuccess;
        if (rank == 16 ? launch_down_tc<16>(x, M, K, l2, alpha, per_tensor, u, status, timeout_ns, st, &e)
                       : launch_down_tc<32>(x, M, K, l2, alpha, per_tensor, u, status, timeout_ns, st, &e))
            return e;
    }
    const unsigned grid = unsigned((M + 15) / 16), block = kDownWarps * 32;
    auto launch = [&](auto kernel, size_t smem) {
        cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
        if (e != cudaSuccess) return e;
        // programmatic dependent launch: x and l2 are read while the quantization runs
        cudaLaunchConfig_t cfg{};
        cfg.gridDim = dim3(grid);
        cfg.blockDim = dim3(block);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, kernel, x, M, K, l2, alpha, per_tensor, u);
        return e == cudaSuccess ? cudaGetLastError() : e;
    };
    if (dtype == TASQ_BF16)
        return rank == 16 ? launch(lowrank_down_kernel<TASQ_BF16, 16>, sizeof(DownSmem<16>))
                          : launch(lowrank_down_kernel<TASQ_BF16, 32>, sizeof(DownSmem<32>));
    return rank == 16 ? launch(lowrank_down_kernel<TASQ_F32, 16>, sizeof(DownSmem<16>))
                      : launch(lowrank_down_kernel<TASQ_F32, 32>, sizeof(DownSmem<32>));
}

}  // namespace tasq
