// Diagnostic probe of the 5th-generation tensor-core MMA kinds on this GPU
// (no counterpart in the paper): cycles per tcgen05.mma and the exactness of
// integer-valued operands, for kind::f16 (the exact route's operand type) and
// kind::f8f6f4 with e4m3 operands (every integer of magnitude <= 16 is exact)
// or e5m2 operands (integers with at most three significant bits, such as a
// weight truncated to b <= 4 planes and a 4-bit activation code: the operand
// type of the 8-bit route).  Both operands come from shared memory in the 128-byte
// swizzled K-major layout the contraction kernels use; one swizzle atom (128
// bytes of every row) is contracted `reps` times into an fp32 accumulator in
// tensor memory, so D = reps * (A . B^T over the atom) -- a long accumulation
// whose exact value the caller knows.
#include <cstdint>

#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {
namespace {

constexpr int PM = 128;         // MMA M (rows of A)
constexpr int ROW = 128;        // bytes of one operand row (one 128-byte swizzle atom)
constexpr int MAX_N = 256;

struct ProbeSmem {
    alignas(1024) uint8_t a[PM * ROW];
    alignas(1024) uint8_t b[MAX_N * ROW];
    uint64_t done;
    uint32_t tmem;
};

// D[tmem] (+)= A[smem] * B[smem]^T
template <int KIND>
__device__ __forceinline__ void mma_ss(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
    if constexpr (KIND == 0) {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc));
    } else {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc));
    }
}

// KIND 0: f16 x f16 (16 elements = 32 bytes per K step); KIND 1: e4m3 x e4m3,
// KIND 2: e5m2 x e5m2 (32 elements = 32 bytes per K step).  Either way an atom
// row is four K steps.
template <int KIND>
__global__ void __launch_bounds__(128) probe_mma_kernel(const uint8_t* __restrict__ ga, const uint8_t* __restrict__ gb,
                                                        int n, int reps, float* __restrict__ gd,
                                                        unsigned long long* __restrict__ cycles,
                                                        unsigned long long timeout_ns) {
    extern __shared__ uint8_t raw[];
    ProbeSmem* s = reinterpret_cast<ProbeSmem*>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // operands into the 128-byte swizzle: 16-byte chunk c of row r at c ^ (r & 7)
    for (int i = threadIdx.x; i < PM * 8; i += blockDim.x) {
        const int r = i >> 3, c = i & 7;
        *reinterpret_cast<uint4*>(s->a + r * ROW + ((c ^ (r & 7)) << 4)) =
            *reinterpret_cast<const uint4*>(ga + r * ROW + c * 16);
    }
    for (int i = threadIdx.x; i < n * 8; i += blockDim.x) {
        const int r = i >> 3, c = i & 7;
        *reinterpret_cast<uint4*>(s->b + r * ROW + ((c ^ (r & 7)) << 4)) =
            *reinterpret_cast<const uint4*>(gb + r * ROW + c * 16);
    }
    ptx::fence_proxy_async_smem();  // generic-proxy writes, read by the tensor core
    if (threadIdx.x == 0) {
        ptx::mbar_init(ptx::smem_u32(&s->done), 1);
        ptx::fence_mbar_init();
    }
    if (warp == 0) {
        ptx::tmem_alloc(ptx::smem_u32(&s->tmem), 512);
        ptx::tmem_relinquish();
        ptx::tc_fence_before();
    }
    ptx::cta_sync();
    ptx::tc_fence_after();
    const uint32_t tmem = s->tmem;
    // instruction descriptor: fp32 D; A and B format 0 (f16 for kind::f16, e4m3 for
    // kind::f8f6f4) or 1 (e5m2 for kind::f8f6f4)
    const uint32_t idesc = KIND == 2 ? ptx::idesc_e5m2_f32(PM, n) : ptx::idesc_f16_f32(PM, n);
    bool ok = true;
    if (threadIdx.x == 0) {
        const uint64_t adesc = ptx::sw128_kmajor_desc(ptx::smem_u32(s->a));
        const uint64_t bdesc = ptx::sw128_kmajor_desc(ptx::smem_u32(s->b));
        const long long c0 = clock64();
        for (int r = 0; r < reps; ++r)
#pragma unroll
            for (int k = 0; k < 4; ++k)  // 32 bytes along the rows per K step
                mma_ss<KIND>(tmem, adesc + uint64_t(2 * k), bdesc + uint64_t(2 * k), idesc, (r | k) ? 1u : 0u);
        ptx::mma_commit(ptx::smem_u32(&s->done));
        const uint32_t addr = ptx::smem_u32(&s->done);
        const uint64_t t0 = ptx::globaltimer();
        while (!ptx::mbar_try_wait(addr, 0)) {
            if (ptx::globaltimer() - t0 > timeout_ns) {
                ok = false;
                break;
            }
        }
        const long long c1 = clock64();
        cycles[blockIdx.x] = ok ? (unsigned long long)(c1 - c0) : 0ull;
    }
    ptx::cta_sync();
    ptx::tc_fence_after();
    if (blockIdx.x == 0 && cycles[0] != 0) {
        // D rows = TMEM lanes: warp w reads lanes 32 w .. 32 w + 31, 16 columns at a time
        for (int c = 0; c < n; c += 16) {
            uint32_t v[16];
            ptx::tmem_ld16(tmem + (uint32_t(warp * 32) << 16) + c, v);
            ptx::tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j) gd[(warp * 32 + lane) * n + c + j] = __uint_as_float(v[j]);
        }
    }
    ptx::tc_fence_before();
    ptx::cta_sync();
    if (warp == 0) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 512);
    }
}

}  // namespace
}  // namespace tasq

extern "C" __attribute__((visibility("default"))) int tasq_probe_mma(int kind, int n, int reps, const uint8_t* d_a,
                                                                    const uint8_t* d_b, float* d_d,
                                                                    unsigned long long* d_cycles, int ctas,
                                                                    tasq_stream stream) {
    using namespace tasq;
    if (kind < 0 || kind > 2) {
        set_noctx_error("kind must be 0 (f16), 1 (e4m3) or 2 (e5m2)");
        return TASQ_ERR_INVALID_ARG;
    }
    if (n < 16 || n > MAX_N || n % 16 || reps < 1 || reps > (1 << 20) || ctas < 1 || ctas > 1024 || !d_a || !d_b ||
        !d_d || !d_cycles) {
        set_noctx_error("need 16 <= n <= 256, n % 16 == 0, 1 <= reps <= 2^20, 1 <= ctas <= 1024 and pointers");
        return TASQ_ERR_INVALID_ARG;
    }
    if ((reinterpret_cast<uintptr_t>(d_a) | reinterpret_cast<uintptr_t>(d_b)) & 15u) {
        set_noctx_error("d_a and d_b must be 16-byte aligned");
        return TASQ_ERR_UNSUPPORTED;
    }
    // at least 120 KB of shared memory: one CTA per SM, so that no CTA waits for
    // another's tensor memory (each allocates all 512 columns)
    const int smem = int(sizeof(ProbeSmem)) + 1024 > 120 * 1024 ? int(sizeof(ProbeSmem)) + 1024 : 120 * 1024;
    auto kernel = kind == 0 ? probe_mma_kernel<0> : kind == 1 ? probe_mma_kernel<1> : probe_mma_kernel<2>;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) {
        kernel<<<ctas, 128, smem, (cudaStream_t)stream>>>(d_a, d_b, n, reps, d_d, d_cycles, 2000000000ull);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) {
        set_noctx_error(cudaGetErrorString(e));
        return TASQ_ERR_CUDA;
    }
    return TASQ_OK;
}
