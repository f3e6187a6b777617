// Masked contraction on int8 operands with int32 accumulators (warp-level
// mma.sync m16n8k32 s8.s8.s32): exact by construction.  Serves linear layers
// and 3x3 convolutions (implicit GEMM over K = 9*Cin, (kh, kw, cin) order).
//
// The operating-precision mask (Eq. hw_rightshift: keep the top b of the
// 8 stored planes) is one AND on each 32-bit register of four weight codes,
// applied right after the weight fragment is loaded from shared memory.
#include "tasq_internal.cuh"

namespace tasq {
namespace {

constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4, THREADS = 256;
constexpr int TILE_BYTES = BM * BK;  // one operand stage (A and B are both 128 x 64 int8)
constexpr int SMEM_BYTES = STAGES * 2 * TILE_BYTES;

// 16-byte chunk c of row r lives at chunk c ^ ((r >> 1) & 3): conflict-free ldmatrix.
__device__ inline uint32_t swz(int r, int c) { return uint32_t(r * BK + ((c ^ ((r >> 1) & 3)) << 4)); }

__device__ inline void cp_async16(uint32_t dst, const void* src, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(valid ? 16 : 0));
}
__device__ inline void cp_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ inline void cp_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}

__device__ inline void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ inline void mma_s8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// ZP: the four-term epilogue of asymmetric weights
template <bool CONV, bool ZP>
__global__ void __launch_bounds__(THREADS) gemm_s8_kernel(const GemmArgs a) {
    extern __shared__ __align__(128) uint8_t smem[];
    const uint32_t gbits = resolve_group_bits(a);
    if (gbits == 0) return;
    const int b = int(gbits & 15u);  // the layer's b (member 0 of a grouped call)

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int wm = warp >> 2, wn = warp & 3;  // 2 x 4 warps, 64 x 32 each
    const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM;
    // weight fragment ni of this thread holds channel n0 + wn * 32 + ni * 8 + lane / 4
    uint32_t wmask[4];
#pragma unroll
    for (int ni = 0; ni < 4; ++ni) wmask[ni] = mask_word(channel_bits(a, gbits, n0 + wn * 32 + ni * 8 + (lane >> 2)));
    const int M = a.M, N = a.N, K = a.K;
    const int8_t* __restrict__ X = reinterpret_cast<const int8_t*>(a.x);
    const int8_t* __restrict__ Wt = a.w;
    const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(smem);

    // Each thread copies chunk column c of rows r0 and r0 + 64, for A and B.
    const int c = tid & 3, r0 = tid >> 2;
    int pix_b[2], pix_h[2], pix_w[2];
    bool a_row_ok[2], b_row_ok[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        int m = m0 + r0 + 64 * i;
        a_row_ok[i] = m < M;
        b_row_ok[i] = n0 + r0 + 64 * i < N;
        if (CONV) {
            int mm = a_row_ok[i] ? m : 0;
            pix_w[i] = mm % a.W;
            pix_h[i] = (mm / a.W) % a.H;
            pix_b[i] = mm / (a.W * a.H);
        }
    }

    const int KT = (K + BK - 1) / BK;
    auto load_stage = [&](int kt, int slot) {
        const uint32_t sA = sbase + slot * 2 * TILE_BYTES, sB = sA + TILE_BYTES;
        const int k = kt * BK + c * 16;
        const bool k_ok = k < K;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int r = r0 + 64 * i;
            // activation chunk
            const int8_t* src = X;
            bool ok = a_row_ok[i] && k_ok;
            if (CONV) {
                int tap = k / a.Cin, cin = k - tap * a.Cin;
                int ih = pix_h[i] + tap / 3 - 1, iw = pix_w[i] + tap % 3 - 1;
                ok = ok && ih >= 0 && ih < a.H && iw >= 0 && iw < a.W;
                if (ok) src = X + ((int64_t(pix_b[i]) * a.H + ih) * a.W + iw) * a.Cin + cin;
            } else if (ok) {
                src = X + int64_t(m0 + r) * K + k;
            }
            cp_async16(sA + swz(r, c), src, ok);
            // weight chunk
            bool okw = b_row_ok[i] && k_ok;
            cp_async16(sB + swz(r, c), okw ? Wt + int64_t(n0 + r) * K + k : Wt, okw);
        }
    };

    int acc[4][4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[i][j][q] = 0;

#pragma unroll
    for (int s = 0; s < STAGES - 1; ++s) {
        if (s < KT) load_stage(s, s);
        cp_commit();
    }

    for (int kt = 0; kt < KT; ++kt) {
        cp_wait<STAGES - 2>();
        __syncthreads();
        {
            int nk = kt + STAGES - 1;
            if (nk < KT) load_stage(nk, nk % STAGES);
            cp_commit();
        }
        const int slot = kt % STAGES;
        const uint32_t sA = sbase + slot * 2 * TILE_BYTES, sB = sA + TILE_BYTES;
#pragma unroll
        for (int ks = 0; ks < 2; ++ks) {
            uint32_t af[4][4], bf[4][2];
#pragma unroll
            for (int mi = 0; mi < 4; ++mi) {
                int r = wm * 64 + mi * 16 + (lane & 15);
                ldmatrix_x4(sA + swz(r, ks * 2 + (lane >> 4)), af[mi][0], af[mi][1], af[mi][2], af[mi][3]);
            }
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                int r = wn * 32 + j * 16 + (lane & 7) + ((lane >> 4) << 3);
                uint32_t t0, t1, t2, t3;
                ldmatrix_x4(sB + swz(r, ks * 2 + ((lane >> 3) & 1)), t0, t1, t2, t3);
                bf[2 * j][0] = t0 & wmask[2 * j];
                bf[2 * j][1] = t1 & wmask[2 * j];
                bf[2 * j + 1][0] = t2 & wmask[2 * j + 1];
                bf[2 * j + 1][1] = t3 & wmask[2 * j + 1];
            }
#pragma unroll
            for (int mi = 0; mi < 4; ++mi)
#pragma unroll
                for (int ni = 0; ni < 4; ++ni) mma_s8(acc[mi][ni], af[mi], bf[ni][0], bf[ni][1]);
        }
    }
    cp_wait<0>();

    // ------------------------------------------------------------ epilogue
    const int g = lane >> 2, t4 = lane & 3;
    const int32_t* ts_b = CONV ? a.ts + int64_t(b - kBMin) * N * 9 : nullptr;
#pragma unroll
    for (int ni = 0; ni < 4; ++ni) {
        const int n = n0 + wn * 32 + ni * 8 + 2 * t4;
        if (n >= N) continue;
        const float cw0 = a.cw[n], cw1 = a.cw[n + 1];
        const float bi0 = a.bias[n], bi1 = a.bias[n + 1];
        // row sums at the channel's b (n and n + 1 belong to one member: group_n % 8 == 0)
        const int32_t* rs_b = a.rs + int64_t(channel_bits(a, gbits, n) - kBMin) * N;
        const int rsl0 = CONV ? 0 : rs_b[n], rsl1 = CONV ? 0 : rs_b[n + 1];
        // asymmetric weights: zero offsets per channel, activation sums per token
        constexpr bool zp = ZP;
        const float zw0 = zp ? a.zcw[n] : 0.f, zw1 = zp ? a.zcw[n + 1] : 0.f;
#pragma unroll
        for (int mi = 0; mi < 4; ++mi)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const int m = m0 + wm * 64 + mi * 16 + g + 8 * hh;
                if (m >= M) continue;
                const float al = a.per_tensor ? a.alpha[0] : a.alpha[m];
                const float z = a.per_tensor ? a.zc[0] : a.zc[m];
                int rs0 = rsl0, rs1 = rsl1;
                if (CONV) {
                    int pw = m % a.W, ph = (m / a.W) % a.H;
                    rs0 = conv_row_sum(ts_b + int64_t(n) * 9, ph, pw, a.H, a.W);
                    rs1 = conv_row_sum(ts_b + int64_t(n + 1) * 9, ph, pw, a.H, a.W);
                }
                const int v0 = acc[mi][ni][2 * hh], v1 = acc[mi][ni][2 * hh + 1];
                uint32_t y0, y1;
                if constexpr (zp) {
                    const float t = CONV ? conv_token_zero_sum(a.code_sums, m, a.H, a.W, a.Cin, z)
                                         : token_zero_sum(a.code_sums[m], a.K, z);
                    y0 = bf16_bits(epilogue_value_zp(v0, al, z, t, rs0, cw0, zw0, bi0));
                    y1 = bf16_bits(epilogue_value_zp(v1, al, z, t, rs1, cw1, zw1, bi1));
                } else {
                    y0 = bf16_bits(epilogue_value(v0, al, z, rs0, cw0, bi0));
                    y1 = bf16_bits(epilogue_value(v1, al, z, rs1, cw1, bi1));
                }
                *reinterpret_cast<uint32_t*>(a.y + int64_t(m) * N + n) = y0 | (y1 << 16);
                if (a.acc) *reinterpret_cast<int2*>(a.acc + int64_t(m) * N + n) = make_int2(v0, v1);
            }
    }
}

}  // namespace

cudaError_t launch_gemm_s8(const GemmArgs& a, int /*num_sms*/, cudaStream_t st) {
    if (a.M == 0 || a.N == 0) return cudaSuccess;
    dim3 grid((a.N + BN - 1) / BN, (a.M + BM - 1) / BM);
    if (grid.y > 65535) return cudaErrorInvalidConfiguration;
    cudaError_t e;
    auto kernel = a.Cin ? (a.code_sums ? gemm_s8_kernel<true, true> : gemm_s8_kernel<true, false>)
                        : (a.code_sums ? gemm_s8_kernel<false, true> : gemm_s8_kernel<false, false>);
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    kernel<<<grid, THREADS, SMEM_BYTES, st>>>(a);
    return cudaGetLastError();
}

}  // namespace tasq
