// Masked contraction on the 5th-generation tensor cores (tcgen05, sm_103a).
//
// sm_103a has no int8 tcgen05 MMA, so the integer contraction runs on the
// fp16 MMA exactly: every int8 code is an exact fp16, every product of two
// codes (|p| <= 2^14) is exact, and an fp32 sum of integer products is exact
// while every partial sum stays within 2^24.  The packed weights carry, for
// each operating precision b, a certificate: the number of 64-wide K blocks
// over which 128 * sum_k |mask_b(w)| <= 2^24 holds for every channel.  The
// accumulator in tensor memory is restarted after each such chunk and
// drained into an int32 running sum (also kept in tensor memory), so the
// final int32 accumulator equals the exact integer result.
//
// Operand roles (D = A * B^T with the output channels on the MMA's M side):
//   A: the weight tile, 128 channels x 64 K.  TMA brings the stored int8 codes
//      into shared memory; a converter warpgroup applies the operating-
//      precision mask (Eq. hw_rightshift: clear the low 8-b planes, one AND
//      per four codes), widens to fp16 and writes the tile straight into
//      tensor memory, where the MMA reads it.
//   B: the activation codes, held as fp16 integers in HBM, brought by TMA
//      into 128-byte-swizzled shared memory (a 2-D tile for a linear layer; a
//      4-D NHWC box shifted by the 3x3 tap for a convolution, whose padding
//      TMA fills with code 0).
//   D: fp32 accumulators in tensor memory, double-buffered so the epilogue
//      of one chunk overlaps the MMAs of the next.
//
// Warp roles (320 threads): warp 0 issues TMA; warp 1 allocates tensor
// memory and issues the MMAs (one thread); warps 2..5 convert weights; warps
// 6..9 drain accumulators and run the fused dequantization epilogue.  The
// grid is persistent: one CTA per SM walks the output tiles.  Every wait is
// bounded by the context's time limit; a wait that gives up records
// TASQ_ERR_DEVICE_TIMEOUT, the CTA drains its copies in flight, frees its
// tensor memory and returns.
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {
namespace {

constexpr int BCH = 128;         // output channels per tile (MMA M)
constexpr int BTOK = 128;        // tokens / output pixels per tile (MMA N)
constexpr int BK = 64;           // K per pipeline stage
constexpr int STAGES = 6;        // shared-memory stages
constexpr int ASLOTS = 4;        // tensor-memory slots of converted weights
constexpr int THREADS = 320;
constexpr int X_STAGE = BTOK * BK * 2;  // 16 KB fp16 codes
constexpr int W_STAGE = BCH * BK;       // 8 KB int8 codes
// tensor memory columns
constexpr uint32_t ACC_COL = 0;                         // 2 x BTOK fp32 accumulators
constexpr uint32_t A_COL = 2 * BTOK;                    // ASLOTS x 32 (64 fp16 per row)
constexpr uint32_t SUM_COL = A_COL + ASLOTS * (BK / 2);  // BTOK int32 running sums
constexpr uint32_t TMEM_COLS = 512;
static_assert(SUM_COL + BTOK <= TMEM_COLS, "tensor memory budget");
constexpr uint32_t IDESC = ptx::idesc_f16_f32(BCH, BTOK);

struct Smem {
    uint8_t x[STAGES][X_STAGE];  // 1024-aligned (128B swizzle atoms)
    uint8_t w[STAGES][W_STAGE];
    uint64_t full[STAGES], empty[STAGES];
    uint64_t afull[ASLOTS], aempty[ASLOTS];
    uint64_t accfull[2], accempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};
constexpr int SMEM_BYTES = sizeof(Smem) + 1024;

struct TcParams {
    GemmArgs a;
    int conv;
    int tiles_ch, tiles_tok;
    int bw, bh, tiles_w, tiles_h;  // conv: token tile = bh x bw pixel rectangle
};

struct Waiter {
    Smem* s;
    const GemmArgs* a;
    // Bounded wait on phase `parity` of an mbarrier; false after a timeout or
    // when another role has aborted the CTA.
    __device__ __forceinline__ bool wait(uint64_t* bar, uint32_t parity, bool ignore_abort = false) const {
        const uint32_t addr = ptx::smem_u32(bar);
        if (ptx::mbar_try_wait(addr, parity)) return true;
        const uint64_t t0 = ptx::globaltimer();
        for (uint32_t it = 1;; ++it) {
            if (ptx::mbar_try_wait(addr, parity)) return true;
            if ((it & 63) == 0) {
                if (!ignore_abort && *(volatile int*)&s->abort) return false;
                if (ptx::globaltimer() - t0 > a->timeout_ns) {
                    set_status(a->status, TASQ_ERR_DEVICE_TIMEOUT);
                    *(volatile int*)&s->abort = 1;
                    return false;
                }
            }
        }
    }
};

// fp16 bit patterns of four masked codes: (w & m) ^ 0x80 per byte gives the
// unsigned code u = v + 128; 0x64uu is the fp16 value 1024 + u; subtracting
// 1152 leaves v exactly.
__device__ __forceinline__ void widen4(uint32_t w, uint32_t m, uint32_t& lo, uint32_t& hi) {
    const uint32_t u = (w & m) ^ 0x80808080u;
    lo = __byte_perm(u, 0x64646464u, 0x5140);
    hi = __byte_perm(u, 0x64646464u, 0x7362);
    const __half2 bias = __halves2half2(__ushort_as_half(0x6480), __ushort_as_half(0x6480));  // 1152
    __half2 l = __hsub2(*reinterpret_cast<__half2*>(&lo), bias);
    __half2 h = __hsub2(*reinterpret_cast<__half2*>(&hi), bias);
    lo = *reinterpret_cast<uint32_t*>(&l);
    hi = *reinterpret_cast<uint32_t*>(&h);
}

__global__ void __launch_bounds__(THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ TcParams p, const __grid_constant__ CUtensorMap tm_x,
                   const __grid_constant__ CUtensorMap tm_w) {
    extern __shared__ uint8_t smem_raw[];
    Smem* s = reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const GemmArgs& a = p.a;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Waiter wt{s, &a};

    const int b = resolve_bits(a);
    if (b == 0) return;  // uniform across the CTA: nothing allocated yet
    const int KT = (a.K + BK - 1) / BK;
    int chunk = a.hdr->chunk_kb[b];
    chunk = chunk < 1 ? 1 : (chunk > KT ? KT : chunk);
    const int nchunks = (KT + chunk - 1) / chunk;
    const int tiles = p.tiles_ch * p.tiles_tok;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->full[i]), 1);
            ptx::mbar_init(ptx::smem_u32(&s->empty[i]), 4 + 1);  // 4 converter warps + MMA commit
        }
        for (int i = 0; i < ASLOTS; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->afull[i]), 4);
            ptx::mbar_init(ptx::smem_u32(&s->aempty[i]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->accfull[i]), 1);
            ptx::mbar_init(ptx::smem_u32(&s->accempty[i]), 4);
        }
        ptx::mbar_init(ptx::smem_u32(&s->drain), 1);
        s->abort = 0;
        ptx::fence_mbar_init();
        ptx::prefetch_tmap(&tm_x);
        ptx::prefetch_tmap(&tm_w);
    }
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&s->tmem_base), TMEM_COLS);
        ptx::tmem_relinquish();
        ptx::tc_fence_before();
    }
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = s->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
                const int ch0 = (t % p.tiles_ch) * BCH;
                const int tt = t / p.tiles_ch;
                int tok0 = 0, img = 0, h0 = 0, w0 = 0;
                if (p.conv) {
                    const int per_img = p.tiles_h * p.tiles_w;
                    img = tt / per_img;
                    h0 = ((tt % per_img) / p.tiles_w) * p.bh;
                    w0 = (tt % p.tiles_w) * p.bw;
                } else {
                    tok0 = tt * BTOK;
                }
                for (int kb = 0; kb < KT; ++kb, ++it) {
                    const int st = it % STAGES;
                    if (!wt.wait(&s->empty[st], ((it / STAGES) & 1) ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fb = ptx::smem_u32(&s->full[st]);
                    ptx::mbar_arrive_expect_tx(fb, X_STAGE + W_STAGE);
                    const int k0 = kb * BK;
                    if (p.conv) {
                        const int tap = k0 / a.Cin, c0 = k0 - tap * a.Cin;
                        ptx::tma_load_4d(ptx::smem_u32(s->x[st]), &tm_x, fb, c0, w0 + tap % 3 - 1, h0 + tap / 3 - 1,
                                         img);
                    } else {
                        ptx::tma_load_2d(ptx::smem_u32(s->x[st]), &tm_x, fb, k0, tok0);
                    }
                    ptx::tma_load_2d(ptx::smem_u32(s->w[st]), &tm_w, fb, k0, ch0);
                }
            }
            // copies still in flight must land before the CTA may exit
            const int first = it > STAGES ? it - STAGES : 0;
            for (int j = first; j < it; ++j) wt.wait(&s->full[j % STAGES], (j / STAGES) & 1, true);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int it = 0, cc = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
                for (int c = 0; c < nchunks && ok; ++c, ++cc) {
                    const int buf = cc & 1;
                    if (!wt.wait(&s->accempty[buf], ((cc >> 1) & 1) ^ 1)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t d = tmem + ACC_COL + buf * BTOK;
                    const int kb_end = min(KT, (c + 1) * chunk);
                    for (int kb = c * chunk; kb < kb_end; ++kb, ++it) {
                        const int st = it % STAGES, sl = it % ASLOTS;
                        if (!wt.wait(&s->full[st], (it / STAGES) & 1) ||
                            !wt.wait(&s->afull[sl], (it / ASLOTS) & 1)) {
                            ok = false;
                            break;
                        }
                        ptx::tc_fence_after();
                        const uint64_t bdesc = ptx::sw128_kmajor_desc(ptx::smem_u32(s->x[st]));
#pragma unroll
                        for (int k = 0; k < BK / 16; ++k)
                            ptx::mma_f16_ts(d, tmem + A_COL + sl * (BK / 2) + k * 8, bdesc + uint64_t((k * 32) >> 4),
                                            IDESC, (kb > c * chunk || k > 0) ? 1u : 0u);
                        ptx::mma_commit(ptx::smem_u32(&s->empty[st]));
                        ptx::mma_commit(ptx::smem_u32(&s->aempty[sl]));
                    }
                    if (ok) ptx::mma_commit(ptx::smem_u32(&s->accfull[buf]));
                }
            }
            // every MMA issued must finish before tensor memory is released
            ptx::mma_commit(ptx::smem_u32(&s->drain));
            wt.wait(&s->drain, 0, true);
        }
    } else if (warp < 6) {
        // ------------------------------------------- weight mask + convert
        const int q = warp & 3;             // tensor-memory lane quadrant
        const int r = q * 32 + lane;        // channel row within the tile
        const uint32_t m = mask_word(b);
        const uint32_t lane_base = tmem + (uint32_t(q * 32) << 16);
        int it = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
            for (int kb = 0; kb < KT; ++kb, ++it) {
                const int st = it % STAGES, sl = it % ASLOTS;
                if (!wt.wait(&s->full[st], (it / STAGES) & 1)) {
                    ok = false;
                    break;
                }
                // 64 codes of row r; 16-byte chunk c sits at c ^ ((r >> 1) & 3) (64-byte swizzle)
                uint4 v[4];
                const uint8_t* row = s->w[st] + r * BK;
#pragma unroll
                for (int c = 0; c < 4; ++c) v[c] = *reinterpret_cast<const uint4*>(row + ((c ^ ((r >> 1) & 3)) << 4));
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->empty[st]));
                if (!wt.wait(&s->aempty[sl], ((it / ASLOTS) & 1) ^ 1)) {
                    ok = false;
                    break;
                }
                uint32_t f[32];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    widen4(v[c].x, m, f[8 * c + 0], f[8 * c + 1]);
                    widen4(v[c].y, m, f[8 * c + 2], f[8 * c + 3]);
                    widen4(v[c].z, m, f[8 * c + 4], f[8 * c + 5]);
                    widen4(v[c].w, m, f[8 * c + 6], f[8 * c + 7]);
                }
                ptx::tmem_st32(lane_base + A_COL + sl * (BK / 2), f);
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->afull[sl]));
            }
        }
    } else {
        // ------------------------------------- accumulator drain + epilogue
        const int q = warp & 3;
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + (uint32_t(q * 32) << 16);
        const int32_t* rs_b = a.rs + int64_t(b - kBMin) * a.N;
        const int32_t* ts_b = p.conv ? a.ts + int64_t(b - kBMin) * a.N * 9 : nullptr;
        int cc = 0;
        bool ok = true;
        for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
            const int ch0 = (t % p.tiles_ch) * BCH;
            const int tt = t / p.tiles_ch;
            const int n = ch0 + r;
            const bool n_ok = n < a.N;
            float cw = 0.f, bias = 0.f;
            int rs = 0;
            int ts[9];
#pragma unroll
            for (int i = 0; i < 9; ++i) ts[i] = 0;
            if (n_ok) {
                cw = a.cw[n];
                bias = a.bias[n];
                if (p.conv) {
#pragma unroll
                    for (int i = 0; i < 9; ++i) ts[i] = ts_b[int64_t(n) * 9 + i];
                } else {
                    rs = rs_b[n];
                }
            }
            int img = 0, h0 = 0, w0 = 0, tok0 = 0;
            if (p.conv) {
                const int per_img = p.tiles_h * p.tiles_w;
                img = tt / per_img;
                h0 = ((tt % per_img) / p.tiles_w) * p.bh;
                w0 = (tt % p.tiles_w) * p.bw;
            } else {
                tok0 = tt * BTOK;
            }
            for (int c = 0; c < nchunks; ++c, ++cc) {
                const int buf = cc & 1;
                if (!wt.wait(&s->accfull[buf], (cc >> 1) & 1)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const bool last = c == nchunks - 1;
#pragma unroll 1
                for (int g = 0; g < BTOK / 32; ++g) {
                    uint32_t v[32];
                    ptx::tmem_ld32(lane_base + ACC_COL + buf * BTOK + g * 32, v);
                    ptx::tmem_wait_ld();
                    int iv[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) iv[j] = __float2int_rn(__uint_as_float(v[j]));
                    if (c > 0) {
                        uint32_t sv[32];
                        ptx::tmem_ld32(lane_base + SUM_COL + g * 32, sv);
                        ptx::tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) iv[j] += int(sv[j]);
                    }
                    if (!last) {
                        uint32_t sv[32];
#pragma unroll
                        for (int j = 0; j < 32; ++j) sv[j] = uint32_t(iv[j]);
                        ptx::tmem_st32(lane_base + SUM_COL + g * 32, sv);
                        ptx::tmem_wait_st();
                        continue;
                    }
                    // final: fused dequantization epilogue for 32 tokens of channel n
                    int tok_lane;  // token (or output pixel) index held by this lane, -1 if none
                    if (p.conv) {
                        const int j = g * 32 + lane;
                        const int h = h0 + j / p.bw, w = w0 + j % p.bw;
                        tok_lane = (h < a.H && w < a.W) ? (img * a.H + h) * a.W + w : -1;
                    } else {
                        const int m = tok0 + g * 32 + lane;
                        tok_lane = m < a.M ? m : -1;
                    }
                    float al_lane = 0.f, zc_lane = 0.f;
                    if (tok_lane >= 0) {
                        al_lane = a.per_tensor ? a.alpha[0] : a.alpha[tok_lane];
                        zc_lane = a.per_tensor ? a.zc[0] : a.zc[tok_lane];
                    }
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int m = __shfl_sync(0xffffffffu, tok_lane, j);
                        const float al = __shfl_sync(0xffffffffu, al_lane, j);
                        const float zc = __shfl_sync(0xffffffffu, zc_lane, j);
                        if (m < 0 || !n_ok) continue;
                        int rsum = rs;
                        if (p.conv) {
                            const int jj = g * 32 + j;
                            rsum = conv_row_sum(ts, h0 + jj / p.bw, w0 + jj % p.bw, a.H, a.W);
                        }
                        const float y = epilogue_value(iv[j], al, zc, rsum, cw, bias);
                        a.y[int64_t(m) * a.N + n] = bf16_bits(y);
                        if (a.acc) a.acc[int64_t(m) * a.N + n] = iv[j];
                    }
                }
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->accempty[buf]));
            }
        }
    }

    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, TMEM_COLS);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void* ptr = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

}  // namespace

cudaError_t launch_gemm_tc(const GemmArgs& a, int num_sms, cudaStream_t st, const char** why) {
    *why = nullptr;
    if (a.M == 0 || a.N == 0) return cudaSuccess;
    auto encode = get_encode();
    if (!encode) {
        *why = "cuTensorMapEncodeTiled is unavailable";
        return cudaSuccess;
    }
    TcParams p{};
    p.a = a;
    p.conv = a.Cin != 0;
    p.tiles_ch = (a.N + BCH - 1) / BCH;
    CUtensorMap tm_x, tm_w;
    CUresult r;
    if (p.conv) {
        if (a.Cin % BK) {
            *why = "convolution needs Cin % 64 == 0";
            return cudaSuccess;
        }
        int bw = 1;
        while (bw < a.W && bw < BTOK) bw <<= 1;
        p.bw = bw;
        p.bh = BTOK / bw;
        p.tiles_w = (a.W + p.bw - 1) / p.bw;
        p.tiles_h = (a.H + p.bh - 1) / p.bh;
        const int64_t tok_tiles = int64_t(a.B) * p.tiles_h * p.tiles_w;
        if (tok_tiles * p.tiles_ch > 0x7FFFFFFF) {
            *why = "too many tiles";
            return cudaSuccess;
        }
        p.tiles_tok = int(tok_tiles);
        cuuint64_t dims[4] = {cuuint64_t(a.Cin), cuuint64_t(a.W), cuuint64_t(a.H), cuuint64_t(a.B)};
        cuuint64_t strides[3] = {cuuint64_t(a.Cin) * 2, cuuint64_t(a.W) * a.Cin * 2, cuuint64_t(a.H) * a.W * a.Cin * 2};
        cuuint32_t box[4] = {BK, cuuint32_t(p.bw), cuuint32_t(p.bh), 1};
        cuuint32_t es[4] = {1, 1, 1, 1};
        r = encode(&tm_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(a.x), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else {
        p.tiles_tok = (a.M + BTOK - 1) / BTOK;
        cuuint64_t dims[2] = {cuuint64_t(a.K), cuuint64_t(a.M)};
        cuuint64_t strides[1] = {cuuint64_t(a.K) * 2};
        cuuint32_t box[2] = {BK, BTOK};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(a.x), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    if (r != CUDA_SUCCESS) {
        *why = "activation tensor map rejected";
        return cudaSuccess;
    }
    {
        cuuint64_t dims[2] = {cuuint64_t(a.K), cuuint64_t(a.N)};
        cuuint64_t strides[1] = {cuuint64_t(a.K)};
        cuuint32_t box[2] = {BK, BCH};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_w, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t*>(a.w), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "weight tensor map rejected";
            return cudaSuccess;
        }
    }
    const int64_t tiles = int64_t(p.tiles_ch) * p.tiles_tok;
    const int grid = int(tiles < num_sms ? tiles : num_sms);
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess) return e;
    gemm_tc_kernel<<<grid, THREADS, SMEM_BYTES, st>>>(p, tm_x, tm_w);
    return cudaGetLastError();
}

}  // namespace tasq
