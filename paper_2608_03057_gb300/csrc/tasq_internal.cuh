// Internal declarations shared by the translation units of libtasq.
// Nothing here is part of the C ABI (include/tasq.h is).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tasq.h"

namespace tasq {

// ---------------------------------------------------------------------------
// Packed layer layout (one contiguous, caller-allocated buffer per layer).
// ---------------------------------------------------------------------------
constexpr uint32_t kPackedMagic = 0x51534154u;  // "TASQ"
constexpr int kBMin = 2, kBMax = 8, kNumB = kBMax - kBMin + 1;
constexpr int kCertKBlock = 64;   // K block of the exactness certificate (TC route BK)
constexpr int64_t kCertLimit = int64_t(1) << 17;  // 2^24 / 128: sum |w| bound per chunk
// Bit table in device memory: a 16-byte header (int32 L, int32 S) then the bits
// [L][S].  The context allocates room for kTableCapacity bits when it is created.
constexpr int kTableHeader = 16;
constexpr size_t kTableCapacity = 65536;
// Most layers one grouped contraction call may hold: with the member list in
// the call's arguments (kMaxGroups), or in device memory (kMaxMembers; the
// tensor-core route resolves every member's b into shared memory).
constexpr int kMaxGroups = 4;
constexpr int kMaxMembers = 256;
// Largest operating precision whose masked weight codes are exact in e5m2: mask_b(v)
// is t * 2^(8-b) with |t| <= 2^(b-1), at most three significant bits for b <= 4.
constexpr int kBMaxF8 = 4;
// Largest activation code magnitude of TASQ_CODES_F16_E5M2 (n <= 4): the exact
// chunk of the tensor-core route is 128 / kF8CodeMax times the one certified for
// 8-bit codes.
constexpr int kF8CodeMax = 8;

struct PackedHeader {
    uint32_t magic;
    int32_t kind, N, K, Cin;
    int32_t chunk_kb[kBMax + 1];  // TC route: K blocks per exact fp32 chunk, indexed by b
    int64_t off_w, off_cw, off_bias, off_rs, off_ts, total;
    int64_t off_zcw;  // fp32 [N] weight zero offsets zcw = 128 - z (zeros unless has_zp)
    int32_t has_zp;   // packed with zero offsets: the four-term epilogue applies
};
static_assert(sizeof(PackedHeader) <= 256, "header must fit in 256 bytes");

__host__ __device__ inline int64_t align_up(int64_t v, int64_t a) { return (v + a - 1) / a * a; }

__host__ __device__ inline PackedHeader packed_layout(int kind, int N, int K) {
    PackedHeader h{};
    h.magic = kPackedMagic;
    h.kind = kind;
    h.N = N;
    h.K = K;
    h.Cin = kind == TASQ_CONV3X3 ? K / 9 : 0;
    h.off_w = 1024;
    h.off_cw = align_up(h.off_w + int64_t(N) * K, 256);
    h.off_bias = align_up(h.off_cw + 4 * int64_t(N), 256);
    h.off_rs = align_up(h.off_bias + 4 * int64_t(N), 256);          // int32 [kNumB][N]
    h.off_ts = align_up(h.off_rs + 4 * int64_t(kNumB) * N, 256);     // int32 [kNumB][N][9] (conv)
    h.off_zcw = align_up(h.off_ts + (kind == TASQ_CONV3X3 ? 4 * int64_t(kNumB) * N * 9 : 0), 256);  // fp32 [N]
    h.total = align_up(h.off_zcw + 4 * int64_t(N), 256);
    return h;
}

// Signed stored code with the low 8-b planes of the unsigned code cleared.
// (v + 128) has the same low planes as v, and 128 is a multiple of 2^(8-b).
__host__ __device__ inline int mask_code(int v, int b) { return v & ~((1 << (8 - b)) - 1); }
// Byte mask replicated over a 32-bit word of four codes.
__host__ __device__ inline uint32_t mask_word(int b) { return 0x01010101u * (0xFFu & (0xFFu << (8 - b))); }

// ---------------------------------------------------------------------------
// Device status word: first error wins.
// ---------------------------------------------------------------------------
__device__ inline void set_status(int* status, int code) {
    if (status) atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// Arguments of the masked contraction kernels (both routes, linear and conv).
// ---------------------------------------------------------------------------
struct GemmArgs {
    const void* x;            // codes: [M][K] (linear) or NHWC (conv)
    const void* x8;           // the same codes as e5m2 bytes [M][K] (linear layers), or NULL
    int chunk_scale;          // exact-chunk multiplier: 128 / the largest code magnitude (1 for 8-bit codes)
    const float* alpha;       // [M] or [1]
    const float* zc;
    const int8_t* w;          // stored codes [N][K]
    const float* cw;          // [N]
    const float* bias;        // [N]
    const int32_t* rs;        // [kNumB][N]
    const int32_t* ts;        // conv: [kNumB][N][9]
    const PackedHeader* hdr;  // device copy of the header
    const uint8_t* table;     // bit table: int32 L, S at offset 0, bits [L][S] at kTableHeader
    const int32_t* d_stage;   // used when stage < 0
    int layer, stage;
    // Grouped call: `groups` layers that read the same activations, stored as one
    // packed buffer of their weights concatenated along N; member g owns output
    // channels [g * group_n, (g + 1) * group_n) and runs at its own b.
    int groups;               // 1 for a single layer
    int group_n;              // N / groups
    int layers[kMaxGroups];   // member layers (layers[0] == layer) when d_layers is NULL
    const int32_t* d_layers;  // member layers in device memory (up to kMaxMembers), or NULL
    int M, N, K;
    int B, H, W, Cin;         // conv geometry (Cin == 0 for a linear layer)
    int per_tensor;
    uint16_t* y;              // bf16 bits
    int32_t* acc;             // optional int32 accumulators
    int32_t* part;            // TC route: per-CTA int32 running sums of multi-chunk tiles
    int32_t* split_buf;       // TC route: int32 partial sums of split-K slices
    int64_t split_cap;        // elements of split_buf
    int* status;
    unsigned long long timeout_ns;
    // Asymmetric weights (App. A.1.1 on the true per-channel range, Eq.
    // weight_dequant with a real zero point): w_hat = c_w * (mask_b(s_w) + zcw).
    // With code_sums set the epilogue adds zcw[n] * t[m], t = sum_k (s_x + zc).
    const float* zcw;          // [N] from the packed buffer (zeros for a symmetric pack)
    const int32_t* code_sums;  // [M] sum_k s_x[m][k] (conv: per input pixel), or NULL (two-term epilogue)
    // 16-bit low-rank branch of an SVD-split layer (linear layers): one more K block
    // after the last one of each tile adds sum_j u'[m][j] * fp16(l1[n][j] / c_w[n]) to
    // the accumulator, u' = fp16((x . l2^T)[m][j] / alpha[m]) from tasq_lowrank_down.
    const uint16_t* lr_u;      // fp16 [M][kLowRankCols] u' (columns >= lr_rank zero), or NULL
    const uint16_t* lr_l1;     // bf16 [N][lr_rank]
    int lr_rank;               // 0, 16 or 32
};

// Resolves the operating precision of every member layer of this launch on
// the device, packed four bits per member (member g in bits 4g..4g+3); returns
// 0 (and records an error) when the stage or a table entry is out of range or
// the header mismatches.  A single layer is the group of one.
__device__ inline uint32_t resolve_group_bits(const GemmArgs& a) {
    // the header fields and the stage do not depend on one another: load them together
    const uint32_t magic = a.hdr->magic;
    const int hdr_n = a.hdr->N, hdr_k = a.hdr->K, hdr_zp = a.hdr->has_zp;
    const int stage = a.stage >= 0 ? a.stage : (a.d_stage ? *a.d_stage : -1);
    // the table's dimensions come from the device copy, so a graph captured before a
    // later tasq_set_schedule reads that schedule's bits (or records the mismatch)
    const int2 dims = *reinterpret_cast<const int2*>(a.table);
    bool ok = stage >= 0 && stage < dims.y && magic == kPackedMagic && hdr_n == a.N && hdr_k == a.K &&
              !(hdr_zp && !a.code_sums);  // a buffer packed with zero offsets needs the code sums
    uint32_t packed = 0;
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g) {
        if (g < a.groups) {
            const int layer = a.layers[g];
            const bool in = ok && layer < dims.x;
            const int b = in ? a.table[kTableHeader + layer * dims.y + stage] : 0;
            ok = in && b >= kBMin && b <= kBMax;
            packed |= uint32_t(b & 15) << (4 * g);
        }
    }
    if (!ok) {
        set_status(a.status, TASQ_ERR_DEVICE);
        return 0;
    }
    return packed;
}

// b of output channel n from the packed member bits.
__device__ __forceinline__ int channel_bits(const GemmArgs& a, uint32_t packed_bits, int n) {
    const int g = a.groups > 1 ? min(n / a.group_n, a.groups - 1) : 0;
    return int((packed_bits >> (4 * g)) & 15u);
}

// b of member g of a call whose member list is in device memory (a.d_layers), or 0
// when the stage, the layer index or its table entry is out of range or the header
// mismatches (the caller records the error).
__device__ inline int resolve_member_bits(const GemmArgs& a, int g) {
    const uint32_t magic = a.hdr->magic;
    const int hdr_n = a.hdr->N, hdr_k = a.hdr->K, hdr_zp = a.hdr->has_zp;
    const int stage = a.stage >= 0 ? a.stage : (a.d_stage ? *a.d_stage : -1);
    const int layer = a.d_layers[g];
    const int2 dims = *reinterpret_cast<const int2*>(a.table);
    const bool ok = stage >= 0 && stage < dims.y && magic == kPackedMagic && hdr_n == a.N && hdr_k == a.K &&
                    !(hdr_zp && !a.code_sums) && layer >= 0 && layer < dims.x;
    const int b = ok ? a.table[kTableHeader + layer * dims.y + stage] : 0;
    return b >= kBMin && b <= kBMax ? b : 0;
}

// x / a rounded to nearest even, from ra = RN(1/a): the quotient estimate
// q = RN(x * ra) lies within one ulp of x / a, and one correction by the exact
// FMA remainder r = x - q * a, q <- RN(q + r * ra), gives the correctly rounded
// quotient for normal operands (Markstein's theorem: ra within half an ulp of
// 1/a and q within one ulp of x/a suffice).  Checked against IEEE division by
// tasq_selftest_quotients over every finite normal bf16 dividend.
__device__ __forceinline__ float div_rn_by(float x, float a, float ra) {
    const float q = __fmul_rn(x, ra);
    const float r = __fmaf_rn(-q, a, x);
    return __fmaf_rn(r, ra, q);
}

// Round half to even of |u| <= 2^22, returned as an int: adding 1.5 * 2^23
// leaves the rounded integer in the low mantissa bits.
__device__ __forceinline__ int rint_small(float u) {
    return int(__float_as_uint(__fadd_rn(u, 12582912.0f)) - 0x4B400000u);
}

// Fused dequantization epilogue in fp32, each operation rounded once to
// nearest even: u = fma(zc, float(rs), float(acc)), s = alpha * cw,
// y = fma(u, s, bias); this equals alpha * cw * (acc + zc * rs) + bias.
__device__ inline float epilogue_value(int acc, float alpha, float zc, int rs, float cw, float bias) {
    const float u = __fmaf_rn(zc, __int2float_rn(rs), __int2float_rn(acc));
    return __fmaf_rn(u, __fmul_rn(alpha, cw), bias);
}

// Asymmetric weights: t = RN(float(sx) + RN(float(K) * zc)), the token's
// activation sum sum_k (s_x + zc) (exact integer sx, |sx| <= 128 K < 2^24),
// and the epilogue with the weight zero-offset term, each step rounded once:
// u1 = fma(zc, float(rs), float(acc)), u2 = fma(zcw, t, u1), y = fma(u2, alpha*cw, bias),
// i.e. y = alpha * cw * (acc + zc * rs + zcw * (sx + K * zc)) + bias.
__device__ __forceinline__ float token_zero_sum(int sx, int K, float zc) {
    return __fadd_rn(__int2float_rn(sx), __fmul_rn(__int2float_rn(K), zc));
}
__device__ inline float epilogue_value_zp(int acc, float alpha, float zc, float t, int rs, float cw, float zcw,
                                          float bias) {
    const float u1 = __fmaf_rn(zc, __int2float_rn(rs), __int2float_rn(acc));
    const float u2 = __fmaf_rn(zcw, t, u1);
    return __fmaf_rn(u2, __fmul_rn(alpha, cw), bias);
}

// fp32 -> bf16 bits, round to nearest even (finite inputs).
__device__ inline uint16_t bf16_bits(float f) {
    uint32_t u = __float_as_uint(f);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

// 3x3 conv with asymmetric weights: for output pixel p, t = RN(float(sxw) +
// RN(float(Kv) * zc)) with sxw the sum of the per-pixel code sums over its
// in-bounds taps and Kv = Cin x (in-bounds taps) (padding is zero in the real
// domain, so a padded tap carries no zero-point term).
__device__ inline float conv_token_zero_sum(const int32_t* code_sums, int p, int H, int W, int Cin, float zc) {
    const int w = p % W, h = (p / W) % H;
    const int base = p - (h * W + w);  // first pixel of the image
    int sum = 0, taps = 0;
#pragma unroll
    for (int dh = -1; dh <= 1; ++dh) {
        const int ih = h + dh;
        if (ih < 0 || ih >= H) continue;
#pragma unroll
        for (int dw = -1; dw <= 1; ++dw) {
            const int iw = w + dw;
            if (iw < 0 || iw >= W) continue;
            sum += code_sums[base + ih * W + iw];
            ++taps;
        }
    }
    return __fadd_rn(__int2float_rn(sum), __fmul_rn(__int2float_rn(taps * Cin), zc));
}

// Sum of the in-bounds taps' per-tap weight sums for output pixel (h, w).
__device__ inline int conv_row_sum(const int32_t* ts_n, int h, int w, int H, int W) {
    int s = 0;
#pragma unroll
    for (int dh = 0; dh < 3; ++dh) {
        int ih = h + dh - 1;
        if (ih < 0 || ih >= H) continue;
#pragma unroll
        for (int dw = 0; dw < 3; ++dw) {
            int iw = w + dw - 1;
            if (iw < 0 || iw >= W) continue;
            s += ts_n[dh * 3 + dw];
        }
    }
    return s;
}

// ---------------------------------------------------------------------------
// Host-side launchers implemented in the kernel translation units.
// ---------------------------------------------------------------------------
// mode: TASQ_SYMRANGE or TASQ_ASYM (then zcw [N] receives 128 - z; may be NULL otherwise)
cudaError_t launch_quant_weights(const void* w, int dtype, int N, int K, int mode, int8_t* sw, float* cw,
                                 float* zcw, float* alpha, cudaStream_t st);
// code_sums: [M] int32 sum_k s[m][k], or NULL
cudaError_t launch_quant_act_token(const void* x, int dtype, int M, int K, int n_bits, int mode, void* codes,
                                   int code_fmt, float* alpha, float* zc, int32_t* code_sums, cudaStream_t st);
cudaError_t launch_quant_act_tensor(const void* x, int dtype, int64_t count, int n_bits, int mode, void* codes,
                                    int code_fmt, float* alpha, float* zc, unsigned int* scratch, cudaStream_t st);
// sums[m] = sum_k codes[m][k] (int8 or fp16 codes, [M][K])
cudaError_t launch_code_row_sums(const void* codes, int code_fmt, int M, int K, int32_t* sums, cudaStream_t st);
// zcw: [N] weight zero offsets, or NULL for a symmetric pack
cudaError_t launch_pack(int kind, const int8_t* sw, const float* cw, const float* zcw, const float* bias, int N, int K,
                        int Cin, void* packed, cudaStream_t st);
cudaError_t launch_gemm_s8(const GemmArgs& a, int num_sms, cudaStream_t st);
// u' = fp16((bf16(x) . l2^T) / alpha[m]) into [M][64] fp16 (columns >= rank zero;
// rank 16 or 32; K % 16 == 0; alpha per token, or one value when per_tensor).
// status / timeout_ns: the device status word and the bound of the kernel's waits.
cudaError_t launch_lowrank_down(const void* x, int dtype, int M, int K, const uint16_t* l2, int rank,
                                const float* alpha, int per_tensor, uint16_t* u, int* status,
                                unsigned long long timeout_ns, cudaStream_t st);
constexpr int kLowRankCols = 64;  // fp16 columns of a u' row (one 128-byte swizzle atom)
// *kernels: how many kernels the call enqueued (the contraction, plus the split-K
// reduction when K is split).
cudaError_t launch_gemm_tc(const GemmArgs& a, int num_sms, cudaStream_t st, const char** why, int* kernels);
// Launch plan of the tensor-core route, decided on the host from the shape
// alone: tile configuration, token tiling, K slices and grid.  launch_gemm_tc
// launches exactly this plan.
struct TcPlan {
    int bch;              // output channels per tile (MMA M)
    int bt;               // tokens per tile (MMA N): 64, 192 or 256
    int nacc;             // accumulator buffers in tensor memory
    int tiles_ch;         // 128-channel blocks
    int64_t tiles_tok;    // token tiles
    int bw_log2, bhx;     // conv: token box of bhx image rows x 2^bw_log2 pixels
    int tiles_w, tiles_h; // conv: boxes across and down one image
    int splits;           // K slices (1: K is not split)
    int grid;             // CTAs of the contraction kernel
    int reduce_grid;      // CTAs of the split-K reduction (0: K is not split)
    const char* why;      // non-null: the route cannot take this shape
};
// Cin != 0 selects the convolution (M = B H W, K = 9 Cin); split_cap: elements
// of split-K scratch (0: no split).
TcPlan plan_gemm_tc(int M, int N, int K, int B, int H, int W, int Cin, int num_sms, int64_t split_cap);
size_t gemm_tc_part_bytes(int num_sms);  // scratch the TC route needs for `num_sms` persistent CTAs
constexpr int64_t kSplitBufBytes = int64_t(32) << 20;  // split-K partial sums (context scratch)
cudaError_t launch_selftest_timeout(int* status, unsigned long long timeout_ns, cudaStream_t st);
void set_noctx_error(const char* msg);
cudaError_t launch_selftest_quotients(const float* x, int nx, const float* a, int na, unsigned long long* mismatches,
                                      cudaStream_t st);

}  // namespace tasq
