// Masked contraction on the 5th-generation tensor cores (tcgen05, sm_103a).
//
// sm_103a has no int8 tcgen05 MMA, so the integer contraction runs on the
// fp16 MMA exactly: every int8 code is an exact fp16, every product of two
// codes (|p| <= 2^14) is exact, and an fp32 sum of integer products is exact
// while every partial sum stays within 2^24.  The packed weights carry, for
// each operating precision b, a certificate: the number of 64-wide K blocks
// over which 128 * sum_k |mask_b(w)| <= 2^24 holds for every channel.  The
// accumulator in tensor memory is restarted after each such chunk and
// drained into an int32 running sum (kept by each epilogue thread in the
// context's per-CTA scratch), so the final int32 accumulator equals the
// exact integer result.
//
// Operand roles (D = A * B^T with the output channels on the MMA's M side):
//   A: the weight tile, 128 channels x 128 K.  TMA brings the stored int8 codes
//      into shared memory; a converter warpgroup applies the operating-
//      precision mask (Eq. hw_rightshift: clear the low 8-b planes, one AND
//      per four codes), widens to fp16 and writes the tile straight into
//      tensor memory, where the MMA reads it.
//   B: the activation codes, held as fp16 integers in HBM, brought by TMA
//      into 128-byte-swizzled shared memory (a 2-D tile for a linear layer; a
//      4-D NHWC box shifted by the 3x3 tap for a convolution, whose padding
//      TMA fills with code 0).  4-bit codes also come as e5m2 bytes; with every
//      member at b <= 4 a linear layer's K loop runs on the 8-bit-float MMA kind
//      (256-code K blocks of two weight tiles).
//   D: fp32 accumulators in tensor memory, double-buffered (192- and 64-token
//      tiles) so the epilogue of one chunk overlaps the MMAs of the next, or
//      single (256-token tiles, one tile per CTA).
//
// Warp roles (608 threads): warp 0 issues the activation TMA; warp 1
// allocates tensor memory and issues the MMAs (one thread); warps 2..5 convert
// weights (and, for a single-tile CTA, join the epilogue once the last K block
// is converted); warps 6..17 drain accumulators and run the fused
// dequantization epilogue (linear outputs leave through TMA stores of
// swizzled [16 token][32 channel] boxes, staged in the idle activation ring on
// the CTA's last tile); warp 18 issues the weight TMA.  The grid is persistent:
// one CTA per SM walks the output tiles.  A call may hold several layers that
// read one input, each at its own b (channels [g Ng, (g+1) Ng) are member g's),
// listed in the arguments or, up to kMaxMembers, in device memory.  The roles
// diverge within warps, so the CTA's barriers count threads (ptx::cta_sync).
// Every wait is bounded by the context's time limit; a wait that gives up
// records TASQ_ERR_DEVICE_TIMEOUT, the CTA drains its copies in flight, frees
// its tensor memory and returns.
#include <cstdio>
#include <cstdlib>
#include <type_traits>

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>

#include "tasq_internal.cuh"
#include "tc_ptx.cuh"

namespace tasq {
namespace {

constexpr int BCH = 128;          // output channels per tile (MMA M)
constexpr int BK = 128;           // K per weight stage and per tensor-memory slot of converted weights
constexpr int XK = 64;            // K per activation TMA box (one 128-byte swizzle atom of fp16 codes)
constexpr int W_STAGES = 3;
constexpr int ASLOTS = 2;         // converted-weight slots in tensor memory (the configurations' default)
// Warps 2 .. 17 are converters (4, one per tensor-memory lane quadrant, or 8, two per
// quadrant each widening half of a K block) followed by epilogue warps (12 or 8).
constexpr int MID_WARPS = 16;
constexpr int MAX_EPI_WARPS = 12;
constexpr int WPROD_WARP = 2 + MID_WARPS;  // weight-tile producer
constexpr int THREADS = (WPROD_WARP + 1) * 32;
constexpr int W_STAGE = BCH * BK;       // 16 KB int8 codes, 128-byte rows
constexpr uint32_t A_SLOT_COLS = BK / 2;
constexpr uint32_t TMEM_COLS = 512;
constexpr int MAX_GPW = 3;              // most 32-token groups one epilogue warp drains
static_assert(BK == 2 * XK, "a stage is two 64-wide swizzle atoms");

// Tile configuration.  BT tokens per tile (MMA N); NACC accumulator buffers in
// tensor memory.  <192, 2>: the epilogue of one tile overlaps the next tile's
// MMAs.  <256, 1>: a wider MMA (the tensor pipe rather than the issuing thread
// bounds N = 256) for launches where every CTA gets a single tile; the
// accumulator then only has to wait for the drain between certified chunks.
// <64, 2>: for launches with few tokens, three times as many CTAs as <192, 2>
// and a third of its per-tile epilogue.
template <int BT_, int NACC_, int CONV_WARPS_ = 4, int AS_ = ASLOTS>
struct Cfg {
    static constexpr int BT = BT_;
    static constexpr int NACC = NACC_;
    static constexpr int AS = AS_;  // converted-weight slots in tensor memory
    static constexpr int CONV_WARPS = CONV_WARPS_;           // converter warps (4 or 8)
    static constexpr int CONV_SPLIT = CONV_WARPS / 4;        // converters per lane quadrant (K split)
    static constexpr int EPI_WARP0 = 2 + CONV_WARPS;         // first epilogue warp
    static constexpr int EPI_WARPS = MID_WARPS - CONV_WARPS; // epilogue warps
    static constexpr int EPI_PARTS = EPI_WARPS / 4;          // epilogue warps per lane quadrant
    // Q activation stages per K block: 1 (a 128-K stage, one wait per K block on
    // the MMA thread) or 2 (64-K stages released half a block earlier, for the
    // N = 256 tile, whose MMAs leave the issuing thread time for a second wait)
    static constexpr int Q = NACC == 2 ? 1 : 2;
    static constexpr int X_STAGES = NACC == 2 ? 3 : 4;  // activation stages in the ring
    static constexpr int X_HALF = BT * XK * 2;           // one 64-wide TMA box of fp16 codes
    static constexpr int X_STAGE = (2 / Q) * X_HALF;
    static constexpr int DONE = 2 * X_STAGES;            // stage-completion barriers (ring of MMA commits)
    static constexpr int GROUPS = BT / 32;               // 32-token column groups of the accumulator
    static constexpr int GPW = (GROUPS + EPI_PARTS - 1) / EPI_PARTS;  // groups per epilogue warp
    // the single-tile configuration lets 4 converter warps, idle once the last K block
    // is converted, drain a fourth share of the tile's groups
    static constexpr bool HELPERS = NACC == 1 && CONV_WARPS == 4;
    static constexpr int EPI_SLOTS = EPI_WARPS + (HELPERS ? 4 : 0);
    // output boxes ([16 tokens][32 channels] bf16, 1 KB) one epilogue warp stores per tile:
    // two per 32-token group it drains (the converter helpers drain at most as many)
    static constexpr int PIECES = 2 * GPW;
    static constexpr uint32_t ACC_COL = 0;               // NACC x BT fp32 accumulators
    static constexpr uint32_t A_COL = NACC * BT;         // ASLOTS x BK/2 columns (fp16 pairs)
    static constexpr uint32_t IDESC = ptx::idesc_f16_f32(BCH, BT);
    static constexpr uint32_t IDESC8 = ptx::idesc_e5m2_f32(BCH, BT);  // the 8-bit route
    static_assert(DONE % X_STAGES == 0 && DONE >= (AS + 1) * Q, "completion ring covers both reuse distances");
    // A converter arrives on K block j's first-stage barrier after the MMAs of block j - AS
    // completed; that barrier last served block j - X_STAGES / Q, whose phase must be closed
    // by then, or the arrival would count toward the wrong phase.
    static_assert(AS * Q <= X_STAGES, "converter arrivals stay within the stage ring");
    static_assert(Q == 1 || X_STAGES % 2 == 0, "first-half stages must keep their parity");
    static_assert(A_COL + AS * A_SLOT_COLS <= TMEM_COLS, "tensor memory budget");
    static_assert(GPW <= MAX_GPW && BT <= 256 && BT % 32 == 0, "tile shape");
    static_assert(!HELPERS || (GROUPS + EPI_PARTS) / (EPI_PARTS + 1) <= GPW, "helpers drain at most GPW groups");
    static_assert(EPI_SLOTS * PIECES * 1024 <= X_STAGES * X_STAGE, "a CTA's last tile stages its boxes in the ring");
    static_assert((CONV_WARPS == 4 || CONV_WARPS == 8) && EPI_WARPS <= MAX_EPI_WARPS, "warp roles");
};
using CfgStd = Cfg<192, 2>;
using CfgWide = Cfg<256, 1>;
// few tokens (cross-attention keys and values): more CTAs, shorter epilogue; its tensor memory
// has room for a third converted-weight slot (2 x 64 + 3 x 64 columns), which gives the
// converters a block more of slack (measured ~1-2 % per layer)
using CfgNarrow = Cfg<64, 2, 4, 3>;
// The two-accumulator tiles for linear layers whose codes also come as e5m2: the 8-bit
// route's block of two weight tiles is shared out between two converter warps per lane
// quadrant (one tile each), with eight epilogue warps.
using CfgStdF8 = Cfg<192, 2, 8>;
using CfgNarrowF8 = Cfg<64, 2, 8, 3>;

// Synchronisation is arranged so that the single MMA-issuing thread, whose
// per-instruction cost bounds the K loop, does one wait and one commit per
// activation stage.  Stage u (u = Q j + i for part i of K block j):
//   xfull[u % X_STAGES]  completes when its activation bytes have landed (TMA
//                 transaction bytes) and, for the first stage of a K block,
//                 when the four converter warps have written the block's
//                 weights into tensor-memory slot j % AS;
//   done[u % DONE]  completes when the MMAs reading stage u have finished; the
//                 activation producer waits on it before refilling the stage
//                 with u + X_STAGES, the converters (on the last stage of block
//                 j) before overwriting slot j % AS with block j + AS.
// The weight ring is separate: a weight stage is released as soon as the
// converters have read it, so weight tiles run several K blocks ahead.
template <class C>
struct Smem {
    uint8_t x[C::X_STAGES][C::X_STAGE];  // 1024-aligned (128-byte swizzle atoms)
    uint8_t w[W_STAGES][W_STAGE];
    float ep_al[C::EPI_SLOTS][C::GPW][32], ep_zc[C::EPI_SLOTS][C::GPW][32];  // per warp, per group, per column
    int ep_tok[C::EPI_SLOTS][C::GPW][32], ep_tap[C::EPI_SLOTS][C::GPW][32];
    float ep_t[C::EPI_SLOTS][C::GPW][32];  // asymmetric weights: per-column activation sums t
    // per-warp bf16 transpose tile, 16 tokens x 32 channels (64-byte rows); linear layers
    // keep it in the output tensor map's 64-byte swizzle (16-byte chunk c of row t at
    // c ^ ((t >> 1) & 3)), whose pattern repeats every 512 bytes
    alignas(1024) uint16_t ep_stage[C::EPI_SLOTS][16 * 32];
    uint64_t xfull[C::X_STAGES], done[C::DONE];
    uint64_t wfull[W_STAGES], wempty[W_STAGES];
    uint64_t accfull[C::NACC], accempty[C::NACC];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    // a member list in device memory: each member's b, and per warp the set of the
    // precisions its members run at (bit b; bit 0 for a member that did not resolve)
    uint8_t mbits[kMaxMembers];
    uint32_t wpresent[THREADS / 32];
};
template <class C>
constexpr int smem_bytes() { return int(sizeof(Smem<C>)) + 1024; }
static_assert(smem_bytes<CfgStd>() <= 227 * 1024 && smem_bytes<CfgWide>() <= 227 * 1024 &&
                  smem_bytes<CfgNarrow>() <= 227 * 1024 && smem_bytes<CfgStdF8>() <= 227 * 1024 &&
                  smem_bytes<CfgNarrowF8>() <= 227 * 1024,
              "shared memory per CTA");

struct TcParams {
    GemmArgs a;
    int conv;
    int tiles_ch, tiles_tok;  // tiles of BCH channels x BT tokens
    // conv: a token tile is a box of bhx rows x 2^bw_log2 pixels
    int bw_log2, bhx, tiles_w, tiles_h;
    // split-K: each tile's K blocks are cut into `splits` contiguous slices; a
    // slice writes its exact int32 partial sums to split_out[slice][token][n]
    // and a second kernel adds the slices and applies the epilogue
    int splits;
    int32_t* split_out;
};

// One unit of work: a tile and a contiguous range of its K blocks.
struct Work {
    int t, slice, kb_lo, kb_hi, nch;
};
__device__ __forceinline__ Work work_item(const TcParams& p, int w, int KT, int chunk) {
    Work r;
    r.t = w / p.splits;
    r.slice = w - r.t * p.splits;
    r.kb_lo = (r.slice * KT) / p.splits;
    r.kb_hi = ((r.slice + 1) * KT) / p.splits;
    r.nch = (r.kb_hi - r.kb_lo + chunk - 1) / chunk;
    return r;
}

template <class C>
struct Waiter {
    Smem<C>* s;
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

// Ring position: slot index and phase parity, advanced without divisions.
template <int N>
struct Ring {
    int slot = 0;
    uint32_t phase = 0;
    __device__ __forceinline__ void next() {
        if (++slot == N) {
            slot = 0;
            phase ^= 1u;
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

// e5m2 bytes of four masked codes whose values have at most three significant bits
// (b <= 4): the upper bytes of their fp16 values (see ptx::e5m2x4).
__device__ __forceinline__ uint32_t masked_e5m2x4(uint32_t w, uint32_t m) {
    uint32_t lo, hi;
    widen4(w, m, lo, hi);
    return ptx::e5m2x4(lo, hi);
}

struct TileCoord {
    int ch0;  // first channel of the tile's 128 rows
    int tok0, img, h0, w0;
};

template <bool CONV, int BT>
__device__ __forceinline__ TileCoord tile_coord(const TcParams& p, int t) {
    TileCoord c;
    c.ch0 = (t % p.tiles_ch) * BCH;
    const int tt = t / p.tiles_ch;
    c.tok0 = c.img = c.h0 = c.w0 = 0;
    if constexpr (CONV) {
        const int per_img = p.tiles_h * p.tiles_w;
        c.img = tt / per_img;
        c.h0 = ((tt % per_img) / p.tiles_w) * p.bhx;
        c.w0 = (tt % p.tiles_w) << p.bw_log2;
    } else {
        c.tok0 = tt * BT;
    }
    return c;
}

// Whether a launch whose codes also come as e5m2 takes the 8-bit route: every member
// layer's b is known (the table lookup succeeded) and at most 4, so that its masked
// weight codes have at most three significant bits.
__device__ __forceinline__ bool f8_route(const GemmArgs& a, uint32_t gbits) {
    bool f8 = gbits != 0;
#pragma unroll
    for (int g = 0; g < kMaxGroups; ++g)
        if (g < a.groups && int((gbits >> (4 * g)) & 15u) > kBMaxF8) f8 = false;
    return f8;
}

// CONV selects the implicit-GEMM 3x3 convolution (one instantiation per operand
// layout, so neither pays for the other's index arithmetic); ZP the four-term
// epilogue of asymmetric weights; F8 a linear layer whose codes also come as e5m2
// bytes (tm_x8): when every member's b is <= 4 the K loop runs on the 8-bit route
// (kind::f8f6f4 MMAs with e5m2 operands, 32 codes of K per instruction), else on
// the fp16 codes as usual; LR a linear layer with a 16-bit low-rank branch: after
// the last K block of each tile one more block of fp16 MMAs adds
// u'[m] . (l1[n] / c_w[n]) to the accumulator (u' in tm_u, the weights' block
// converted from l1 by the converters), so that the epilogue's dequantization
// scales it back to u . l1 (unsplit launches only); MANY a grouped linear layer whose
// member list is in device memory (a.d_layers, up to kMaxMembers members; unsplit
// launches only): every CTA resolves each member's b into shared memory.
template <bool CONV, bool ZP, class C, bool F8 = false, bool LR = false, bool MANY = false>
__global__ void __maxnreg__(96)
    gemm_tc_kernel(const __grid_constant__ TcParams p, const __grid_constant__ CUtensorMap tm_x,
                   const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_y,
                   const __grid_constant__ CUtensorMap tm_x8, const __grid_constant__ CUtensorMap tm_u) {
    constexpr int X_STAGES = C::X_STAGES, X_HALF = C::X_HALF, X_STAGE = C::X_STAGE, NACC = C::NACC;
    constexpr int Q = C::Q, DONE = C::DONE;
    constexpr int BT = C::BT, GPW = C::GPW;
    constexpr int EPI_WARP0 = C::EPI_WARP0, EPI_WARPS = C::EPI_WARPS, EPI_PARTS = C::EPI_PARTS;
    constexpr int CONV_WARPS = C::CONV_WARPS;
    extern __shared__ uint8_t smem_raw[];
    Smem<C>* s = reinterpret_cast<Smem<C>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const GemmArgs& a = p.a;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const Waiter<C> wt{s, &a};

    // Set-up that does not depend on b (tensor memory, descriptor prefetch) overlaps the
    // loads that resolve it.
    if (warp == 1) {
        ptx::tmem_alloc(ptx::smem_u32(&s->tmem_base), TMEM_COLS);
        ptx::tmem_relinquish();
        ptx::tc_fence_before();
    }
    // the certificate of every b is loaded alongside the stage and table reads
    int cert[kNumB];
#pragma unroll
    for (int i = 0; i < kNumB; ++i) cert[i] = a.hdr->chunk_kb[kBMin + i];
    // b of every member layer (one member unless the call is grouped); b = member 0's.
    // A member list in device memory (MANY): one thread per member resolves its b into
    // shared memory and each warp gathers the set of precisions present; gbits then
    // stands for that set (bit b for each b present, 0 when a member did not resolve)
    // once the barrier below has passed.
    uint32_t gbits = 0;
    if constexpr (MANY) {
        uint32_t present = 0;
        if (int(threadIdx.x) < a.groups) {
            const int bg = resolve_member_bits(a, int(threadIdx.x));
            s->mbits[threadIdx.x] = uint8_t(bg);
            present = 1u << bg;
        }
        present = __reduce_or_sync(0xFFFFFFFFu, present);
        if (lane == 0) s->wpresent[warp] = present;
        ptx::cta_sync();
#pragma unroll
        for (int i = 0; i < THREADS / 32; ++i) gbits |= s->wpresent[i];
        if (gbits & 1u) {
            if (threadIdx.x == 0) set_status(a.status, TASQ_ERR_DEVICE);
            gbits = 0;
        }
    } else {
        gbits = resolve_group_bits(a);
    }
    const int b = int(gbits & 15u);
    // the shortest certified chunk over the members' precisions is valid for all of them
    int chunk_kb = 0x7FFFFFFF;
    if constexpr (MANY) {
#pragma unroll
        for (int i = 0; i < kNumB; ++i)
            if ((gbits >> (kBMin + i)) & 1u) chunk_kb = min(chunk_kb, cert[i]);
    } else {
#pragma unroll
        for (int g = 0; g < kMaxGroups; ++g) {
            const int bg = int((gbits >> (4 * g)) & 15u);
#pragma unroll
            for (int i = 0; i < kNumB; ++i)
                if (g < a.groups && bg == kBMin + i) chunk_kb = min(chunk_kb, cert[i]);
        }
    }
    // The 8-bit route (uniform over the grid).  Its K block is 256 codes: their e5m2 bytes
    // fill exactly the activation stage, the tensor-memory weight slot and the MMA
    // descriptors of a 128-code fp16 block (a 128-byte row segment per 32-byte K step
    // either way), so both routes share every ring; only the MMA kind, the activation
    // tensor map, the weight tiles per block (two) and the converters' arithmetic differ.
    // It needs an unsplit launch and an exact chunk of at least one such block.
    const int64_t chunk_k64 = int64_t(chunk_kb) * a.chunk_scale;  // exact chunk in 64-code blocks
    const bool f8 = F8 && p.splits == 1 && chunk_k64 >= 2 * BK / kCertKBlock &&
                    (MANY ? gbits != 0 && (gbits >> (kBMaxF8 + 1)) == 0 : f8_route(a, gbits));
    const int KBLK = f8 ? 2 * BK : BK;  // codes of K per block
    if (threadIdx.x == 0) {
        for (int i = 0; i < X_STAGES; ++i)  // producer's expect_tx (+ the converter warps on first stages)
            ptx::mbar_init(ptx::smem_u32(&s->xfull[i]), i % Q == 0 ? 1 + CONV_WARPS : 1);
        for (int i = 0; i < DONE; ++i) ptx::mbar_init(ptx::smem_u32(&s->done[i]), 1);  // the MMA commit
        for (int i = 0; i < W_STAGES; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->wfull[i]), 1);
            ptx::mbar_init(ptx::smem_u32(&s->wempty[i]), CONV_WARPS);  // every converter warp, every tile
        }
        for (int i = 0; i < NACC; ++i) {
            ptx::mbar_init(ptx::smem_u32(&s->accfull[i]), 1);
            ptx::mbar_init(ptx::smem_u32(&s->accempty[i]), EPI_WARPS);
        }
        ptx::mbar_init(ptx::smem_u32(&s->drain), 1);
        s->abort = 0;
        ptx::fence_mbar_init();
        ptx::prefetch_tmap(f8 ? &tm_x8 : &tm_x);
        ptx::prefetch_tmap(&tm_w);
        if constexpr (!CONV) ptx::prefetch_tmap(&tm_y);
    }
    const int KT = (a.K + KBLK - 1) / KBLK;
    // the exact chunk is in 64-wide K blocks; a run of c64 of them covers c64 / (KBLK / 64) of ours
    const int64_t chunk64 = chunk_k64 / (KBLK / kCertKBlock);
    const int chunk = chunk64 < 1 ? 1 : (chunk64 > KT ? KT : int(chunk64));
    const int works = p.tiles_ch * p.tiles_tok * p.splits;
    const int unit = int(blockIdx.x), units = int(gridDim.x);
    ptx::cta_sync();
    ptx::tc_fence_after();
    const uint32_t tmem = s->tmem_base;
    if (MANY ? gbits == 0 : b == 0) {  // uniform across the grid (a launch-wide check, recorded in the status word)
        if (warp == 1) ptx::tmem_dealloc(tmem, TMEM_COLS);
        return;
    }
    // b of output channel n: its member layer's
    auto bits_of = [&](int n) {
        if constexpr (MANY) return int(s->mbits[min(n / a.group_n, a.groups - 1)]);
        else return channel_bits(a, gbits, n);
    };
    // Programmatic dependent launch: this grid may start while the previous kernel
    // (normally the quantization of this layer's activations) still runs.  Only the
    // activation codes and the per-token scales come from it, so only the warps that
    // read those (the activation producer and the epilogue) wait for it; the packed
    // weights, the bit table and the stage were complete before that kernel began,
    // so the weight ring, the converters and the MMA issuer start at once.

    if (warp == 0) {
        // --------------------------------------------- activation producer
        if (lane == 0) {
            ptx::grid_dependency_wait();
            int u = 0;  // activation stages issued by this CTA
            bool ok = true;
            for (int w = unit; w < works && ok; w += units) {
                const Work wk = work_item(p, w, KT, chunk);
                const TileCoord tc = tile_coord<CONV, BT>(p, wk.t);
                // (LR: the tile's last block is the low-rank block, stages of u' rows)
                for (int kq = wk.kb_lo * Q; kq < (wk.kb_hi + (LR ? 1 : 0)) * Q; ++kq, ++u) {
                    if (u >= X_STAGES && !wt.wait(&s->done[(u - X_STAGES) % DONE], ((u - X_STAGES) / DONE) & 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fb = ptx::smem_u32(&s->xfull[u % X_STAGES]);
                    const uint32_t dst = ptx::smem_u32(s->x[u % X_STAGES]);
                    ptx::mbar_arrive_expect_tx(fb, X_STAGE);
#pragma unroll
                    for (int hh = 0; hh < 2 / Q; ++hh) {
                        // box hh of the stage: 128 bytes of each token's row, 64 fp16 codes
                        // or 128 e5m2 codes
                        const int kh = kq * (BK / Q) + hh * XK;
                        if (LR && kq >= wk.kb_hi * Q) {
                            // u' columns 0..63; the block's other boxes lie past the 64
                            // columns and are filled with zeros
                            ptx::tma_load_2d(dst + hh * X_HALF, &tm_u, fb, kh - wk.kb_hi * BK, tc.tok0);
                        } else if constexpr (CONV) {
                            // a 128-wide K block may straddle two taps when Cin % 128 == 64
                            const int tap = kh / a.Cin, c0 = kh - tap * a.Cin;
                            ptx::tma_load_4d(dst + hh * X_HALF, &tm_x, fb, c0, tc.w0 + tap % 3 - 1, tc.h0 + tap / 3 - 1,
                                             tc.img);
                        } else if (F8 && f8) {
                            ptx::tma_load_2d(dst + hh * X_HALF, &tm_x8, fb, 2 * kh, tc.tok0);
                        } else {
                            ptx::tma_load_2d(dst + hh * X_HALF, &tm_x, fb, kh, tc.tok0);
                        }
                    }
                }
            }
            // the next kernel may be launched while this grid drains
            ptx::grid_launch_dependents();
            // copies still in flight must land before the CTA may exit: the MMAs
            // of the last stages consumed them (or the CTA is aborting)
            for (int i = u - X_STAGES < 0 ? 0 : u - X_STAGES; i < u; ++i)
                wt.wait(&s->done[i % DONE], (i / DONE) & 1, true);
        }
    } else if (warp == WPROD_WARP) {
        // ------------------------------------------------ weight producer
        if (lane == 0) {
            Ring<W_STAGES> rw;
            int nw = 0;
            bool ok = true;
            const int wpb = f8 ? 2 : 1;  // 128-code weight tiles per K block
            for (int w = unit; w < works && ok; w += units) {
                const Work wk = work_item(p, w, KT, chunk);
                const int ch0 = tile_coord<CONV, BT>(p, wk.t).ch0;
                for (int kw = wk.kb_lo * wpb; kw < wk.kb_hi * wpb; ++kw, ++nw, rw.next()) {
                    if (!wt.wait(&s->wempty[rw.slot], rw.phase ^ 1)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fb = ptx::smem_u32(&s->wfull[rw.slot]);
                    ptx::mbar_arrive_expect_tx(fb, W_STAGE);
                    ptx::tma_load_2d(ptx::smem_u32(s->w[rw.slot]), &tm_w, fb, kw * BK, ch0);
                    if (nw == W_STAGES - 1) {
                        // the ring is full: pull the first tile's next weight tiles into L2
                        // ahead of it (after its first loads, which the converters wait for)
                        for (int k2 = kw + 1; k2 < wk.kb_hi * wpb && k2 < (wk.kb_lo + 8) * wpb; ++k2)
                            ptx::tma_prefetch_2d(&tm_w, k2 * BK, ch0);
                    }
                }
            }
            for (int j = nw - W_STAGES < 0 ? 0 : nw - W_STAGES; j < nw; ++j)
                wt.wait(&s->wfull[j % W_STAGES], (j / W_STAGES) & 1, true);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int it = 0, cc = 0;
            bool ok = true;
            for (int w = unit; w < works && ok; w += units) {
                const Work wk = work_item(p, w, KT, chunk);
                for (int c = 0; c < wk.nch && ok; ++c, ++cc) {
                    const int buf = cc % NACC;
                    if (!wt.wait(&s->accempty[buf], ((cc / NACC) & 1) ^ 1)) {
                        ok = false;
                        break;
                    }
                    ptx::tc_fence_after();
                    const uint32_t d = tmem + C::ACC_COL + buf * BT;
                    const int kb0 = wk.kb_lo + c * chunk;
                    // (LR: the last chunk also takes the low-rank block, kb == kb_hi)
                    const int kb_end = min(wk.kb_hi, kb0 + chunk) + (LR && c == wk.nch - 1 ? 1 : 0);
                    for (int kb = kb0; kb < kb_end && ok; ++kb, ++it) {
                        const uint32_t acol = tmem + C::A_COL + (it % C::AS) * A_SLOT_COLS;
                        const bool lrb = LR && kb == wk.kb_hi;  // the low-rank block: fp16, 64 columns of K
                        for (int i = 0; i < Q; ++i) {
                            const int u = it * Q + i;
                            // activations landed (and, for i == 0, the converters wrote slot it % AS)
                            if (!wt.wait(&s->xfull[u % X_STAGES], (u / X_STAGES) & 1)) {
                                ok = false;
                                break;
                            }
                            ptx::tc_fence_after();
                            for (int hh = 0; hh < 2 / Q; ++hh) {
                                // one 128-byte swizzle atom per row (64 fp16 or 128 e5m2 codes); a K
                                // step (16 fp16 or 32 e5m2 codes) is 32 bytes along its rows
                                const uint64_t bdesc =
                                    ptx::sw128_kmajor_desc(ptx::smem_u32(s->x[u % X_STAGES] + hh * X_HALF));
                                const int k0 = (i * (2 / Q) + hh) * (XK / 16);  // K step within the block
                                if (lrb) {
                                    if (k0 == 0)
                                        for (int kk = 0; kk < XK / 16; ++kk)
                                            ptx::mma_f16_ts(d, acol + kk * 8, bdesc + uint64_t((kk * 32) >> 4),
                                                            C::IDESC, 1u);
                                } else if (F8 && f8) {
                                    for (int kk = 0; kk < XK / 16; ++kk)
                                        ptx::mma_f8_ts(d, acol + (k0 + kk) * 8, bdesc + uint64_t((kk * 32) >> 4),
                                                       C::IDESC8, (kb > kb0 || k0 + kk > 0) ? 1u : 0u);
                                } else {
                                    for (int kk = 0; kk < XK / 16; ++kk)
                                        ptx::mma_f16_ts(d, acol + (k0 + kk) * 8, bdesc + uint64_t((kk * 32) >> 4),
                                                        C::IDESC, (kb > kb0 || k0 + kk > 0) ? 1u : 0u);
                                }
                            }
                            ptx::mma_commit(ptx::smem_u32(&s->done[u % DONE]));
                        }
                    }
                    if (ok) ptx::mma_commit(ptx::smem_u32(&s->accfull[buf]));
                }
            }
            // every MMA issued must finish before tensor memory is released
            ptx::mma_commit(ptx::smem_u32(&s->drain));
            wt.wait(&s->drain, 0, true);
        }
    } else if (warp < EPI_WARP0) {
        // ------------------------------------------- weight mask + convert
        // Converter warp c serves the 32 channel rows of lane quadrant c % 4 and part
        // kp = (c - 2) / 4 of each K block: the fp16 route's block (one 128-code weight
        // tile) is cut into CONV_SPLIT runs of codes, the 8-bit route's block (two tiles)
        // into CONV_SPLIT runs of tiles.  Either way a part fills 64 / CONV_SPLIT
        // tensor-memory columns of the block's slot.
        constexpr int SPLIT = C::CONV_SPLIT;
        constexpr int CH = 8 / SPLIT;        // fp16 route: 16-byte chunks of a row per part
        constexpr int NF = 64 / SPLIT;       // 32-bit words (columns) per part and block
        const int q = warp & 3;              // tensor-memory lane quadrant
        const int kp = (warp - 2) >> 2;      // K part
        const int r = q * 32 + lane;         // channel row within the tile
        const uint32_t lane_base = tmem + (uint32_t(q * 32) << 16);
        Ring<W_STAGES> rw;
        int it = 0;
        bool ok = true;
        for (int w = unit; w < works && ok; w += units) {
            const Work wk = work_item(p, w, KT, chunk);
            // this row's channel runs at its layer's b (a grouped call holds several layers)
            const uint32_t m = mask_word(bits_of(tile_coord<CONV, BT>(p, wk.t).ch0 + r));
            if constexpr (LR) {  // the low-rank block's l1 row, read after the tile's K blocks
                const int n = tile_coord<CONV, BT>(p, wk.t).ch0 + r;
                if (kp == 0 && n < a.N) asm volatile("prefetch.global.L1 [%0];" ::"l"(a.lr_l1 + int64_t(n) * a.lr_rank));
            }
            // (LR: the tile's last block is the low-rank block, kb == kb_hi)
            for (int kb = wk.kb_lo; kb < wk.kb_hi + (LR ? 1 : 0); ++kb, ++it) {
                // Row r of a tile holds 128 codes; 16-byte chunk c sits at c ^ (r & 7) (128-byte
                // swizzle).  Mask and widen before waiting for the slot, so that only the
                // tensor-memory store remains once the MMA releases it.
                uint32_t f[NF];
                if (LR && kb == wk.kb_hi) {
                    // the low-rank block's weights: fp16(l1[n][j] * RN(1 / c_w[n])) for the
                    // rank columns j (the first part's first words), zeros elsewhere; no
                    // tile of the weight ring
#pragma unroll
                    for (int i = 0; i < NF; ++i) f[i] = 0u;
                    const int n = tile_coord<CONV, BT>(p, wk.t).ch0 + r;
                    if (kp == 0 && n < a.N) {
                        const float rcw = __frcp_rn(a.cw[n]);
                        const uint4* lp = reinterpret_cast<const uint4*>(a.lr_l1 + int64_t(n) * a.lr_rank);
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {  // rank 32: four 16-byte loads; rank 16: two
                            if (q4 >= a.lr_rank / 8) break;
                            const uint4 v = __ldg(lp + q4);
                            const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const float lo = __fmul_rn(__uint_as_float(wv[i] << 16), rcw);
                                const float hi = __fmul_rn(__uint_as_float(wv[i] & 0xFFFF0000u), rcw);
                                const __half2 h = __floats2half2_rn(lo, hi);
                                f[4 * q4 + i] = *reinterpret_cast<const uint32_t*>(&h);
                            }
                        }
                    }
                } else if (F8 && f8) {
                    // e5m2 (b <= 4): one word per 4 codes, 32 words per tile.  Every
                    // converter warp passes both tiles of the block through the ring in
                    // order (a part that skipped the other part's tiles could wait on a
                    // slot two phases ahead, which one parity bit cannot tell apart) and
                    // converts its own: both tiles, or tile kp of two parts.
#pragma unroll
                    for (int t = 0; t < 2; ++t) {
                        if (!wt.wait(&s->wfull[rw.slot], rw.phase)) {
                            ok = false;
                            break;
                        }
                        if (SPLIT == 1 || t == kp) {
                            const int o = SPLIT == 1 ? 32 * t : 0;
                            const uint8_t* row = s->w[rw.slot] + r * BK;
#pragma unroll
                            for (int c = 0; c < 8; ++c) {
                                const uint4 u = *reinterpret_cast<const uint4*>(row + ((c ^ (r & 7)) << 4));
                                f[o + 4 * c + 0] = masked_e5m2x4(u.x, m);
                                f[o + 4 * c + 1] = masked_e5m2x4(u.y, m);
                                f[o + 4 * c + 2] = masked_e5m2x4(u.z, m);
                                f[o + 4 * c + 3] = masked_e5m2x4(u.w, m);
                            }
                        }
                        __syncwarp();
                        if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->wempty[rw.slot]));
                        rw.next();
                    }
                    if (!ok) break;
                } else {
                    // fp16: two words per 4 codes
                    if (!wt.wait(&s->wfull[rw.slot], rw.phase)) {
                        ok = false;
                        break;
                    }
                    const uint8_t* row = s->w[rw.slot] + r * BK;
#pragma unroll
                    for (int c = 0; c < CH; ++c) {
                        const uint4 u = *reinterpret_cast<const uint4*>(row + (((kp * CH + c) ^ (r & 7)) << 4));
                        widen4(u.x, m, f[8 * c + 0], f[8 * c + 1]);
                        widen4(u.y, m, f[8 * c + 2], f[8 * c + 3]);
                        widen4(u.z, m, f[8 * c + 4], f[8 * c + 5]);
                        widen4(u.w, m, f[8 * c + 6], f[8 * c + 7]);
                    }
                    __syncwarp();
                    if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->wempty[rw.slot]));
                    rw.next();
                }
                // slot it % AS last held K block it - AS: its MMAs must have finished
                // (the last activation stage of that block completes after all its MMAs)
                if (it >= C::AS && !wt.wait(&s->done[((it - C::AS) * Q + Q - 1) % DONE],
                                            (((it - C::AS) * Q + Q - 1) / DONE) & 1)) {
                    ok = false;
                    break;
                }
                {
                    const uint32_t dst = lane_base + C::A_COL + (it % C::AS) * A_SLOT_COLS + kp * NF;
#pragma unroll
                    for (int h = 0; h < NF / 32; ++h)
                        ptx::tmem_st32(dst + 32 * h, *reinterpret_cast<const uint32_t(*)[32]>(&f[32 * h]));
                }
                ptx::tmem_wait_st();
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&s->xfull[(it * Q) % X_STAGES]));
            }
        }
    }
    // Helper mode (uniform over the CTA): a single-tile CTA whose tile is one
    // certified chunk (linear layers) drains it with the converter warps too,
    // four warps per lane quadrant instead of three.
    const bool helpers = !CONV && C::HELPERS && unit < works && works <= units &&
                         work_item(p, unit, KT, chunk).nch == 1;
    if ((warp >= EPI_WARP0 && warp < EPI_WARP0 + EPI_WARPS) || (helpers && warp >= 2 && warp < EPI_WARP0)) {
        // ------------------------------------- accumulator drain + epilogue
        ptx::grid_dependency_wait();  // per-token scales come from the previous kernel
        // shared-scratch slot: epilogue warps 0..11, converter warps 12..15
        const int e = warp >= EPI_WARP0 ? warp - EPI_WARP0 : EPI_WARPS + (warp - 2);
        const int q = warp & 3;              // lane quadrant: channels q*32 .. q*32+31
        const int part = e >> 2;             // which share of the tile's 32-token groups
        const int gpw = helpers ? (C::GROUPS + EPI_PARTS) / (EPI_PARTS + 1) : GPW;  // groups per share
        const int r = q * 32 + lane;
        const uint32_t lane_base = tmem + (uint32_t(q * 32) << 16);
        // row sums at each channel's b (convolutions are never grouped)
        const int32_t* ts_b = CONV ? a.ts + int64_t(b - kBMin) * a.N * 9 : nullptr;
        auto rs_of = [&](int n) { return a.rs[int64_t(bits_of(n) - kBMin) * a.N + n]; };
        constexpr bool zp = ZP;  // asymmetric weights: the four-term epilogue
        int cc = 0;
        bool ok = true;
        for (int w = unit; w < works && ok; w += units) {
            const Work wk = work_item(p, w, KT, chunk);
            const int nchunks = wk.nch;
            const TileCoord tc = tile_coord<CONV, BT>(p, wk.t);
            const int n = tc.ch0 + r;
            const bool n_ok = n < a.N;
            // row sums as fp32: |sum| < 2^24, so the values and every partial sum
            // of in-bounds taps below are exact, equal to float(int sum)
            float cw = 0.f, bias = 0.f, rs = 0.f;
            [[maybe_unused]] float zcw_l = 0.f;  // asymmetric weights: this lane's channel zero offset
            float ts[9];
#pragma unroll
            for (int i = 0; i < 9; ++i) ts[i] = 0.f;
            if (n_ok) {
                cw = a.cw[n];
                bias = a.bias[n];
                if constexpr (zp) zcw_l = a.zcw[n];
                if constexpr (CONV) {
#pragma unroll
                    for (int i = 0; i < 9; ++i) ts[i] = __int2float_rn(ts_b[int64_t(n) * 9 + i]);
                } else {
                    rs = __int2float_rn(rs_of(n));
                }
            }

            // Linear layers drain the accumulator in the mma-fragment layout (see
            // finish16f): this thread's channels are lane/4 + 8k, k = 0..3.
            [[maybe_unused]] float cwf[4], biasf[4], rsf[4], zcwf[4];
            if constexpr (!CONV) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int nk = tc.ch0 + q * 32 + (lane >> 2) + 8 * k;
                    const bool ok_k = nk < a.N;
                    cwf[k] = ok_k ? a.cw[nk] : 0.f;
                    biasf[k] = ok_k ? a.bias[nk] : 0.f;
                    rsf[k] = ok_k ? __int2float_rn(rs_of(nk)) : 0.f;
                    zcwf[k] = ok_k && zp ? a.zcw[nk] : 0.f;
                }
            }

            // Token index, (conv) in-bounds taps and per-token scales of column j = lane of
            // each of this warp's two groups, written to this warp's shared scratch before
            // the accumulator wait, so the global loads' latency hides under the MMAs.
            bool all_tok_g[GPW];
            // where this tile's output boxes are staged: this warp's box (step 0), or (the
            // CTA's last tile) a 1 KB box per piece in the activation ring
            uint32_t stg_base = ptx::smem_u32(s->ep_stage[e]), stg_step = 0;
            __syncwarp();  // the previous tile's reads of the scratch are done
#pragma unroll
            for (int gi = 0; gi < GPW; ++gi) {
                // beyond the tile (no token) when part * gpw + gi >= GROUPS or gi >= gpw
                const int jt = gi < gpw ? (part * gpw + gi) * 32 + lane : BT;
                int tok = -1, tap = 0;
                if constexpr (CONV) {
                    const int hh = tc.h0 + (jt >> p.bw_log2), ww = tc.w0 + (jt & ((1 << p.bw_log2) - 1));
                    if (hh < a.H && ww < a.W) {
                        tok = (tc.img * a.H + hh) * a.W + ww;
#pragma unroll
                        for (int dh = 0; dh < 3; ++dh)
#pragma unroll
                            for (int dw = 0; dw < 3; ++dw) {
                                const int ih = hh + dh - 1, iw = ww + dw - 1;
                                if (ih >= 0 && ih < a.H && iw >= 0 && iw < a.W) tap |= 1 << (dh * 3 + dw);
                            }
                    }
                } else {
                    tok = jt < BT && tc.tok0 + jt < a.M ? tc.tok0 + jt : -1;
                }
                if constexpr (CONV) {
                    if (jt >= BT) tok = -1;
                }
                if constexpr (zp) {
                    // asymmetric weights: the column's activation sum t (conv: over in-bounds taps)
                    float t = 0.f;
                    if (tok >= 0)
                        t = CONV ? conv_token_zero_sum(a.code_sums, tok, a.H, a.W, a.Cin, a.zc[0])
                                 : token_zero_sum(a.code_sums[tok], a.K, a.zc[tok]);
                    s->ep_t[e][gi][lane] = t;
                }
                s->ep_tok[e][gi][lane] = tok;
                s->ep_tap[e][gi][lane] = tap;
                s->ep_al[e][gi][lane] = tok >= 0 ? (a.per_tensor ? a.alpha[0] : a.alpha[tok]) : 0.f;
                s->ep_zc[e][gi][lane] = tok >= 0 ? (a.per_tensor ? a.zc[0] : a.zc[tok]) : 0.f;
                all_tok_g[gi] = __all_sync(0xffffffffu, tok >= 0);
            }
            __syncwarp();
            // Epilogue of 16 consecutive columns j0..j0+15 of group g from exact
            // accumulator values (float-held integers when `fl`, else int32).
            // FL: the accumulator values are float-held integers (single-chunk tiles), else int32
            auto finish16 = [&](int gi, int j0, const uint32_t (&v)[16], auto fl_tag, bool all_tok) {
                constexpr bool fl = decltype(fl_tag)::value;
                [[maybe_unused]] const int g = part * gpw + gi;
                const float* my_al = s->ep_al[e][gi];
                const float* my_zc = s->ep_zc[e][gi];
                const int* my_tok = s->ep_tok[e][gi];
                [[maybe_unused]] const int* my_tap = s->ep_tap[e][gi];
                uint32_t yb2[8];
#pragma unroll
                for (int j4 = 0; j4 < 4; ++j4) {
                    const float4 al4 = *reinterpret_cast<const float4*>(my_al + j0 + 4 * j4);
                    const float4 zc4 = *reinterpret_cast<const float4*>(my_zc + j0 + 4 * j4);
                    const float al[4] = {al4.x, al4.y, al4.z, al4.w};
                    const float zc[4] = {zc4.x, zc4.y, zc4.z, zc4.w};
                    int4 tp4 = make_int4(0, 0, 0, 0);
                    if constexpr (CONV) tp4 = *reinterpret_cast<const int4*>(my_tap + j0 + 4 * j4);
                    [[maybe_unused]] const int tp[4] = {tp4.x, tp4.y, tp4.z, tp4.w};
                    float4 t4 = make_float4(0.f, 0.f, 0.f, 0.f);
                    if constexpr (zp) t4 = *reinterpret_cast<const float4*>(s->ep_t[e][gi] + j0 + 4 * j4);
                    [[maybe_unused]] const float tz[4] = {t4.x, t4.y, t4.z, t4.w};
                    float yf[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        float rsum = rs;
                        if constexpr (CONV) {
                            rsum = 0.f;
#pragma unroll
                            for (int k9 = 0; k9 < 9; ++k9) rsum = __fadd_rn(rsum, (tp[u] >> k9) & 1 ? ts[k9] : 0.f);
                        }
                        const uint32_t raw = v[4 * j4 + u];
                        float acc_f;
                        if constexpr (fl) acc_f = __uint_as_float(raw);
                        else acc_f = __int2float_rn(int(raw));
                        float uu = __fmaf_rn(zc[u], rsum, acc_f);
                        if constexpr (zp) uu = __fmaf_rn(zcw_l, tz[u], uu);  // asymmetric weights
                        yf[u] = __fmaf_rn(uu, __fmul_rn(al[u], cw), bias);
                    }
                    // two results per round-to-nearest-even conversion
#pragma unroll
                    for (int u = 0; u < 4; u += 2) {
                        const __nv_bfloat162 hb = __floats2bfloat162_rn(yf[u], yf[u + 1]);
                        yb2[2 * j4 + u / 2] = *reinterpret_cast<const uint32_t*>(&hb);
                    }
                }
                // Transpose the warp's 32 channels x 16 tokens through shared memory:
                // a [16 tokens][32 channels] bf16 box (64-byte rows).
                // (convolutions only: linear layers finish in finish16f)
                uint16_t* stg = s->ep_stage[e];
                __syncwarp();
#pragma unroll
                for (int j = 0; j < 16; ++j) stg[j * 32 + lane] = uint16_t(yb2[j >> 1] >> (16 * (j & 1)));
                {
                    // the box's pixels need not be consecutive rows of y: 16-byte stores
                    __syncwarp();
                    const int qc = lane & 3;  // 8-channel chunk of the row
                    const int nq = tc.ch0 + (warp & 3) * 32 + qc * 8;
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        const int t = rr * 8 + (lane >> 2);  // token row within the 16
                        const uint4 val = *reinterpret_cast<const uint4*>(stg + t * 32 + qc * 8);
                        const int tok = my_tok[j0 + t];
                        if (tok >= 0 && nq < a.N) *reinterpret_cast<uint4*>(a.y + int64_t(tok) * a.N + nq) = val;
                    }
                    __syncwarp();  // the box is read before the next one is written
                }
                if (a.acc && n_ok) {  // int32 accumulators (a debugging output): plain stores
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int tok = my_tok[j0 + j];
                        if (tok >= 0) a.acc[int64_t(tok) * a.N + n] = fl ? __float2int_rn(__uint_as_float(v[j])) : int(v[j]);
                    }
                }
            };

            // Linear-layer epilogue of 16 consecutive columns j0..j0+15 of group g from
            // values in the mma-fragment layout: with s = lane % 4, v[(k>>1)*8 + (k&1)*2
            // + 4*tp + e] is channel lane/4 + 8k, token j0 + 8*tp + 2s + e.  Four 8x8
            // transposed matrix stores build the [16 tokens][32 channels] box.
            [[maybe_unused]] auto finish16f = [&](int gi, int j0, const uint32_t (&v)[16], auto fl_tag) {
                constexpr bool fl = decltype(fl_tag)::value;
                const int g = part * gpw + gi;
                const int s4 = lane & 3;
                const float2 al0 = *reinterpret_cast<const float2*>(s->ep_al[e][gi] + j0 + 2 * s4);
                const float2 al1 = *reinterpret_cast<const float2*>(s->ep_al[e][gi] + j0 + 8 + 2 * s4);
                const float2 zc0 = *reinterpret_cast<const float2*>(s->ep_zc[e][gi] + j0 + 2 * s4);
                const float2 zc1 = *reinterpret_cast<const float2*>(s->ep_zc[e][gi] + j0 + 8 + 2 * s4);
                const float alv[4] = {al0.x, al0.y, al1.x, al1.y}, zcv[4] = {zc0.x, zc0.y, zc1.x, zc1.y};
                [[maybe_unused]] float tv[4] = {0.f, 0.f, 0.f, 0.f};  // asymmetric weights: token sums
                if constexpr (zp) {
                    const float2 t0 = *reinterpret_cast<const float2*>(s->ep_t[e][gi] + j0 + 2 * s4);
                    const float2 t1 = *reinterpret_cast<const float2*>(s->ep_t[e][gi] + j0 + 8 + 2 * s4);
                    tv[0] = t0.x, tv[1] = t0.y, tv[2] = t1.x, tv[3] = t1.y;
                }
                uint32_t pk[4][2];  // [channel k][token pair tp]
#pragma unroll
                for (int k = 0; k < 4; ++k) {
#pragma unroll
                    for (int tp = 0; tp < 2; ++tp) {
                        // two tokens of channel k at once, each lane rounded as the scalar
                        // sequence u = fma(zc, rs, acc), s = alpha * cw, y = fma(u, s, bias)
                        const int i0 = (k >> 1) * 8 + (k & 1) * 2 + 4 * tp;
                        float2 acc2;
                        if constexpr (fl) {
                            acc2 = make_float2(__uint_as_float(v[i0]), __uint_as_float(v[i0 + 1]));
                        } else {
                            acc2 = make_float2(__int2float_rn(int(v[i0])), __int2float_rn(int(v[i0 + 1])));
                        }
                        float2 u2 = ptx::ffma2(make_float2(zcv[2 * tp], zcv[2 * tp + 1]), make_float2(rsf[k], rsf[k]),
                                               acc2);
                        // asymmetric weights: u = fma(zcw, t, u)
                        if constexpr (zp) u2 = ptx::ffma2(make_float2(zcwf[k], zcwf[k]), make_float2(tv[2 * tp], tv[2 * tp + 1]), u2);
                        const float2 s2 = ptx::fmul2(make_float2(alv[2 * tp], alv[2 * tp + 1]), make_float2(cwf[k], cwf[k]));
                        const float2 y2 = ptx::ffma2(u2, s2, make_float2(biasf[k], biasf[k]));
                        const __nv_bfloat162 hb = __floats2bfloat162_rn(y2.x, y2.y);
                        pk[k][tp] = *reinterpret_cast<const uint32_t*>(&hb);
                    }
                }
                // The CTA's last tile stages every box in its own 1 KB of the activation ring,
                // idle once the tile's last MMA has completed, so no box waits for the store
                // of the one before; other tiles share this warp's box.
                const uint32_t stg = stg_base + uint32_t(gi * 2 + (j0 >> 4)) * stg_step;
                if (stg_step == 0 && lane == 0) ptx::bulk_wait_read0();  // the previous box has left the buffer
                __syncwarp();
                {
                    // stored matrix i = lane / 8: (channel block, token block) = (i & 1, i >> 1), plus
                    // two channel blocks for the second store; row k = lane % 8 is token 8 * tb + k
                    // 16-byte chunks placed in the 64-byte swizzle of the output tensor map,
                    // so the eight rows of each stored matrix fall in eight different bank groups
                    const int i = lane >> 3, kr = lane & 7;
                    const int t = (i >> 1) * 8 + kr, sw = (t >> 1) & 3;
                    const uint32_t row = stg + uint32_t(t * 64);
                    ptx::stmatrix_x4_trans(row + uint32_t((((i & 1)) ^ sw) << 4), pk[0][0], pk[1][0], pk[0][1], pk[1][1]);
                    ptx::stmatrix_x4_trans(row + uint32_t(((2 + (i & 1)) ^ sw) << 4), pk[2][0], pk[3][0], pk[2][1],
                                           pk[3][1]);
                }
                ptx::fence_proxy_async_smem();
                __syncwarp();
                const int xc = tc.ch0 + q * 32, yt = tc.tok0 + g * 32 + j0;
                if (lane == 0 && xc < a.N && yt < a.M) {
                    ptx::tma_store_2d(&tm_y, stg, xc, yt);
                    ptx::bulk_commit();
                }
                if (a.acc) {  // int32 accumulators (a debugging output): plain stores
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int nk = tc.ch0 + q * 32 + (lane >> 2) + 8 * k;
#pragma unroll
                        for (int tp = 0; tp < 2; ++tp)
#pragma unroll
                            for (int ee = 0; ee < 2; ++ee) {
                                const int tok = yt + 8 * tp + 2 * s4 + ee;
                                const uint32_t raw = v[(k >> 1) * 8 + (k & 1) * 2 + 4 * tp + ee];
                                if (tok < a.M && nk < a.N)
                                    a.acc[int64_t(tok) * a.N + nk] = fl ? __float2int_rn(__uint_as_float(raw)) : int(raw);
                            }
                    }
                }
            };

            // Multi-chunk tiles keep their int32 running sums in this warp's slice of the
            // per-CTA scratch (32 channels x 32 * MAX_GPW tokens); each value is only
            // re-read by the thread that wrote it.
            // (helper converter warps, e >= EPI_WARPS, only run single-chunk tiles and never touch it)
            int32_t* my_part = a.part + (int64_t(blockIdx.x) * EPI_WARPS + (e < EPI_WARPS ? e : 0)) * (MAX_GPW * 32 * 32) + lane;
            for (int c = 0; c < nchunks; ++c, ++cc) {
                const int buf = cc % NACC;
                if (!wt.wait(&s->accfull[buf], (cc / NACC) & 1)) {
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint32_t acc_base = lane_base + C::ACC_COL + buf * BT;
                const bool last = c == nchunks - 1;
                // the last chunk of the CTA's last tile: no activation stage is loaded or read
                // again (its last MMA has completed), so the ring can hold the output boxes
                if (!CONV && last && w + units >= works) {
                    stg_base = ptx::smem_u32(&s->x[0][0]) + uint32_t(e * C::PIECES) * 1024u;
                    stg_step = 1024;
                    ptx::fence_proxy_async_smem();  // after the ring's TMA writes and MMA reads
                }
#pragma unroll 1
                for (int gi = 0; gi < gpw; ++gi) {
                    const int g = part * gpw + gi;
                    if (g >= C::GROUPS) break;
                    const bool all_tok = all_tok_g[gi];
#pragma unroll 1
                    for (int h = 0; h < 2; ++h) {
                        uint32_t v[16];
                        const bool frag = !CONV && p.splits == 1;  // linear, not split: fragment layout
                        if (frag) {
                            // lanes q*32 .. +15 and +16 .. +31 of the quadrant, 16 columns each
                            ptx::tmem_ld16x256b_x2(acc_base + g * 32 + h * 16, v);
                            ptx::tmem_ld16x256b_x2(acc_base + (16u << 16) + g * 32 + h * 16, v + 8);
                        } else {
                            ptx::tmem_ld16(acc_base + g * 32 + h * 16, v);
                        }
                        ptx::tmem_wait_ld();
                        if (nchunks > 1) {
                            int32_t* pp = my_part + (gi * 32 + h * 16) * 32;
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                if (LR && last) {
                                    // the last chunk holds the low-rank block's fraction: keep it
                                    v[j] = __float_as_uint(__fadd_rn(__int2float_rn(pp[j * 32]), __uint_as_float(v[j])));
                                    continue;
                                }
                                int x = __float2int_rn(__uint_as_float(v[j]));
                                if (c > 0) x += pp[j * 32];
                                if (last) v[j] = uint32_t(x);
                                else pp[j * 32] = x;
                            }
                        }
                        if (last && p.splits > 1) {
                            // exact int32 partial sums of this K slice, one coalesced
                            // 128-byte row per token
                            if (n_ok) {
                                int32_t* po = p.split_out + int64_t(wk.slice) * a.M * a.N + n;
#pragma unroll
                                for (int j = 0; j < 16; ++j) {
                                    const int tok = s->ep_tok[e][gi][h * 16 + j];
                                    if (tok >= 0)
                                        po[int64_t(tok) * a.N] =
                                            nchunks == 1 ? __float2int_rn(__uint_as_float(v[j])) : int(v[j]);
                                }
                            }
                        } else if (last) {
                            if constexpr (!CONV) {
                                if (nchunks == 1 || LR) finish16f(gi, h * 16, v, std::true_type{});
                                else finish16f(gi, h * 16, v, std::false_type{});
                            } else {
                                if (nchunks == 1) finish16(gi, h * 16, v, std::true_type{}, all_tok);
                                else finish16(gi, h * 16, v, std::false_type{}, all_tok);
                            }
                        }
                    }
                }
                ptx::tc_fence_before();
                __syncwarp();
                // (helper converter warps only join the tile's single chunk: nothing waits for them)
                if (lane == 0 && e < EPI_WARPS) ptx::mbar_arrive(ptx::smem_u32(&s->accempty[buf]));
            }
        }
    }

    // every thread of the CTA, the epilogue's last tensor-memory reads included, is past
    // its role before tensor memory is released (a barrier that counts threads: see
    // ptx::cta_sync)
    ptx::cta_sync();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, TMEM_COLS);
    }
    // epilogue TMA stores complete before the CTA exits
    if (!CONV && lane == 0 &&
        ((warp >= EPI_WARP0 && warp < EPI_WARP0 + EPI_WARPS) || (helpers && warp >= 2 && warp < EPI_WARP0)))
        ptx::bulk_wait0();
}

// Split-K second half: adds the slices' exact int32 partial sums in slice
// order and applies the same fused epilogue as the contraction kernel, four
// channels per thread (16-byte loads, 8-byte bf16 stores).
__global__ void __launch_bounds__(256) splitk_epilogue_kernel(const GemmArgs a, const int32_t* __restrict__ parts,
                                                              int S) {
    ptx::grid_dependency_wait();
    const uint32_t gbits = resolve_group_bits(a);
    if (gbits == 0) return;
    const int b = int(gbits & 15u);
    const int N4 = a.N / 4;
    const int64_t total = int64_t(a.M) * N4;
    const int32_t* ts_b = a.Cin ? a.ts + int64_t(b - kBMin) * a.N * 9 : nullptr;
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < total; i += int64_t(gridDim.x) * blockDim.x) {
        const int m = int(i / N4);
        const int n = int(i - int64_t(m) * N4) * 4;
        int4 acc = make_int4(0, 0, 0, 0);
        for (int sl = 0; sl < S; ++sl) {
            const int4 v = __ldcg(reinterpret_cast<const int4*>(parts + (int64_t(sl) * a.M + m) * a.N + n));
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        const float al = a.per_tensor ? a.alpha[0] : a.alpha[m];
        const float zc = a.per_tensor ? a.zc[0] : a.zc[m];
        const bool zp = a.code_sums != nullptr;  // asymmetric weights
        const float t = !zp ? 0.f
                            : a.Cin ? conv_token_zero_sum(a.code_sums, m, a.H, a.W, a.Cin, zc)
                                    : token_zero_sum(a.code_sums[m], a.K, zc);
        int tap = 0x1FF;
        if (a.Cin) {
            const int ww = m % a.W, hh = (m / a.W) % a.H;
            tap = 0;
#pragma unroll
            for (int dh = 0; dh < 3; ++dh)
#pragma unroll
                for (int dw = 0; dw < 3; ++dw) {
                    const int ih = hh + dh - 1, iw = ww + dw - 1;
                    if (ih >= 0 && ih < a.H && iw >= 0 && iw < a.W) tap |= 1 << (dh * 3 + dw);
                }
        }
        const int accs[4] = {acc.x, acc.y, acc.z, acc.w};
        float y[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            float rsum;
            if (a.Cin) {
                rsum = 0.f;
#pragma unroll
                for (int k9 = 0; k9 < 9; ++k9)
                    rsum = __fadd_rn(rsum, (tap >> k9) & 1 ? __int2float_rn(ts_b[int64_t(n + q) * 9 + k9]) : 0.f);
            } else {
                // the four channels n..n+3 belong to one member (group_n % 8 == 0)
                rsum = __int2float_rn(a.rs[int64_t(channel_bits(a, gbits, n) - kBMin) * a.N + n + q]);
            }
            float u = __fmaf_rn(zc, rsum, __int2float_rn(accs[q]));
            if (zp) u = __fmaf_rn(a.zcw[n + q], t, u);
            y[q] = __fmaf_rn(u, __fmul_rn(al, a.cw[n + q]), a.bias[n + q]);
        }
        const __nv_bfloat162 h0 = __floats2bfloat162_rn(y[0], y[1]);
        const __nv_bfloat162 h1 = __floats2bfloat162_rn(y[2], y[3]);
        uint2 pk;
        pk.x = *reinterpret_cast<const uint32_t*>(&h0);
        pk.y = *reinterpret_cast<const uint32_t*>(&h1);
        *reinterpret_cast<uint2*>(a.y + int64_t(m) * a.N + n) = pk;
        if (a.acc) *reinterpret_cast<int4*>(a.acc + int64_t(m) * a.N + n) = acc;
    }
    ptx::grid_launch_dependents();
}

}  // namespace

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

size_t gemm_tc_part_bytes(int num_sms) { return size_t(num_sms) * MAX_EPI_WARPS * MAX_GPW * 32 * 32 * sizeof(int32_t); }

namespace {

// Token tiles of a launch with BT-token tiles (conv: boxes of bhx rows x 2^bwl
// pixels, 2^bwl dividing BT).
struct TokTiling {
    int64_t tiles;
    int bw_log2, bhx, tiles_w, tiles_h;
};
TokTiling token_tiling(const GemmArgs& a, int BT) {
    TokTiling t{};
    if (a.Cin) {
        int bwl = 0;
        while ((1 << bwl) < a.W && (1 << bwl) < 64) ++bwl;
        t.bw_log2 = bwl;
        t.bhx = BT >> bwl;
        const int bw = 1 << bwl;
        t.tiles_w = (a.W + bw - 1) / bw;
        t.tiles_h = (a.H + t.bhx - 1) / t.bhx;
        t.tiles = int64_t(a.B) * t.tiles_h * t.tiles_w;
    } else {
        t.tiles = (a.M + BT - 1) / BT;
    }
    return t;
}

}  // namespace

TcPlan plan_gemm_tc(int M, int N, int K, int B, int H, int W, int Cin, int num_sms, int64_t split_cap) {
    TcPlan p{};
    GemmArgs a{};
    a.M = M;
    a.N = N;
    a.K = K;
    a.B = B;
    a.H = H;
    a.W = W;
    a.Cin = Cin;
    p.bch = BCH;
    p.tiles_ch = (N + BCH - 1) / BCH;
    p.splits = 1;
    if (Cin && Cin % 64) {
        p.why = "convolution needs Cin % 64 == 0";
        return p;
    }
    if (M <= 0 || N <= 0) return p;
    // The wide single-tile configuration when it covers the output in one wave
    // of CTAs and the standard one would need more than one; the narrow one when
    // the standard tiles would leave most SMs idle.
    const int64_t std_tiles = p.tiles_ch * token_tiling(a, CfgStd::BT).tiles;
    const int64_t wide_tiles = p.tiles_ch * token_tiling(a, CfgWide::BT).tiles;
    if (std_tiles > num_sms && wide_tiles <= num_sms) {
        p.bt = CfgWide::BT;
        p.nacc = CfgWide::NACC;
    } else if (std_tiles * 2 <= num_sms) {
        p.bt = CfgNarrow::BT;
        p.nacc = CfgNarrow::NACC;
    } else {
        p.bt = CfgStd::BT;
        p.nacc = CfgStd::NACC;
    }
    const TokTiling tt = token_tiling(a, p.bt);  // conv: 2^bw_log2 divides BT (192 = 64 * 3, 256)
    p.tiles_tok = tt.tiles;
    p.bw_log2 = tt.bw_log2;
    p.bhx = tt.bhx;
    p.tiles_w = tt.tiles_w;
    p.tiles_h = tt.tiles_h;
    const int64_t tiles = int64_t(p.tiles_ch) * p.tiles_tok;
    if (tiles > 0x7FFFFFFF) {
        p.why = "too many tiles";
        return p;
    }
    // Split K when the tiles alone would leave most SMs idle and each slice keeps
    // at least 8 K blocks: a tile's fixed latency (pipeline fill, epilogue) is
    // not reduced by splitting, only its K loop is.
    if (p.nacc == 2 && split_cap > 0 && tiles * 2 <= num_sms) {
        const int KT = (K + BK - 1) / BK;
        int64_t S = num_sms / tiles;
        S = S < KT / 8 ? S : KT / 8;
        static const int max_splits = [] {
            const char* v = getenv("TASQ_TC_MAX_SPLITS");  // tuning knob; default 16
            return v ? atoi(v) : 16;
        }();
        S = S < max_splits ? S : max_splits;
        const int64_t fit = split_cap / (int64_t(M) * N);
        S = S < fit ? S : fit;
        if (S >= 2) p.splits = int(S);
    }
    const int64_t works = tiles * p.splits;
    p.grid = int(works < num_sms ? works : num_sms);
    if (p.splits > 1) {
        // the reduction reads 4 channels per thread, 256 threads per block
        const int64_t blocks = (int64_t(M) * (N / 4) + 255) / 256;
        p.reduce_grid = int(blocks < 8 * int64_t(num_sms) ? blocks : 8 * int64_t(num_sms));
    }
    return p;
}

namespace {

template <class C>
cudaError_t launch_cfg(const GemmArgs& a, const TcPlan& plan, cudaStream_t st, const char** why, int* kernels) {
    constexpr int BTOK = C::BT;
    auto encode = get_encode();
    if (!encode) {
        *why = "cuTensorMapEncodeTiled is unavailable";
        return cudaSuccess;
    }
    TcParams p{};
    p.a = a;
    p.conv = a.Cin != 0;
    p.tiles_ch = (a.N + BCH - 1) / BCH;
    CUtensorMap tm_x, tm_w, tm_y, tm_x8, tm_u;
    CUresult r;
    p.tiles_tok = int(plan.tiles_tok);
    if (p.conv) {
        p.bw_log2 = plan.bw_log2;
        p.bhx = plan.bhx;
        const int bw = 1 << plan.bw_log2;
        p.tiles_w = plan.tiles_w;
        p.tiles_h = plan.tiles_h;
        cuuint64_t dims[4] = {cuuint64_t(a.Cin), cuuint64_t(a.W), cuuint64_t(a.H), cuuint64_t(a.B)};
        cuuint64_t strides[3] = {cuuint64_t(a.Cin) * 2, cuuint64_t(a.W) * a.Cin * 2, cuuint64_t(a.H) * a.W * a.Cin * 2};
        cuuint32_t box[4] = {XK, cuuint32_t(bw), cuuint32_t(p.bhx), 1};
        cuuint32_t es[4] = {1, 1, 1, 1};
        r = encode(&tm_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(a.x), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else {
        cuuint64_t dims[2] = {cuuint64_t(a.K), cuuint64_t(a.M)};
        cuuint64_t strides[1] = {cuuint64_t(a.K) * 2};
        cuuint32_t box[2] = {XK, cuuint32_t(BTOK)};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_x, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(a.x), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    if (r != CUDA_SUCCESS) {
        *why = "activation tensor map rejected";
        return cudaSuccess;
    }
    const bool f8 = !p.conv && a.x8 != nullptr;
    if (f8) {
        // the same codes as e5m2 bytes [M][K]: 128 codes of a token are one
        // 128-byte swizzle atom
        cuuint64_t dims[2] = {cuuint64_t(a.K), cuuint64_t(a.M)};
        cuuint64_t strides[1] = {cuuint64_t(a.K)};
        cuuint32_t box[2] = {BK, cuuint32_t(BTOK)};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_x8, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(a.x8), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "e5m2 activation tensor map rejected";
            return cudaSuccess;
        }
    } else {
        tm_x8 = tm_x;  // unused
    }
    if (a.lr_rank) {
        // the low-rank block's activations: u' [M][64] fp16, one 64-wide box per stage half
        cuuint64_t dims[2] = {cuuint64_t(kLowRankCols), cuuint64_t(a.M)};
        cuuint64_t strides[1] = {cuuint64_t(kLowRankCols) * 2};
        cuuint32_t box[2] = {XK, cuuint32_t(BTOK)};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_u, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<uint16_t*>(a.lr_u), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "low-rank tensor map rejected";
            return cudaSuccess;
        }
    } else {
        tm_u = tm_x;  // unused
    }
    {
        cuuint64_t dims[2] = {cuuint64_t(a.K), cuuint64_t(a.N)};
        cuuint64_t strides[1] = {cuuint64_t(a.K)};
        cuuint32_t box[2] = {BK, BCH};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_w, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<int8_t*>(a.w), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "weight tensor map rejected";
            return cudaSuccess;
        }
    }
    if (!p.conv) {
        // output y [M][N] bf16: the epilogue stores [16 tokens][32 channels] boxes
        cuuint64_t dims[2] = {cuuint64_t(a.N), cuuint64_t(a.M)};
        cuuint64_t strides[1] = {cuuint64_t(a.N) * 2};
        cuuint32_t box[2] = {32, 16};
        cuuint32_t es[2] = {1, 1};
        r = encode(&tm_y, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, a.y, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                   CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) {
            *why = "output tensor map rejected";
            return cudaSuccess;
        }
    } else {
        tm_y = tm_x;  // unused by the convolution instantiation
    }
    p.splits = plan.splits;
    p.split_out = plan.splits > 1 ? a.split_buf : nullptr;
    const int units = plan.grid;
    static const bool verbose = getenv("TASQ_TC_VERBOSE") != nullptr;
    if (verbose)
        fprintf(stderr, "tasq tc: M=%d N=%d K=%d BT=%d tiles=%lld splits=%d grid=%d\n", a.M, a.N, a.K, BTOK,
                (long long)p.tiles_ch * p.tiles_tok, p.splits, units);
    const int smem = smem_bytes<C>();
    auto kernel = [&] {
        // the eight-converter tiles only serve linear layers with e5m2 codes; the
        // low-rank branch only symmetric linear layers
        if constexpr (C::CONV_WARPS == 8)
            return a.d_layers    ? gemm_tc_kernel<false, false, C, true, false, true>
                   : a.lr_rank   ? gemm_tc_kernel<false, false, C, true, true>
                   : a.code_sums ? gemm_tc_kernel<false, true, C, true>
                                 : gemm_tc_kernel<false, false, C, true>;
        else
            return p.conv        ? (a.code_sums ? gemm_tc_kernel<true, true, C> : gemm_tc_kernel<true, false, C>)
                   : a.d_layers ? (f8 ? gemm_tc_kernel<false, false, C, true, false, true>
                                      : gemm_tc_kernel<false, false, C, false, false, true>)
                   : a.lr_rank ? (f8 ? gemm_tc_kernel<false, false, C, true, true> : gemm_tc_kernel<false, false, C, false, true>)
                   : f8        ? (a.code_sums ? gemm_tc_kernel<false, true, C, true> : gemm_tc_kernel<false, false, C, true>)
                               : (a.code_sums ? gemm_tc_kernel<false, true, C> : gemm_tc_kernel<false, false, C>);
    }();
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    // programmatic dependent launch: the grid may start while the previous
    // kernel drains; it waits (griddepcontrol.wait) before reading inputs
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(units);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kernel, p, tm_x, tm_w, tm_y, tm_x8, tm_u);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e == cudaSuccess) *kernels = 1;
    if (e == cudaSuccess && p.splits > 1) {
        cudaLaunchConfig_t rc{};
        rc.gridDim = dim3(unsigned(plan.reduce_grid));
        rc.blockDim = dim3(256);
        rc.stream = st;
        rc.attrs = attr;  // programmatic dependent launch
        rc.numAttrs = 1;
        e = cudaLaunchKernelEx(&rc, splitk_epilogue_kernel, a, static_cast<const int32_t*>(p.split_out), p.splits);
        if (e == cudaSuccess) e = cudaGetLastError();
        if (e == cudaSuccess) *kernels = 2;
    }
    if (e == cudaErrorLaunchOutOfResources) {
        // report what the kernel asked for, to make the failure actionable
        static char msg[256];
        cudaFuncAttributes fa{};
        cudaFuncGetAttributes(&fa, kernel);
        snprintf(msg, sizeof msg,
                 "launch out of resources: %d threads x %d registers, %d B dynamic smem (kernel max %d threads, "
                 "%zu B static smem)",
                 THREADS, fa.numRegs, smem, fa.maxThreadsPerBlock, fa.sharedSizeBytes);
        *why = msg;
        return cudaSuccess;
    }
    return e;
}

}  // namespace

cudaError_t launch_gemm_tc(const GemmArgs& a, int num_sms, cudaStream_t st, const char** why, int* kernels) {
    *why = nullptr;
    *kernels = 0;
    if (!a.part) {
        *why = "no accumulator scratch";
        return cudaSuccess;
    }
    if (a.M == 0 || a.N == 0) return cudaSuccess;
    // (the split-K reduction has no low-rank term and reads at most kMaxGroups members'
    // precisions from the arguments: such launches stay unsplit)
    const TcPlan plan = plan_gemm_tc(a.M, a.N, a.K, a.B, a.H, a.W, a.Cin, num_sms,
                                     a.split_buf && !a.lr_rank && !a.d_layers ? a.split_cap : 0);
    if (plan.why) {
        *why = plan.why;
        return cudaSuccess;
    }
    const bool x8 = a.Cin == 0 && a.x8 != nullptr;  // a linear layer with e5m2 codes
    if (plan.bt == CfgWide::BT) return launch_cfg<CfgWide>(a, plan, st, why, kernels);
    if (plan.bt == CfgNarrow::BT)
        return x8 ? launch_cfg<CfgNarrowF8>(a, plan, st, why, kernels) : launch_cfg<CfgNarrow>(a, plan, st, why, kernels);
    // 192-token tiles: eight converters pay off once the K loop is long enough to
    // hide their longer (eight-warp) epilogue (measured: 4096 x 4096 x 4096 at b = 4
    // 66.6 against 72.7 us; 4096 x 3456 x 1152 27.8 against 26.1 us)
    if (x8 && a.K >= 2048) return launch_cfg<CfgStdF8>(a, plan, st, why, kernels);
    return launch_cfg<CfgStd>(a, plan, st, why, kernels);
}

}  // namespace tasq
