/*
 * tasq.h -- C ABI of the GB300 (sm_103a) masked-W8A8 library for TASQ
 * (Temporal-Adaptive Bit Sparsification Quantization, arXiv 2608.03057).
 *
 * What the library computes.  Each quantized layer keeps ONE shared 8-bit
 * weight buffer (Sec. 3.1, Eq. truncquant; App. F.1).  At denoising stage s
 * the layer runs at an operating precision b = table[layer][s] in 2..8 (the
 * bit-allocation map of App. F.1): the 8 - b least-significant planes of the
 * stored code are dropped (Eqs. lsb_extraction, lsb_masking, hw_rightshift,
 * hw_multi_lsb) and the truncated weight multiplies the quantized activations
 * (Eq. qalora, Y = Q(X) Q(W)), with the dequantization of App. A.1 folded
 * into an epilogue that writes bf16.
 *
 * Conventions shared by every call:
 *  - Pointers named d_* are DEVICE pointers on the context's device; h_* are
 *    host pointers.  The caller owns every buffer it passes; the library never
 *    keeps a caller pointer beyond the call, except d_stage of
 *    tasq_set_stage_device (documented there).
 *  - Calls that take a `stream` only enqueue work on that stream (a
 *    cudaStream_t; NULL is the legacy default stream).  They do not allocate,
 *    do not synchronize, and return as soon as the work is queued.  Calls
 *    without a stream are set-up calls and may allocate or synchronize, as
 *    documented on each.
 *  - The context's device must be the current CUDA device of the calling
 *    thread; a mismatch returns TASQ_ERR_INVALID_ARG.
 *  - Every call returns TASQ_OK (0) or an error code; tasq_last_error() then
 *    describes the failure.  Arguments are validated on the host before
 *    anything is launched: an invalid call launches nothing.
 *  - Errors that only the device can see (an out-of-range stage read from
 *    device memory, a packed buffer that does not match N/K, a pipeline wait
 *    that ran past its time limit) are recorded in a device status word that
 *    tasq_device_status() reads; the kernel then returns early without
 *    trapping, and the CUDA context stays usable.
 *  - A context may be used from one host thread at a time.  Two kinds of
 *    call use per-context device scratch: per-tensor activation quantization
 *    (a 16-byte reduction) and tensor-core contractions whose certificate
 *    splits K into several chunks (int32 running sums, 96 KB per SM).  Calls
 *    of either kind on different streams of one context must not overlap;
 *    use one context per concurrent stream.  Split-K contractions (few
 *    output tiles, long K) also use the context's 32 MB of partial sums.
 *  - Kernels are launched with programmatic dependent launch: a contraction
 *    or quantization may start while the previous kernel in the stream
 *    drains.  Each one waits for that kernel before it reads the
 *    activations, codes or scales, or writes any output.  The contraction
 *    reads the stage (argument or device int), the bit table and the packed
 *    buffer before that wait, so write those with work that precedes the
 *    previous kernel (as the library's own calls do), not with the kernel
 *    launched immediately before the contraction.  The quantization only
 *    prefetches its input into L2 before the wait, which is safe whoever
 *    writes it.
 *
 * Data layouts: row-major, innermost index last.  Activations of a linear
 * layer are [M][K] (M tokens); of a conv, NHWC [B][H][W][Cin].  Weights are
 * [N][K] (linear) or [Cout][3][3][Cin] = [N][9*Cin] (conv).  Outputs are bf16
 * [M][N] (linear) or NHWC [B][H][W][Cout] (conv), as uint16_t bit patterns.
 * Shape rules: K % 16 == 0 and N % 8 == 0 (conv: Cin % 16 == 0); M >= 0 may
 * be anything (M == 0 is a no-op).  Every device pointer must be 16-byte
 * aligned.
 */
#ifndef TASQ_H
#define TASQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TASQ_ABI_VERSION 5

/* Return codes. */
enum {
    TASQ_OK = 0,
    TASQ_ERR_INVALID_ARG = 1,    /* bad pointer, range, enum or device */
    TASQ_ERR_UNSUPPORTED = 2,    /* legal but unsupported shape, alignment or mode */
    TASQ_ERR_CUDA = 3,           /* a CUDA runtime call or launch failed */
    TASQ_ERR_DEVICE_TIMEOUT = 4, /* (device status) a pipeline wait ran past its limit */
    TASQ_ERR_DEVICE = 5          /* (device status) a check inside a kernel failed */
};

enum { TASQ_LINEAR = 0, TASQ_CONV3X3 = 1 };               /* layer kinds */
enum { TASQ_F32 = 0, TASQ_BF16 = 1 };                     /* float tensor dtypes */
enum { TASQ_SYMRANGE = 0, TASQ_ASYM = 1 };                /* quantization range */
enum { TASQ_PER_TOKEN = 0, TASQ_PER_TENSOR = 1 };         /* activation granularity */
/* Storage of activation codes s = Q - 2^(n-1): one signed byte, or the same
 * integer held exactly in an IEEE fp16 (the operand type of the tensor-core
 * route; every integer in [-128, 127] is exact in fp16).  TASQ_CODES_F16_E5M2
 * (activation precision n <= 4, |s| <= 8) stores the fp16 codes [M][K] and,
 * right after them, the same codes as OCP e5m2 bytes [M][K] (every integer of
 * magnitude <= 8 has at most three significant bits and is exact in e5m2):
 * 3 * M * K bytes.  With it a linear tensor-core contraction runs its K loop on
 * the 8-bit-float MMA kind (twice the K per instruction) whenever the operating
 * precision is b <= 4, because the masked weight code mask_b(s_w) then has at
 * most three significant bits and is exact in e5m2 too (unsplit launches); for
 * b > 4, split-K launches and convolutions it reads the fp16 codes.  Either way
 * the bound |s| <= 8 lets an exact fp32 chunk run 16 times as long as the one
 * certified for 8-bit codes; codes outside it are outside the format. */
enum { TASQ_CODES_S8 = 0, TASQ_CODES_F16 = 1, TASQ_CODES_F16_E5M2 = 2 };
/* Contraction routes.  TC: tcgen05 MMA on fp16-held integer codes with fp32
 * accumulation in tensor memory, drained to int32 in chunks whose exactness
 * is certified at pack time (needs TASQ_CODES_F16).  MMA_S8: warp-level
 * mma.sync with int8 operands and int32 accumulators (needs TASQ_CODES_S8).
 * AUTO picks the route that matches the code storage. */
enum { TASQ_ROUTE_AUTO = 0, TASQ_ROUTE_TC = 1, TASQ_ROUTE_MMA_S8 = 2 };

typedef struct tasq_ctx_s* tasq_ctx;
typedef void* tasq_stream; /* cudaStream_t */

/* ABI version of the loaded library (TASQ_ABI_VERSION). */
int tasq_version(void);

/* Create a context on CUDA device `device`.  Set-up call: allocates the
 * context's device status word, its reduction scratch, the bit table (room
 * for 65,536 entries), the tensor-core route's accumulator scratch (96 KB per
 * SM: about 14.6 MB on a GB300) and its split-K partial sums (32 MB), and
 * leaves the calling thread's current device unchanged.  *out is NULL on
 * failure. */
int tasq_create(tasq_ctx* out, int device);

/* Destroy a context and free what it allocated.  Synchronizes the device.
 * NULL is ignored. */
void tasq_destroy(tasq_ctx ctx);

/* Text of the last error on this context (valid until the next call on it);
 * with ctx == NULL, the last tasq_create failure of this thread. */
const char* tasq_last_error(tasq_ctx ctx);

/* Device status: synchronizes the device, returns TASQ_OK or the first
 * device-side error code recorded since the last read (TASQ_ERR_DEVICE_TIMEOUT,
 * TASQ_ERR_DEVICE) in *out, then clears it.  Set-up call. */
int tasq_device_status(tasq_ctx ctx, int* out);

/* Number of kernels that tasq_quant_act, tasq_masked_gemm and
 * tasq_masked_conv3x3 have enqueued on this context since it was created
 * (a contraction enqueues one, or two when it splits K; per-tensor
 * quantization enqueues two).  Host-side count, no synchronization; a launch
 * captured into a CUDA graph counts once, at capture.  Diagnostic only (the
 * paper has no counterpart). */
int tasq_kernel_count(tasq_ctx ctx, unsigned long long* out);

/* Route used by tasq_masked_gemm / tasq_masked_conv3x3 (TASQ_ROUTE_*). */
int tasq_set_route(tasq_ctx ctx, int route);

/* Time limit of every pipeline wait inside the kernels, in nanoseconds
 * (default 2e9; 0 restores the default).  A wait that runs past it records
 * TASQ_ERR_DEVICE_TIMEOUT in the device status and its kernel returns. */
int tasq_set_timeout_ns(tasq_ctx ctx, uint64_t ns);

/* Failure-detection self test: launches one block that waits on a barrier
 * nothing ever arrives at, bounded by `timeout_ns`.  The wait gives up,
 * records TASQ_ERR_DEVICE_TIMEOUT in the device status and the kernel
 * returns, leaving the context usable.  Enqueue call. */
int tasq_selftest_timeout(tasq_ctx ctx, uint64_t timeout_ns, tasq_stream stream);

/* Arithmetic self test of the activation quantizer: the quantizer divides
 * x / alpha with a reciprocal computed once per group followed by two exact
 * remainder corrections (Markstein's method) instead of a hardware division
 * per element.  For every pair (d_x[i], d_a[j]), i < nx, j < na, this adds 1
 * to *d_mismatches (caller-zeroed uint64 on the device) when that quotient's
 * bit pattern differs from IEEE round-to-nearest division.  Enqueue call. */
int tasq_selftest_quotients(tasq_ctx ctx, const float* d_x, int nx, const float* d_a, int na,
                            unsigned long long* d_mismatches, tasq_stream stream);

/*
 * Weight quantization, App. A.1.1 (Eqs. weight_quant, weight_scale,
 * weight_dequant), per output channel, with the range taken symmetric,
 * [-max|w|, +max|w|] (so alpha = max|w| / 128 and z = 128):
 *   Q = clamp(floor(w / alpha + z), 0, 255),  stored s_w = Q - 128 (int8),
 *   c_w = (256/255) * alpha   so that   w_hat = c_w * s_w.
 * fp32 operation order (each step rounds to nearest even): alpha =
 * (hi - lo) / 256, z = -lo / alpha, Q = floor((w / alpha) + z),
 * c_w = alpha * (256/255).  An all-zero channel gets alpha = 1, z = 128.
 * d_w: [N][K] of `dtype` (TASQ_F32 or TASQ_BF16).  Outputs d_sw [N][K] int8,
 * d_cw [N] fp32, d_alpha [N] fp32 (may be NULL).  Enqueue call.
 */
int tasq_quant_weights(tasq_ctx ctx, const void* d_w, int dtype, int N, int K, int8_t* d_sw, float* d_cw,
                       float* d_alpha, tasq_stream stream);

/*
 * Weight quantization with a weight zero point: App. A.1.1 (Eqs. weight_quant,
 * weight_scale, weight_dequant) applied as written, on each output channel's
 * true range [min(w), max(w)]:
 *   alpha = (max - min) / 256,  z = -min / alpha  (real valued),
 *   Q = clamp(floor(w / alpha + z), 0, 255),  stored s_w = Q - 128 (int8),
 *   c_w = (256/255) * alpha,  zcw = 128 - z,
 * so that w_hat = c_w * (Q - z) = c_w * (s_w + zcw), and at operating
 * precision b, w_hat_b = c_w * (mask_b(s_w) + zcw).  Same fp32 operation order
 * as tasq_quant_weights, then zcw = 128 - z rounded once.  A constant channel
 * gets alpha = 1, z = -min.  Outputs d_sw [N][K] int8, d_cw [N], d_zcw [N]
 * fp32, d_alpha [N] (may be NULL).  Pack the result with
 * tasq_pack_weights_zp.  Enqueue call.
 */
int tasq_quant_weights_asym(tasq_ctx ctx, const void* d_w, int dtype, int N, int K, int8_t* d_sw, float* d_cw,
                            float* d_zcw, float* d_alpha, tasq_stream stream);

/*
 * Bytes of the packed form of one layer (see tasq_pack_weights), for
 * kind TASQ_LINEAR (K = in features) or TASQ_CONV3X3 (K = 9*Cin).
 * Returns 0 for invalid shapes.
 */
size_t tasq_packed_bytes(int kind, int N, int K);

/*
 * Pack one layer's stored 8-bit weights once (App. F.1: the stored buffer is
 * not copied per stage).  d_packed (caller-allocated, tasq_packed_bytes
 * bytes, 256-byte aligned) receives:
 *   - a copy of d_sw [N][K] (the shared buffer every stage reads),
 *   - c_w [N] and bias [N] (zeros when d_bias is NULL),
 *   - for each b in 2..8 the row sums rs_b[n] = sum_k mask_b(s_w[n][k])
 *     (they carry the activation zero point through the integer sum), and
 *     for a conv the per-tap sums of the same,
 *   - for each b the exactness certificate of the TC route: the longest run
 *     of 64-wide K blocks over which 128 * sum |mask_b(s_w[n][k])| <= 2^24
 *     for every channel n, so that fp32 partial sums of int8 x int8 products
 *     stay exact integers (|s_x| <= 128).
 * mask_b(v) drops the 8-b low planes of the unsigned code v + 128
 * (Eq. hw_rightshift); on the signed byte this is v & (0xFF << (8-b)).
 * kind: TASQ_LINEAR (K = in features, Cin ignored) or TASQ_CONV3X3
 * (K = 9*Cin, weights ordered (kh, kw, cin)).  Enqueue call.
 */
int tasq_pack_weights(tasq_ctx ctx, int kind, const int8_t* d_sw, const float* d_cw, const float* d_bias, int N,
                      int K, int Cin, void* d_packed, tasq_stream stream);

/*
 * tasq_pack_weights for a layer quantized with a weight zero point
 * (tasq_quant_weights_asym; a conv's weights as rows [Cout][9*Cin]): also
 * stores zcw [N] and marks the buffer, so that the contraction must be given
 * the activations' code sums (tasq_masked_gemm_zp, tasq_masked_conv3x3_zp).
 * tasq_masked_gemm / tasq_masked_conv3x3 on such a buffer record
 * TASQ_ERR_DEVICE and write nothing.  Same buffer size (tasq_packed_bytes).
 * Other arguments as tasq_pack_weights.  Enqueue call.
 */
int tasq_pack_weights_zp(tasq_ctx ctx, int kind, const int8_t* d_sw, const float* d_cw, const float* d_zcw,
                         const float* d_bias, int N, int K, int Cin, void* d_packed, tasq_stream stream);

/*
 * Bit-allocation map (App. F.1): h_bits [L][S] uint8, each value in 2..8,
 * copied into device memory owned by the context.  Set-up call: validates
 * every entry first, synchronizes the device, then copies synchronously.
 * The context creates its table with room for 65,536 entries; the kernels
 * read L and S from the device copy, not from their launch arguments, so a
 * CUDA graph captured before this call runs the new schedule when replayed
 * (a captured call whose layer or stage falls outside the new L x S records
 * TASQ_ERR_DEVICE and writes nothing).  Only a schedule with more than
 * 65,536 entries moves the table to a new buffer; graphs captured before
 * that call keep reading the old buffer, which stays allocated, unchanged,
 * until tasq_destroy, and must be captured again to see the new schedule.
 * Changing stage afterwards needs no host work: it is an argument of the
 * next call, or a device int (tasq_set_stage_device).
 */
int tasq_set_schedule(tasq_ctx ctx, const uint8_t* h_bits, int L, int S);

/*
 * Optional device-resident stage: with d_stage set, a call whose `stage`
 * argument is -1 reads the stage from *d_stage when its kernel runs, so one
 * captured CUDA graph serves every stage.  The context keeps the pointer
 * until it is replaced or cleared (NULL); the caller keeps it alive.
 */
int tasq_set_stage_device(tasq_ctx ctx, const int32_t* d_stage);

/*
 * Activation quantization, App. A.1.2 (Eqs. act_quant, act_scale):
 *   alpha = (max - min) / (2^n - 1),  z = -min / alpha,
 *   Q = clamp(round_half_even(x / alpha + z), 0, 2^n - 1),
 * stored as the signed code s = Q - 2^(n-1), with zc = 2^(n-1) - z so that
 * x_hat = alpha * (Q - z) = alpha * (s + zc).
 * fp32 order (each step rounds to nearest even): alpha = (hi - lo) / (2^n-1),
 * z = -lo / alpha, u = (x / alpha) + z, Q = rint(u), zc = 2^(n-1) - z.
 * A constant group gets alpha = 1 and z = 2^(n-1) (SYMRANGE) or -min (ASYM).
 * mode: TASQ_SYMRANGE ([lo, hi] = [-max|x|, max|x|]) or TASQ_ASYM (min, max).
 * gran: TASQ_PER_TOKEN (one alpha/zc per row of d_x [M][K]) or
 * TASQ_PER_TENSOR (one for the whole tensor; d_x may then be any [M][K] view
 * of a contiguous tensor, e.g. NHWC with M = B*H*W, K = Cin).
 * n_bits in 2..8.  d_x: [M][K] of `dtype`; d_codes: [M][K] int8 or fp16 per
 * code_fmt; d_alpha, d_zc: [M] (per token) or [1] (per tensor) fp32.
 * Enqueue call (per tensor: two kernels and a 16-byte memset).
 */
int tasq_quant_act(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, int n_bits, int mode, int gran,
                   void* d_codes, int code_fmt, float* d_alpha, float* d_zc, tasq_stream stream);

/*
 * tasq_quant_act that also writes d_code_sums [M] int32, the sum over k of
 * the stored codes s[m][k] of each row of d_x (exact; per tensor the rows are
 * still summed one by one: for NHWC activations, one sum per pixel).  The
 * four-term epilogue of asymmetric weights needs it (tasq_masked_gemm_zp,
 * tasq_masked_conv3x3_zp).  Enqueue call (per tensor: one more kernel).
 */
int tasq_quant_act_sums(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, int n_bits, int mode, int gran,
                        void* d_codes, int code_fmt, float* d_alpha, float* d_zc, int32_t* d_code_sums,
                        tasq_stream stream);

/*
 * Masked linear layer (Eq. qalora with the Temporal-Spatial LSB mask of
 * Eq. lsb_masking at operating precision b = table[layer][stage]):
 *   acc[m][n] = sum_k s_x[m][k] * mask_b(s_w[n][k])            (exact int32)
 * (exact whenever the sum fits in int32, which |s| <= 128 guarantees for
 * K <= 131072; past that, adversarial codes could wrap it)
 *   u = fma(zc[m], float(rs_b[n]), float(acc)),  s = alpha[m] * c_w[n],
 *   y[m][n] = bf16(fma(u, s, bias[n]))
 * with every fp32 operation (and each fused multiply-add) rounded once to
 * nearest even, in that order; y = alpha*c_w*(acc + zc*rs_b) + bias.
 * stage: 0..S-1, or -1 to read it from the device int of
 * tasq_set_stage_device.  d_codes: [M][K] activation codes (code_fmt);
 * d_alpha/d_zc: [M] per-token scales from tasq_quant_act.  d_packed: from
 * tasq_pack_weights with kind TASQ_LINEAR and the same N, K.  d_y: [M][N]
 * bf16 bits.  d_acc: [M][N] int32, or NULL (then acc is not written).
 * The mask is applied inside the kernel as each weight tile is loaded; the
 * stored buffer is never modified.  Enqueue call.
 */
int tasq_masked_gemm(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt, const float* d_alpha,
                     const float* d_zc, int M, const void* d_packed, int N, int K, uint16_t* d_y, int32_t* d_acc,
                     tasq_stream stream);

/*
 * Grouped masked linear layers: `groups` (1..4) layers that read the same
 * activations -- e.g. the key and value projections of a cross-attention,
 * which both take the text tokens -- contracted in one launch, each at its own
 * operating precision b_g = table[h_layers[g]][stage] (App. F.1: the bit map
 * is per layer).  The layers' stored weights are packed together, once, as one
 * TASQ_LINEAR buffer of N = groups * Ng rows ([layer 0's Ng rows][layer 1's]
 * ...; tasq_pack_weights on the concatenated [N][K] codes, scales and biases),
 * and member g owns output channels [g Ng, (g + 1) Ng).  Output channel n of
 * member g is exactly what tasq_masked_gemm computes for layer h_layers[g]
 * alone (same contraction, mask and epilogue at b_g), so d_y [M][N] holds the
 * members' outputs side by side (and d_acc their int32 accumulators).
 * h_layers: host array of `groups` layer indices, read during the call.
 * Needs N % groups == 0 and Ng % 8 == 0; other arguments and rules as
 * tasq_masked_gemm (groups == 1 is tasq_masked_gemm).  The activations are
 * quantized once for the group, and the launch overhead is paid once.
 * Enqueue call.
 */
int tasq_masked_gemm_grouped(tasq_ctx ctx, const int32_t* h_layers, int groups, int stage, const void* d_codes,
                             int code_fmt, const float* d_alpha, const float* d_zc, int M, const void* d_packed,
                             int N, int K, uint16_t* d_y, int32_t* d_acc, tasq_stream stream);

/*
 * Many masked linear layers that read one input, in one launch: the grouped
 * call with its member list in device memory, for up to 256 members -- e.g. the
 * key and value projections of every cross-attention block of a denoising
 * step, which all take the same text tokens (the caption embedding is computed
 * once per forward pass), so that their activations are quantized once and
 * their weights streamed by one launch.  Member g is layer d_layers[g] and
 * runs at b_g = table[d_layers[g]][stage] (App. F.1: the bit map is per
 * layer); it owns output channels [g Ng, (g + 1) Ng), Ng = N / n_layers, of
 * one TASQ_LINEAR buffer packed from the members' [Ng][K] codes, scales and
 * biases concatenated along N, and its outputs are exactly what
 * tasq_masked_gemm computes for that layer alone.  d_layers: device int32
 * array of n_layers (1..256) layer indices, 4-byte aligned, owned by the
 * caller and read by every launch (a graph that captured the call reads it at
 * each replay); an index outside 0..L-1 is found on the device and recorded
 * as TASQ_ERR_DEVICE in the status word (tasq_device_status), with no output
 * written.  Needs N % n_layers == 0, Ng % 8 == 0, fp16 codes
 * (TASQ_CODES_F16 or TASQ_CODES_F16_E5M2) and the tensor-core route; the
 * launch is never split along K.  Other arguments and rules as
 * tasq_masked_gemm.  Enqueue call.
 */
int tasq_masked_gemm_shared_input(tasq_ctx ctx, const int32_t* d_layers, int n_layers, int stage,
                                  const void* d_codes, int code_fmt, const float* d_alpha, const float* d_zc, int M,
                                  const void* d_packed, int N, int K, uint16_t* d_y, int32_t* d_acc,
                                  tasq_stream stream);

/*
 * 16-bit low-rank branch of an SVD-split linear layer (the frozen SVD branch
 * that the paper's SVDQuant+TASQ pipelines carry beside the masked weights:
 * rank 32 for the 4-bit setting, 16 for the 6-bit one, Sec. 4 setup and the
 * training-setting table): y = Q(x) Q_b(R)^T + (x l2^T) l1^T.  The masked
 * contraction adds the up-projection inside its accumulator, in the
 * accumulator's units, as one more K block of fp16 tensor-core MMAs after the
 * last one of each output tile:
 *   acc'[m][n] = acc[m][n] + sum_j u'[m][j] * fp16(l1[n][j] * RN(1 / c_w[n])),
 *   u'[m][j] = fp16((sum_k bf16(x[m][k]) * l2[j][k]) / alpha[m]),
 * so that the epilogue's alpha[m] * c_w[n] scales it back to u . l1; the
 * epilogue then runs as for tasq_masked_gemm on acc' (held in fp32).
 *
 * tasq_lowrank_down: u' above (the sum over k accumulated in fp32 on the tensor
 * cores, order unspecified; one IEEE division by alpha[m]; fp16 rounding to
 * nearest even) into d_u [M][64] fp16 bits, columns >= rank zero.  d_x: the
 * layer's input [M][K], fp32 or bf16 (dtype; fp32 rounded to bf16 first);
 * d_l2: [rank][K] bf16 bits; d_alpha: [M] per-token scales of the layer's
 * activation codes (tasq_quant_act, per token).  rank 16 or 32, K % 16 == 0;
 * d_x 8-byte (fp32) or 4-byte (bf16) aligned, d_l2 4-byte and d_u 16-byte
 * aligned.  Enqueue call (one kernel), after the quantization.
 *
 * tasq_masked_gemm_lr: tasq_masked_gemm with the branch.  d_u: from
 * tasq_lowrank_down on this layer's input; d_l1: [N][rank] bf16 bits, 16-byte
 * aligned.  d_acc must be NULL (the accumulator carries the branch's fraction).
 * Tensor-core route only (fp16 or fp16 + e5m2 codes; the branch's block is fp16
 * either way); the launch is never split along K.  Other arguments as
 * tasq_masked_gemm.  Enqueue call.
 */
int tasq_lowrank_down(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, const uint16_t* d_l2, int rank,
                      const float* d_alpha, uint16_t* d_u, tasq_stream stream);
int tasq_masked_gemm_lr(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt, const float* d_alpha,
                        const float* d_zc, int M, const void* d_packed, int N, int K, const uint16_t* d_u,
                        const uint16_t* d_l1, int rank, uint16_t* d_y, int32_t* d_acc, tasq_stream stream);

/*
 * Masked linear layer with asymmetric weights (Eq. weight_dequant with the
 * zero point of tasq_quant_weights_asym, Eq. act_dequant):
 *   sum_k x_hat w_hat_b = alpha * c_w * (acc + zc * rs_b + zcw * t),
 *   t[m] = sum_k (s_x[m][k] + zc[m]) = sx[m] + K * zc[m],
 * in fp32 with each step rounded once, in this order:
 *   t = sx + K * zc (per token; K * zc rounded first), u = fma(zc, rs_b, acc),
 *   u = fma(zcw, t, u), s = alpha * c_w, y = bf16(fma(u, s, bias)).
 * d_code_sums: [M] from tasq_quant_act_sums.  d_packed: from
 * tasq_pack_weights_zp (zcw stored) or tasq_pack_weights (zcw = 0: the
 * result equals tasq_masked_gemm's).  Other arguments as tasq_masked_gemm.
 * Enqueue call.
 */
int tasq_masked_gemm_zp(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt, const float* d_alpha,
                        const float* d_zc, const int32_t* d_code_sums, int M, const void* d_packed, int N, int K,
                        uint16_t* d_y, int32_t* d_acc, tasq_stream stream);

/*
 * Masked 3x3 convolution, stride 1, padding 1, as an implicit GEMM over
 * K = 9*Cin (kh, kw, cin): same contraction and epilogue as
 * tasq_masked_gemm with one activation scale for the tensor (d_alpha[0],
 * d_zc[0], from a TASQ_PER_TENSOR quantization).  Padding is zero in the real
 * domain: a tap outside the image contributes nothing, so its weights are
 * left out of the row sum of that output pixel.
 * d_codes: NHWC [B][H][W][Cin]; d_y: NHWC [B][H][W][Cout] bf16 bits;
 * d_acc: [B*H*W][Cout] int32 or NULL.  d_packed: kind TASQ_CONV3X3 with
 * N = Cout, K = 9*Cin.  Enqueue call.
 */
int tasq_masked_conv3x3(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt, const float* d_alpha,
                        const float* d_zc, int B, int H, int W, int Cin, const void* d_packed, int Cout, uint16_t* d_y,
                        int32_t* d_acc, tasq_stream stream);

/*
 * Masked 3x3 convolution with asymmetric weights.  Padding is zero in the
 * real domain, so for output pixel p only its in-bounds taps carry zero-point
 * terms:
 *   y = alpha * c_w * (acc + zc * rs_b[p] + zcw * t[p]) + bias,
 *   t[p] = sxw[p] + Kv[p] * zc,
 * sxw[p] = sum of d_code_sums over the in-bounds taps' input pixels,
 * Kv[p] = Cin * (number of in-bounds taps), rs_b[p] as in tasq_masked_conv3x3.
 * fp32 order: t = sxw + (Kv * zc), u = fma(zc, rs_b, acc), u = fma(zcw, t, u),
 * y = bf16(fma(u, alpha * c_w, bias)).  d_code_sums: [B*H*W] per-pixel code
 * sums from tasq_quant_act_sums with TASQ_PER_TENSOR.  d_packed: from
 * tasq_pack_weights_zp with kind TASQ_CONV3X3.  Other arguments as
 * tasq_masked_conv3x3.  Enqueue call.
 */
int tasq_masked_conv3x3_zp(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                           const float* d_alpha, const float* d_zc, const int32_t* d_code_sums, int B, int H, int W,
                           int Cin, const void* d_packed, int Cout, uint16_t* d_y, int32_t* d_acc,
                           tasq_stream stream);

/* Launch plan of the tensor-core route for one contraction (see tasq_plan_tc). */
typedef struct {
    int tile_channels;      /* output channels per tile (MMA M): 128 */
    int tile_tokens;        /* tokens per tile (MMA N): 64, 192 or 256 */
    int acc_buffers;        /* fp32 accumulator buffers in tensor memory: 1 or 2 */
    int tiles_ch;           /* channel tiles: ceil(N / 128) */
    long long tiles_tok;    /* token tiles; a convolution tiles each image into boxes */
    int box_rows, box_cols; /* convolution: token box of box_rows image rows x box_cols pixels
                               (box_rows * box_cols == tile_tokens); 0 for a linear layer */
    int splits;             /* K slices, each summed by its own CTAs (1: K is not split) */
    int grid;               /* CTAs of the contraction kernel (persistent: at most num_sms) */
    int reduce_grid;        /* CTAs of the split-K reduction kernel (0 when splits == 1) */
    int kernels;            /* kernels the call enqueues: 1, 2 with split-K, 0 when M == 0 */
} tasq_tc_plan;

/*
 * The launch plan that tasq_masked_gemm(_zp) or tasq_masked_conv3x3(_zp) on
 * the tensor-core route (TASQ_ROUTE_TC) follows for this shape, on a device
 * with `num_sms` SMs and a context's own split-K scratch.  The plan depends on
 * the shape alone, not on the bits b or on the data.  Host-only: needs no
 * context and no device, enqueues nothing.  Diagnostic (the paper has no
 * counterpart): it lets a caller see how a layer is tiled without a GPU.
 * kind TASQ_LINEAR: M tokens, N outputs, K inputs (B, H, W, Cin ignored).
 * kind TASQ_CONV3X3: B, H, W, Cin and N = Cout (M = B*H*W and K = 9*Cin are
 * implied; the M and K arguments are ignored).  *out is zeroed first.
 * Returns TASQ_ERR_INVALID_ARG (bad kind, negative size, NULL out,
 * num_sms < 1) or TASQ_ERR_UNSUPPORTED (a shape the contraction calls would
 * reject on this route: K % 16, N % 8, Cin % 64 for a convolution), with the
 * text in tasq_last_error(NULL) on the calling thread.
 */
int tasq_plan_tc(int kind, int M, int N, int K, int B, int H, int W, int Cin, int num_sms, tasq_tc_plan* out);

/*
 * Probe of the tensor-core MMA kinds (diagnostic; the paper has no
 * counterpart).  Launches `ctas` CTAs (one per SM); each loads A (128 rows)
 * and B (n rows) of 128 bytes per row from d_a / d_b (row-major bytes: fp16
 * values for kind 0, e4m3 values for kind 1, e5m2 values for kind 2), and one
 * thread issues 4 * reps tcgen05.mma of that kind (kind 0: kind::f16, 16
 * elements of K per instruction; kind 1: kind::f8f6f4 with e4m3 A and B, kind 2:
 * kind::f8f6f4 with e5m2 A and B, 32 elements), M = 128,
 * N = n, accumulating D = reps * A . B^T (over the 64 or 128 elements of a row)
 * in fp32 in tensor memory.  d_cycles[i] receives CTA i's clock cycles from the
 * first MMA to the completion of the last (0 if that wait gave up after 2 s);
 * CTA 0 writes D to d_d [128][n] fp32.  16 <= n <= 256, n % 16 == 0,
 * 1 <= reps <= 2^20, 1 <= ctas <= 1024.  Enqueue call; no context.  Errors are
 * described by tasq_last_error(NULL) on the calling thread.
 */
int tasq_probe_mma(int kind, int n, int reps, const uint8_t* d_a, const uint8_t* d_b, float* d_d,
                   unsigned long long* d_cycles, int ctas, tasq_stream stream);

/*
 * Per-tensor activation quantization without any allocation (no context).
 * The paper has no counterpart to this call: it exists for callers that
 * cannot allocate device memory at run time -- for example an inference
 * plugin whose host framework forbids allocation while it enqueues work, or
 * a deployment whose device memory is planned once before serving -- and so
 * cannot create a context (tasq_create allocates).
 * It computes exactly what tasq_quant_act computes with gran =
 * TASQ_PER_TENSOR (same arguments and layouts; d_alpha and d_zc hold one
 * value each), but its reduction scratch is a 16 KB array compiled into the
 * library, which every GPU that loads the library keeps until the process
 * exits.  The call itself allocates nothing: it enqueues two kernels on
 * `stream` and returns.
 *  - Limit: M * K <= 67,108,864 elements (2048 slices of 32,768); larger
 *    tensors return TASQ_ERR_UNSUPPORTED without launching anything.
 *  - The first call on a device looks up the array's device address once
 *    (cudaGetSymbolAddress, with that device current); make that first call
 *    before capturing a stream into a CUDA graph.  The address is kept for
 *    the life of the process: it does not survive cudaDeviceReset (or any
 *    other reset of the device's primary context), after which this call
 *    must not be used in that process.
 *  - Every call uses the same array, and each call rewrites the slots it
 *    reads, so nothing carries over between calls; but calls whose kernels
 *    overlap on the GPU (different streams, or one device used from several
 *    threads without ordering) race on the array and must be serialized.
 *  - Errors are described by tasq_last_error(NULL) on the calling thread.
 */
int tasq_quant_act_tensor_noalloc(const void* d_x, int dtype, int M, int K, int n_bits, int mode, void* d_codes,
                                  int code_fmt, float* d_alpha, float* d_zc, tasq_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* TASQ_H */
