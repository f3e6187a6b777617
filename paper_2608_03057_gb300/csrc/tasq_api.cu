// Host side of the C ABI declared in include/tasq.h: the context, argument
// validation (nothing is launched for an invalid call) and kernel launches.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "tasq_internal.cuh"

#define TASQ_API extern "C" __attribute__((visibility("default")))

struct tasq_ctx_s {
    int device = 0;
    int num_sms = 0;
    int* d_words = nullptr;  // [0] status, [16..19] reduction scratch
    int32_t* d_part = nullptr;  // tensor-core route: int32 running sums of multi-chunk tiles
    int32_t* d_split = nullptr;  // tensor-core route: split-K partial sums
    // bit table: a 16-byte header (int32 L, S) followed by the bits [L][S]; kernels
    // read L and S from the header, so a captured graph follows later schedules
    uint8_t* d_table = nullptr;
    size_t table_cap = 0;              // bits the current buffer holds
    std::vector<uint8_t*> old_tables;  // replaced buffers, kept until tasq_destroy
    int L = 0, S = 0;
    const int32_t* d_stage = nullptr;
    int route = TASQ_ROUTE_AUTO;
    unsigned long long timeout_ns = 2000000000ull;
    unsigned long long kernels = 0;  // kernels enqueued by quant_act / masked_gemm / masked_conv3x3
    std::string err;
};

namespace {

thread_local std::string g_create_err;

int fail(tasq_ctx ctx, int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (ctx) ctx->err = buf;
    else g_create_err = buf;
    return code;
}

int cuda_fail(tasq_ctx ctx, cudaError_t e, const char* what) {
    return fail(ctx, TASQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int check_ctx(tasq_ctx ctx) {
    if (!ctx) return TASQ_ERR_INVALID_ARG;
    int cur = -1;
    cudaError_t e = cudaGetDevice(&cur);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaGetDevice");
    if (cur != ctx->device)
        return fail(ctx, TASQ_ERR_INVALID_ARG, "current device %d is not the context's device %d", cur, ctx->device);
    ctx->err.clear();
    return TASQ_OK;
}

#define CHECK_CTX(ctx)                      \
    do {                                    \
        int rc_ = check_ctx(ctx);           \
        if (rc_ != TASQ_OK) return rc_;     \
    } while (0)

#define REQUIRE(cond, code, ...)                          \
    do {                                                  \
        if (!(cond)) return fail(ctx, code, __VA_ARGS__); \
    } while (0)

}  // namespace

TASQ_API int tasq_version(void) { return TASQ_ABI_VERSION; }

TASQ_API int tasq_create(tasq_ctx* out, int device) {
    if (!out) return fail(nullptr, TASQ_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    int count = 0;
    cudaError_t e = cudaGetDeviceCount(&count);
    if (e != cudaSuccess) return fail(nullptr, TASQ_ERR_CUDA, "cudaGetDeviceCount: %s", cudaGetErrorString(e));
    if (device < 0 || device >= count) return fail(nullptr, TASQ_ERR_INVALID_ARG, "device %d out of range", device);
    cudaDeviceProp prop;
    if ((e = cudaGetDeviceProperties(&prop, device)) != cudaSuccess)
        return fail(nullptr, TASQ_ERR_CUDA, "cudaGetDeviceProperties: %s", cudaGetErrorString(e));
    if (prop.major != 10 || prop.minor != 3)
        return fail(nullptr, TASQ_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a", device,
                    prop.major, prop.minor);
    int prev = 0;
    cudaGetDevice(&prev);
    if ((e = cudaSetDevice(device)) != cudaSuccess)
        return fail(nullptr, TASQ_ERR_CUDA, "cudaSetDevice: %s", cudaGetErrorString(e));
    tasq_ctx ctx = new tasq_ctx_s();
    ctx->device = device;
    ctx->num_sms = prop.multiProcessorCount;
    e = cudaMalloc(&ctx->d_words, 256);
    if (e == cudaSuccess) e = cudaMemset(ctx->d_words, 0, 256);
    if (e == cudaSuccess) e = cudaMalloc(&ctx->d_part, tasq::gemm_tc_part_bytes(ctx->num_sms));
    if (e == cudaSuccess) e = cudaMalloc(&ctx->d_split, tasq::kSplitBufBytes);
    if (e == cudaSuccess) e = cudaMalloc(&ctx->d_table, tasq::kTableHeader + tasq::kTableCapacity);
    if (e == cudaSuccess) e = cudaMemset(ctx->d_table, 0, tasq::kTableHeader);  // L = S = 0: no schedule yet
    if (e == cudaSuccess) ctx->table_cap = tasq::kTableCapacity;
    cudaSetDevice(prev);
    if (e != cudaSuccess) {
        cudaFree(ctx->d_words);
        cudaFree(ctx->d_part);
        cudaFree(ctx->d_split);
        cudaFree(ctx->d_table);
        delete ctx;
        return fail(nullptr, TASQ_ERR_CUDA, "allocating context buffers: %s", cudaGetErrorString(e));
    }
    *out = ctx;
    return TASQ_OK;
}

TASQ_API void tasq_destroy(tasq_ctx ctx) {
    if (!ctx) return;
    int prev = 0;
    cudaGetDevice(&prev);
    cudaSetDevice(ctx->device);
    cudaDeviceSynchronize();
    cudaFree(ctx->d_words);
    cudaFree(ctx->d_part);
    cudaFree(ctx->d_split);
    cudaFree(ctx->d_table);
    for (uint8_t* t : ctx->old_tables) cudaFree(t);
    cudaSetDevice(prev);
    delete ctx;
}

TASQ_API const char* tasq_last_error(tasq_ctx ctx) { return ctx ? ctx->err.c_str() : g_create_err.c_str(); }

namespace tasq {
// Error text of calls made without a context (read by tasq_last_error(NULL)).
void set_noctx_error(const char* msg) { g_create_err = msg; }
}  // namespace tasq

TASQ_API int tasq_device_status(tasq_ctx ctx, int* out) {
    CHECK_CTX(ctx);
    REQUIRE(out, TASQ_ERR_INVALID_ARG, "out is NULL");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaDeviceSynchronize");
    int v = 0;
    if ((e = cudaMemcpy(&v, ctx->d_words, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(ctx, e, "reading the status word");
    if ((e = cudaMemset(ctx->d_words, 0, sizeof v)) != cudaSuccess) return cuda_fail(ctx, e, "clearing the status word");
    *out = v;
    return TASQ_OK;
}

TASQ_API int tasq_kernel_count(tasq_ctx ctx, unsigned long long* out) {
    CHECK_CTX(ctx);
    REQUIRE(out, TASQ_ERR_INVALID_ARG, "out is NULL");
    *out = ctx->kernels;
    return TASQ_OK;
}

TASQ_API int tasq_set_route(tasq_ctx ctx, int route) {
    CHECK_CTX(ctx);
    REQUIRE(route >= TASQ_ROUTE_AUTO && route <= TASQ_ROUTE_MMA_S8, TASQ_ERR_INVALID_ARG, "route %d", route);
    ctx->route = route;
    return TASQ_OK;
}

TASQ_API int tasq_set_timeout_ns(tasq_ctx ctx, uint64_t ns) {
    CHECK_CTX(ctx);
    ctx->timeout_ns = ns ? ns : 2000000000ull;
    return TASQ_OK;
}

TASQ_API int tasq_selftest_timeout(tasq_ctx ctx, uint64_t timeout_ns, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(timeout_ns > 0 && timeout_ns <= 10000000000ull, TASQ_ERR_INVALID_ARG, "timeout_ns must be in (0, 1e10]");
    cudaError_t e = tasq::launch_selftest_timeout(ctx->d_words, timeout_ns, (cudaStream_t)stream);
    return e == cudaSuccess ? TASQ_OK : cuda_fail(ctx, e, "selftest launch");
}

TASQ_API int tasq_selftest_quotients(tasq_ctx ctx, const float* d_x, int nx, const float* d_a, int na,
                                    unsigned long long* d_mismatches, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(nx > 0 && na > 0 && d_x && d_a && d_mismatches, TASQ_ERR_INVALID_ARG, "need nx, na > 0 and pointers");
    cudaError_t e = tasq::launch_selftest_quotients(d_x, nx, d_a, na, d_mismatches, (cudaStream_t)stream);
    return e == cudaSuccess ? TASQ_OK : cuda_fail(ctx, e, "selftest launch");
}

namespace {

int quant_weights(tasq_ctx ctx, const void* d_w, int dtype, int N, int K, int mode, int8_t* d_sw, float* d_cw,
                  float* d_zcw, float* d_alpha, tasq_stream stream) {
    REQUIRE(dtype == TASQ_F32 || dtype == TASQ_BF16, TASQ_ERR_INVALID_ARG, "dtype %d", dtype);
    REQUIRE(N >= 0 && K > 0, TASQ_ERR_INVALID_ARG, "N=%d K=%d", N, K);
    REQUIRE(K % 16 == 0, TASQ_ERR_UNSUPPORTED, "K=%d must be a multiple of 16", K);
    REQUIRE(N == 0 || (d_w && d_sw && d_cw && (mode == TASQ_SYMRANGE || d_zcw)), TASQ_ERR_INVALID_ARG,
            "NULL pointer");
    REQUIRE(aligned16(d_w) && aligned16(d_sw) && aligned16(d_cw) && aligned16(d_alpha) && aligned16(d_zcw),
            TASQ_ERR_UNSUPPORTED, "pointers must be 16-byte aligned");
    cudaError_t e = tasq::launch_quant_weights(d_w, dtype, N, K, mode, d_sw, d_cw, d_zcw, d_alpha, (cudaStream_t)stream);
    return e == cudaSuccess ? TASQ_OK : cuda_fail(ctx, e, "quant_weights launch");
}

}  // namespace

TASQ_API int tasq_quant_weights(tasq_ctx ctx, const void* d_w, int dtype, int N, int K, int8_t* d_sw, float* d_cw,
                                float* d_alpha, tasq_stream stream) {
    CHECK_CTX(ctx);
    return quant_weights(ctx, d_w, dtype, N, K, TASQ_SYMRANGE, d_sw, d_cw, nullptr, d_alpha, stream);
}

TASQ_API int tasq_quant_weights_asym(tasq_ctx ctx, const void* d_w, int dtype, int N, int K, int8_t* d_sw,
                                     float* d_cw, float* d_zcw, float* d_alpha, tasq_stream stream) {
    CHECK_CTX(ctx);
    return quant_weights(ctx, d_w, dtype, N, K, TASQ_ASYM, d_sw, d_cw, d_zcw, d_alpha, stream);
}

TASQ_API size_t tasq_packed_bytes(int kind, int N, int K) {
    if ((kind != TASQ_LINEAR && kind != TASQ_CONV3X3) || N < 0 || K <= 0) return 0;
    if (kind == TASQ_CONV3X3 && K % 9) return 0;
    return (size_t)tasq::packed_layout(kind, N, K).total;
}

namespace {

int pack_weights(tasq_ctx ctx, int kind, const int8_t* d_sw, const float* d_cw, const float* d_zcw,
                 const float* d_bias, int N, int K, int Cin, void* d_packed, tasq_stream stream) {
    REQUIRE(kind == TASQ_LINEAR || kind == TASQ_CONV3X3, TASQ_ERR_INVALID_ARG, "kind %d", kind);
    REQUIRE(N > 0 && K > 0, TASQ_ERR_INVALID_ARG, "N=%d K=%d", N, K);
    REQUIRE(K % 16 == 0 && N % 8 == 0, TASQ_ERR_UNSUPPORTED, "need K %% 16 == 0 and N %% 8 == 0 (N=%d K=%d)", N, K);
    if (kind == TASQ_CONV3X3) {
        REQUIRE(Cin > 0 && K == 9 * Cin, TASQ_ERR_INVALID_ARG, "conv: K=%d must be 9*Cin (Cin=%d)", K, Cin);
        REQUIRE(Cin % 16 == 0, TASQ_ERR_UNSUPPORTED, "conv: Cin=%d must be a multiple of 16", Cin);
    }
    REQUIRE(d_sw && d_cw && d_packed, TASQ_ERR_INVALID_ARG, "NULL pointer");
    REQUIRE((reinterpret_cast<uintptr_t>(d_packed) & 255u) == 0, TASQ_ERR_UNSUPPORTED, "d_packed must be 256-byte aligned");
    REQUIRE(aligned16(d_sw) && aligned16(d_cw) && aligned16(d_bias) && aligned16(d_zcw), TASQ_ERR_UNSUPPORTED,
            "pointers must be 16-byte aligned");
    cudaError_t e = tasq::launch_pack(kind, d_sw, d_cw, d_zcw, d_bias, N, K, kind == TASQ_CONV3X3 ? Cin : 0, d_packed,
                                      (cudaStream_t)stream);
    return e == cudaSuccess ? TASQ_OK : cuda_fail(ctx, e, "pack launch");
}

}  // namespace

TASQ_API int tasq_pack_weights(tasq_ctx ctx, int kind, const int8_t* d_sw, const float* d_cw, const float* d_bias,
                               int N, int K, int Cin, void* d_packed, tasq_stream stream) {
    CHECK_CTX(ctx);
    return pack_weights(ctx, kind, d_sw, d_cw, nullptr, d_bias, N, K, Cin, d_packed, stream);
}

TASQ_API int tasq_pack_weights_zp(tasq_ctx ctx, int kind, const int8_t* d_sw, const float* d_cw, const float* d_zcw,
                                  const float* d_bias, int N, int K, int Cin, void* d_packed, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(d_zcw, TASQ_ERR_INVALID_ARG, "NULL pointer");
    return pack_weights(ctx, kind, d_sw, d_cw, d_zcw, d_bias, N, K, Cin, d_packed, stream);
}

TASQ_API int tasq_set_schedule(tasq_ctx ctx, const uint8_t* h_bits, int L, int S) {
    CHECK_CTX(ctx);
    REQUIRE(h_bits && L > 0 && S > 0, TASQ_ERR_INVALID_ARG, "need h_bits, L > 0, S > 0");
    REQUIRE((int64_t)L * S <= (int64_t(1) << 30), TASQ_ERR_INVALID_ARG, "table too large");
    for (int64_t i = 0; i < (int64_t)L * S; ++i)
        REQUIRE(h_bits[i] >= tasq::kBMin && h_bits[i] <= tasq::kBMax, TASQ_ERR_INVALID_ARG,
                "bits[%lld] = %d is outside 2..8", (long long)i, (int)h_bits[i]);
    cudaError_t e = cudaDeviceSynchronize();  // no kernel may be reading the old table
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaDeviceSynchronize");
    size_t bytes = (size_t)L * S;
    if (bytes > ctx->table_cap) {
        // a larger buffer; the old one stays allocated (graphs captured before this
        // call still name it) until tasq_destroy
        uint8_t* t = nullptr;
        if ((e = cudaMalloc(&t, tasq::kTableHeader + bytes)) != cudaSuccess)
            return cuda_fail(ctx, e, "allocating the table");
        ctx->old_tables.push_back(ctx->d_table);
        ctx->d_table = t;
        ctx->table_cap = bytes;
    }
    const int32_t dims[4] = {L, S, 0, 0};
    if ((e = cudaMemcpy(ctx->d_table + tasq::kTableHeader, h_bits, bytes, cudaMemcpyHostToDevice)) != cudaSuccess ||
        (e = cudaMemcpy(ctx->d_table, dims, sizeof dims, cudaMemcpyHostToDevice)) != cudaSuccess)
        return cuda_fail(ctx, e, "copying the table");
    ctx->L = L;
    ctx->S = S;
    return TASQ_OK;
}

TASQ_API int tasq_set_stage_device(tasq_ctx ctx, const int32_t* d_stage) {
    CHECK_CTX(ctx);
    REQUIRE((reinterpret_cast<uintptr_t>(d_stage) & 3u) == 0, TASQ_ERR_INVALID_ARG, "d_stage must be 4-byte aligned");
    ctx->d_stage = d_stage;
    return TASQ_OK;
}

namespace {

int quant_act(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, int n_bits, int mode, int gran, void* d_codes,
              int code_fmt, float* d_alpha, float* d_zc, int32_t* d_code_sums, tasq_stream stream) {
    REQUIRE(dtype == TASQ_F32 || dtype == TASQ_BF16, TASQ_ERR_INVALID_ARG, "dtype %d", dtype);
    REQUIRE(mode == TASQ_SYMRANGE || mode == TASQ_ASYM, TASQ_ERR_INVALID_ARG, "mode %d", mode);
    REQUIRE(gran == TASQ_PER_TOKEN || gran == TASQ_PER_TENSOR, TASQ_ERR_INVALID_ARG, "gran %d", gran);
    REQUIRE(code_fmt == TASQ_CODES_S8 || code_fmt == TASQ_CODES_F16 || code_fmt == TASQ_CODES_F16_E5M2,
            TASQ_ERR_INVALID_ARG, "code_fmt %d", code_fmt);
    REQUIRE(n_bits >= 2 && n_bits <= 8, TASQ_ERR_INVALID_ARG, "n_bits %d outside 2..8", n_bits);
    REQUIRE(code_fmt != TASQ_CODES_F16_E5M2 || n_bits <= 4, TASQ_ERR_UNSUPPORTED,
            "e5m2 codes need n_bits <= 4 (codes of magnitude <= 8), got %d", n_bits);
    REQUIRE(M >= 0 && K > 0, TASQ_ERR_INVALID_ARG, "M=%d K=%d", M, K);
    REQUIRE(K % 16 == 0, TASQ_ERR_UNSUPPORTED, "K=%d must be a multiple of 16", K);
    if (M == 0) return TASQ_OK;
    REQUIRE(d_x && d_codes && d_alpha && d_zc, TASQ_ERR_INVALID_ARG, "NULL pointer");
    REQUIRE(aligned16(d_x) && aligned16(d_codes), TASQ_ERR_UNSUPPORTED, "pointers must be 16-byte aligned");
    cudaError_t e;
    if (gran == TASQ_PER_TOKEN)
        e = tasq::launch_quant_act_token(d_x, dtype, M, K, n_bits, mode, d_codes, code_fmt, d_alpha, d_zc, d_code_sums,
                                         (cudaStream_t)stream);
    else
        e = tasq::launch_quant_act_tensor(d_x, dtype, (int64_t)M * K, n_bits, mode, d_codes, code_fmt, d_alpha, d_zc,
                                          reinterpret_cast<unsigned int*>(ctx->d_words + 16), (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "quant_act launch");
    ctx->kernels += gran == TASQ_PER_TOKEN ? 1 : 2;
    if (gran == TASQ_PER_TENSOR && d_code_sums) {
        // per-row code sums of a per-tensor quantization (conv: one row per pixel)
        e = tasq::launch_code_row_sums(d_codes, code_fmt, M, K, d_code_sums, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "code sums launch");
        ctx->kernels += 1;
    }
    return TASQ_OK;
}

}  // namespace

TASQ_API int tasq_quant_act(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, int n_bits, int mode, int gran,
                            void* d_codes, int code_fmt, float* d_alpha, float* d_zc, tasq_stream stream) {
    CHECK_CTX(ctx);
    return quant_act(ctx, d_x, dtype, M, K, n_bits, mode, gran, d_codes, code_fmt, d_alpha, d_zc, nullptr, stream);
}

TASQ_API int tasq_quant_act_sums(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, int n_bits, int mode,
                                 int gran, void* d_codes, int code_fmt, float* d_alpha, float* d_zc,
                                 int32_t* d_code_sums, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(M == 0 || d_code_sums, TASQ_ERR_INVALID_ARG, "NULL pointer");
    return quant_act(ctx, d_x, dtype, M, K, n_bits, mode, gran, d_codes, code_fmt, d_alpha, d_zc, d_code_sums, stream);
}

namespace {

// layers[0..groups): the member layers of a grouped call (one for a single layer), or
// d_layers[0..groups): the same list in device memory (then layers is unused)
int masked_contraction(tasq_ctx ctx, int kind, const int* layers, int groups, int stage, const void* d_codes,
                       int code_fmt, const float* d_alpha, const float* d_zc, const int32_t* d_code_sums, int M,
                       const void* d_packed, int N, int K, int B, int H, int W, int Cin, uint16_t* d_y,
                       int32_t* d_acc, tasq_stream stream, const uint16_t* d_lr_u = nullptr,
                       const uint16_t* d_lr_l1 = nullptr, int lr_rank = 0, const int32_t* d_layers = nullptr) {
    REQUIRE(ctx->L > 0, TASQ_ERR_INVALID_ARG, "no schedule: call tasq_set_schedule first");
    if (d_layers) {
        REQUIRE(groups >= 1 && groups <= tasq::kMaxMembers, TASQ_ERR_INVALID_ARG, "layers %d outside 1..%d", groups,
                tasq::kMaxMembers);
        REQUIRE((reinterpret_cast<uintptr_t>(d_layers) & 3u) == 0, TASQ_ERR_UNSUPPORTED,
                "d_layers must be 4-byte aligned");
    } else {
        REQUIRE(layers && groups >= 1 && groups <= tasq::kMaxGroups, TASQ_ERR_INVALID_ARG,
                "groups %d outside 1..%d", groups, tasq::kMaxGroups);
        for (int g = 0; g < groups; ++g)
            REQUIRE(layers[g] >= 0 && layers[g] < ctx->L, TASQ_ERR_INVALID_ARG, "layer %d outside 0..%d", layers[g],
                    ctx->L - 1);
    }
    REQUIRE(stage >= -1 && stage < ctx->S, TASQ_ERR_INVALID_ARG, "stage %d outside -1..%d", stage, ctx->S - 1);
    REQUIRE(stage >= 0 || ctx->d_stage, TASQ_ERR_INVALID_ARG, "stage -1 needs tasq_set_stage_device");
    REQUIRE(code_fmt == TASQ_CODES_S8 || code_fmt == TASQ_CODES_F16 || code_fmt == TASQ_CODES_F16_E5M2,
            TASQ_ERR_INVALID_ARG, "code_fmt %d", code_fmt);
    REQUIRE(M >= 0 && N > 0 && K > 0, TASQ_ERR_INVALID_ARG, "M=%d N=%d K=%d", M, N, K);
    REQUIRE(K % 16 == 0 && N % 8 == 0, TASQ_ERR_UNSUPPORTED, "need K %% 16 == 0 and N %% 8 == 0 (N=%d K=%d)", N, K);
    REQUIRE(groups == 1 || (N % groups == 0 && (N / groups) % 8 == 0), TASQ_ERR_UNSUPPORTED,
            "grouped call: N=%d must split into %d members of a multiple of 8 channels", N, groups);
    int route = ctx->route;
    if (route == TASQ_ROUTE_AUTO) route = code_fmt == TASQ_CODES_S8 ? TASQ_ROUTE_MMA_S8 : TASQ_ROUTE_TC;
    REQUIRE((route == TASQ_ROUTE_TC) == (code_fmt != TASQ_CODES_S8), TASQ_ERR_UNSUPPORTED,
            "route %d cannot read code format %d", route, code_fmt);
    REQUIRE(!d_layers || route == TASQ_ROUTE_TC, TASQ_ERR_UNSUPPORTED,
            "a member list in device memory needs the tensor-core route");
    if (M == 0) return TASQ_OK;
    REQUIRE(d_codes && d_alpha && d_zc && d_packed && d_y, TASQ_ERR_INVALID_ARG, "NULL pointer");
    REQUIRE(aligned16(d_codes) && aligned16(d_y) && aligned16(d_acc), TASQ_ERR_UNSUPPORTED,
            "pointers must be 16-byte aligned");
    REQUIRE((reinterpret_cast<uintptr_t>(d_packed) & 255u) == 0, TASQ_ERR_UNSUPPORTED, "d_packed must be 256-byte aligned");
    if (lr_rank) {
        REQUIRE(route == TASQ_ROUTE_TC, TASQ_ERR_UNSUPPORTED, "the low-rank branch runs on the tensor-core route");
        REQUIRE(d_lr_u && d_lr_l1, TASQ_ERR_INVALID_ARG, "NULL pointer");
        REQUIRE(!d_acc, TASQ_ERR_INVALID_ARG, "no int32 accumulators with the low-rank branch (d_acc must be NULL)");
        REQUIRE(aligned16(d_lr_u) && aligned16(d_lr_l1), TASQ_ERR_UNSUPPORTED, "d_u and d_l1 must be 16-byte aligned");
    }

    const tasq::PackedHeader lay = tasq::packed_layout(kind, N, K);
    const char* p = reinterpret_cast<const char*>(d_packed);
    tasq::GemmArgs a{};
    a.x = d_codes;
    // the e5m2 copy of the codes follows the M x K fp16 codes (linear layers use it)
    a.x8 = code_fmt == TASQ_CODES_F16_E5M2 && kind == TASQ_LINEAR
               ? static_cast<const char*>(d_codes) + int64_t(M) * K * 2
               : nullptr;
    // the certificate bounds sum |mask_b(s_w)| for codes of magnitude <= 128; codes of
    // magnitude <= 8 keep 16 times as long a run below 2^24
    a.chunk_scale = code_fmt == TASQ_CODES_F16_E5M2 ? 128 / tasq::kF8CodeMax : 1;
    a.alpha = d_alpha;
    a.zc = d_zc;
    a.w = reinterpret_cast<const int8_t*>(p + lay.off_w);
    a.cw = reinterpret_cast<const float*>(p + lay.off_cw);
    a.bias = reinterpret_cast<const float*>(p + lay.off_bias);
    a.rs = reinterpret_cast<const int32_t*>(p + lay.off_rs);
    a.ts = kind == TASQ_CONV3X3 ? reinterpret_cast<const int32_t*>(p + lay.off_ts) : nullptr;
    a.hdr = reinterpret_cast<const tasq::PackedHeader*>(p);
    a.table = ctx->d_table;
    a.d_stage = ctx->d_stage;
    a.stage = stage;
    a.groups = groups;
    a.group_n = N / groups;
    if (d_layers) {
        a.layer = -1;
        a.d_layers = d_layers;
    } else {
        a.layer = layers[0];
        for (int g = 0; g < groups; ++g) a.layers[g] = layers[g];
    }
    a.M = M;
    a.N = N;
    a.K = K;
    a.B = B;
    a.H = H;
    a.W = W;
    a.Cin = Cin;
    a.per_tensor = kind == TASQ_CONV3X3;
    a.y = d_y;
    a.acc = d_acc;
    a.part = ctx->d_part;
    a.split_buf = ctx->d_split;
    a.split_cap = tasq::kSplitBufBytes / int64_t(sizeof(int32_t));
    a.status = ctx->d_words;
    a.timeout_ns = ctx->timeout_ns;
    a.zcw = reinterpret_cast<const float*>(p + lay.off_zcw);
    a.code_sums = d_code_sums;
    a.lr_u = d_lr_u;
    a.lr_l1 = d_lr_l1;
    a.lr_rank = lr_rank;
    cudaError_t e;
    int kernels = 0;
    if (route == TASQ_ROUTE_TC) {
        const char* why = nullptr;
        e = tasq::launch_gemm_tc(a, ctx->num_sms, (cudaStream_t)stream, &why, &kernels);
        if (why) return fail(ctx, TASQ_ERR_UNSUPPORTED, "tensor-core route: %s", why);
    } else {
        e = tasq::launch_gemm_s8(a, ctx->num_sms, (cudaStream_t)stream);
        kernels = 1;
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "masked contraction launch");
    ctx->kernels += kernels;
    return TASQ_OK;
}

}  // namespace

TASQ_API int tasq_masked_gemm(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                              const float* d_alpha, const float* d_zc, int M, const void* d_packed, int N, int K,
                              uint16_t* d_y, int32_t* d_acc, tasq_stream stream) {
    CHECK_CTX(ctx);
    return masked_contraction(ctx, TASQ_LINEAR, &layer, 1, stage, d_codes, code_fmt, d_alpha, d_zc, nullptr, M,
                              d_packed, N, K, 1, 0, 0, 0, d_y, d_acc, stream);
}

TASQ_API int tasq_masked_gemm_lr(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                                 const float* d_alpha, const float* d_zc, int M, const void* d_packed, int N, int K,
                                 const uint16_t* d_u, const uint16_t* d_l1, int rank, uint16_t* d_y, int32_t* d_acc,
                                 tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(rank == 16 || rank == 32, TASQ_ERR_INVALID_ARG, "rank %d: 16 or 32", rank);
    return masked_contraction(ctx, TASQ_LINEAR, &layer, 1, stage, d_codes, code_fmt, d_alpha, d_zc, nullptr, M,
                              d_packed, N, K, 1, 0, 0, 0, d_y, d_acc, stream, d_u, d_l1, rank);
}

TASQ_API int tasq_lowrank_down(tasq_ctx ctx, const void* d_x, int dtype, int M, int K, const uint16_t* d_l2, int rank,
                               const float* d_alpha, uint16_t* d_u, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(dtype == TASQ_F32 || dtype == TASQ_BF16, TASQ_ERR_INVALID_ARG, "dtype %d", dtype);
    REQUIRE(rank == 16 || rank == 32, TASQ_ERR_INVALID_ARG, "rank %d: 16 or 32", rank);
    REQUIRE(M >= 0 && K > 0, TASQ_ERR_INVALID_ARG, "M=%d K=%d", M, K);
    REQUIRE(K % 16 == 0, TASQ_ERR_UNSUPPORTED, "K=%d must be a multiple of 16", K);
    if (M == 0) return TASQ_OK;
    REQUIRE(d_x && d_l2 && d_alpha && d_u, TASQ_ERR_INVALID_ARG, "NULL pointer");
    REQUIRE((reinterpret_cast<uintptr_t>(d_x) & (dtype == TASQ_F32 ? 7u : 3u)) == 0 &&
                (reinterpret_cast<uintptr_t>(d_l2) & 3u) == 0 && aligned16(d_u),
            TASQ_ERR_UNSUPPORTED,
            "d_x must be 8-byte (fp32) or 4-byte (bf16) aligned, d_l2 4-byte and d_u 16-byte aligned");
    const cudaError_t e = tasq::launch_lowrank_down(d_x, dtype, M, K, d_l2, rank, d_alpha, 0, d_u, ctx->d_words,
                                                    ctx->timeout_ns, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "low-rank launch");
    ctx->kernels += 1;
    return TASQ_OK;
}

TASQ_API int tasq_masked_gemm_zp(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                                 const float* d_alpha, const float* d_zc, const int32_t* d_code_sums, int M,
                                 const void* d_packed, int N, int K, uint16_t* d_y, int32_t* d_acc,
                                 tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(M == 0 || d_code_sums, TASQ_ERR_INVALID_ARG, "NULL pointer");
    return masked_contraction(ctx, TASQ_LINEAR, &layer, 1, stage, d_codes, code_fmt, d_alpha, d_zc, d_code_sums, M,
                              d_packed, N, K, 1, 0, 0, 0, d_y, d_acc, stream);
}

TASQ_API int tasq_masked_gemm_grouped(tasq_ctx ctx, const int32_t* h_layers, int groups, int stage,
                                      const void* d_codes, int code_fmt, const float* d_alpha, const float* d_zc,
                                      int M, const void* d_packed, int N, int K, uint16_t* d_y, int32_t* d_acc,
                                      tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(h_layers, TASQ_ERR_INVALID_ARG, "NULL pointer");
    int layers[tasq::kMaxGroups] = {};
    for (int g = 0; g < groups && g < tasq::kMaxGroups; ++g) layers[g] = h_layers[g];
    return masked_contraction(ctx, TASQ_LINEAR, layers, groups, stage, d_codes, code_fmt, d_alpha, d_zc, nullptr, M,
                              d_packed, N, K, 1, 0, 0, 0, d_y, d_acc, stream);
}

TASQ_API int tasq_masked_gemm_shared_input(tasq_ctx ctx, const int32_t* d_layers, int n_layers, int stage,
                                           const void* d_codes, int code_fmt, const float* d_alpha,
                                           const float* d_zc, int M, const void* d_packed, int N, int K,
                                           uint16_t* d_y, int32_t* d_acc, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(d_layers, TASQ_ERR_INVALID_ARG, "NULL pointer");
    REQUIRE(code_fmt != TASQ_CODES_S8, TASQ_ERR_UNSUPPORTED, "a member list in device memory needs fp16 codes");
    return masked_contraction(ctx, TASQ_LINEAR, nullptr, n_layers, stage, d_codes, code_fmt, d_alpha, d_zc, nullptr,
                              M, d_packed, N, K, 1, 0, 0, 0, d_y, d_acc, stream, nullptr, nullptr, 0, d_layers);
}

TASQ_API int tasq_masked_conv3x3(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                                 const float* d_alpha, const float* d_zc, int B, int H, int W, int Cin,
                                 const void* d_packed, int Cout, uint16_t* d_y, int32_t* d_acc, tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(B >= 0 && H > 0 && W > 0 && Cin > 0, TASQ_ERR_INVALID_ARG, "B=%d H=%d W=%d Cin=%d", B, H, W, Cin);
    REQUIRE(Cin % 16 == 0, TASQ_ERR_UNSUPPORTED, "conv: Cin=%d must be a multiple of 16", Cin);
    REQUIRE((int64_t)B * H * W <= 0x7FFFFFFF && (int64_t)9 * Cin <= 0x7FFFFFFF, TASQ_ERR_UNSUPPORTED, "too large");
    return masked_contraction(ctx, TASQ_CONV3X3, &layer, 1, stage, d_codes, code_fmt, d_alpha, d_zc, nullptr,
                              B * H * W, d_packed, Cout, 9 * Cin, B, H, W, Cin, d_y, d_acc, stream);
}

TASQ_API int tasq_masked_conv3x3_zp(tasq_ctx ctx, int layer, int stage, const void* d_codes, int code_fmt,
                                    const float* d_alpha, const float* d_zc, const int32_t* d_code_sums, int B, int H,
                                    int W, int Cin, const void* d_packed, int Cout, uint16_t* d_y, int32_t* d_acc,
                                    tasq_stream stream) {
    CHECK_CTX(ctx);
    REQUIRE(B >= 0 && H > 0 && W > 0 && Cin > 0, TASQ_ERR_INVALID_ARG, "B=%d H=%d W=%d Cin=%d", B, H, W, Cin);
    REQUIRE(Cin % 16 == 0, TASQ_ERR_UNSUPPORTED, "conv: Cin=%d must be a multiple of 16", Cin);
    REQUIRE((int64_t)B * H * W <= 0x7FFFFFFF && (int64_t)9 * Cin <= 0x7FFFFFFF, TASQ_ERR_UNSUPPORTED, "too large");
    REQUIRE(B == 0 || d_code_sums, TASQ_ERR_INVALID_ARG, "NULL pointer");
    return masked_contraction(ctx, TASQ_CONV3X3, &layer, 1, stage, d_codes, code_fmt, d_alpha, d_zc, d_code_sums,
                              B * H * W, d_packed, Cout, 9 * Cin, B, H, W, Cin, d_y, d_acc, stream);
}

TASQ_API int tasq_plan_tc(int kind, int M, int N, int K, int B, int H, int W, int Cin, int num_sms,
                          tasq_tc_plan* out) {
    const tasq_ctx ctx = nullptr;  // host-only call: errors go to tasq_last_error(NULL)
    REQUIRE(out, TASQ_ERR_INVALID_ARG, "out is NULL");
    *out = tasq_tc_plan{};
    REQUIRE(kind == TASQ_LINEAR || kind == TASQ_CONV3X3, TASQ_ERR_INVALID_ARG, "kind %d", kind);
    REQUIRE(num_sms > 0, TASQ_ERR_INVALID_ARG, "num_sms=%d", num_sms);
    if (kind == TASQ_CONV3X3) {
        // the checks of tasq_masked_conv3x3
        REQUIRE(B >= 0 && H > 0 && W > 0 && Cin > 0, TASQ_ERR_INVALID_ARG, "B=%d H=%d W=%d Cin=%d", B, H, W, Cin);
        REQUIRE(Cin % 16 == 0, TASQ_ERR_UNSUPPORTED, "conv: Cin=%d must be a multiple of 16", Cin);
        REQUIRE((int64_t)B * H * W <= 0x7FFFFFFF && (int64_t)9 * Cin <= 0x7FFFFFFF, TASQ_ERR_UNSUPPORTED,
                "too large");
        M = B * H * W;
        K = 9 * Cin;
    } else {
        B = 1;
        H = W = Cin = 0;
    }
    // the checks every contraction call makes
    REQUIRE(M >= 0 && N > 0 && K > 0, TASQ_ERR_INVALID_ARG, "M=%d N=%d K=%d", M, N, K);
    REQUIRE(K % 16 == 0 && N % 8 == 0, TASQ_ERR_UNSUPPORTED, "need K %% 16 == 0 and N %% 8 == 0 (N=%d K=%d)", N, K);
    const tasq::TcPlan p =
        tasq::plan_gemm_tc(M, N, K, B, H, W, Cin, num_sms, tasq::kSplitBufBytes / int64_t(sizeof(int32_t)));
    REQUIRE(!p.why, TASQ_ERR_UNSUPPORTED, "tensor-core route: %s", p.why);
    out->tile_channels = p.bch;
    out->tiles_ch = p.tiles_ch;
    if (M == 0) return TASQ_OK;
    out->tile_tokens = p.bt;
    out->acc_buffers = p.nacc;
    out->tiles_tok = p.tiles_tok;
    if (Cin) {
        out->box_rows = p.bhx;
        out->box_cols = 1 << p.bw_log2;
    }
    out->splits = p.splits;
    out->grid = p.grid;
    out->reduce_grid = p.reduce_grid;
    out->kernels = p.splits > 1 ? 2 : 1;
    return TASQ_OK;
}
