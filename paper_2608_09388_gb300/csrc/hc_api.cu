// C ABI of libhc (include/hc.h): host-side argument checks, the per-device
// context and status word, the per-stream workspace, and dispatch to the
// kernels. Every entry point validates before it launches anything.
#include <cuda_runtime.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <map>
#include <mutex>
#include <utility>

#include "hc_internal.cuh"

namespace hc {

// Sticky per-device status word (kernels OR kErr* bits into it) and the
// pipeline-wait limit the kernels read beside it.
__device__ DeviceWord g_device_word = {0u, 0u, kWaitLimitNs};

// Group-norm path forced by a test (hc_test_set_option), 0 = automatic.
static std::atomic<int> g_test_gn_path{0};
int test_group_norm_path() {
    return g_test_gn_path.load(std::memory_order_relaxed);
}

static thread_local char t_last_error[512];

void set_error(const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_last_error, sizeof t_last_error, fmt, ap);
    va_end(ap);
}

hc_status check_cuda(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return HC_OK;
    set_error("%s: %s", what, cudaGetErrorString(e));
    return HC_ERR_CUDA;
}

static constexpr int kMaxDevices = 64;
static DeviceCtx g_ctx[kMaxDevices];
static bool g_ctx_ready[kMaxDevices];
static std::mutex g_ctx_mutex;

const DeviceCtx* device_ctx() {
    int dev = -1;
    if (check_cuda(cudaGetDevice(&dev), "cudaGetDevice") != HC_OK) return nullptr;
    if (dev < 0 || dev >= kMaxDevices) {
        set_error("device ordinal %d out of range", dev);
        return nullptr;
    }
    std::lock_guard<std::mutex> lock(g_ctx_mutex);
    if (!g_ctx_ready[dev]) {
        DeviceCtx c;
        c.device = dev;
        if (check_cuda(cudaDeviceGetAttribute(&c.num_sms, cudaDevAttrMultiProcessorCount, dev),
                       "cudaDeviceGetAttribute") != HC_OK)
            return nullptr;
        void* p = nullptr;
        if (check_cuda(cudaGetSymbolAddress(&p, g_device_word), "cudaGetSymbolAddress") != HC_OK)
            return nullptr;
        c.status = &static_cast<DeviceWord*>(p)->status;
        g_ctx[dev] = c;
        g_ctx_ready[dev] = true;
    }
    return &g_ctx[dev];
}

struct Workspace {
    void* ptr = nullptr;
    size_t bytes = 0;
};
static std::map<std::pair<int, cudaStream_t>, Workspace> g_ws;
static std::mutex g_ws_mutex;

void* stream_workspace(cudaStream_t s, size_t bytes) {
    int dev = -1;
    if (check_cuda(cudaGetDevice(&dev), "cudaGetDevice") != HC_OK) return nullptr;
    std::lock_guard<std::mutex> lock(g_ws_mutex);
    Workspace& w = g_ws[std::make_pair(dev, s)];
    if (w.bytes >= bytes) return w.ptr;
    size_t want = bytes < 4096 ? 4096 : bytes;
    if (w.ptr) {
        // The old buffer may still be read by work queued on this stream.
        if (check_cuda(cudaStreamSynchronize(s), "cudaStreamSynchronize") != HC_OK) return nullptr;
        cudaFree(w.ptr);
        w.ptr = nullptr;
        w.bytes = 0;
    }
    void* p = nullptr;
    if (check_cuda(cudaMalloc(&p, want), "cudaMalloc(workspace)") != HC_OK) return nullptr;
    w.ptr = p;
    w.bytes = want;
    return p;
}

static bool misaligned(const void* p, size_t a) {
    return ((uintptr_t)p) % a != 0;
}

// Conv kernels: tensor cores when supported (bf16, 16-byte aligned rows),
// CUDA cores otherwise.
hc_status dispatch_conv(const DeviceCtx* ctx, ConvArgs& a, hc_dtype dt, cudaStream_t s) {
    a.status = ctx->status;
    if (conv_tc_supported(a, dt)) {
        if (const size_t pb = conv_tc_pad_bytes(a)) {
            a.pad_ws = stream_workspace(s, pb);
            if (!a.pad_ws) return HC_ERR_CUDA;
        }
        return launch_conv_tc(ctx, a, s);
    }
    return launch_conv_simt(ctx, a, dt, s);
}

}  // namespace hc

using namespace hc;

#define HC_REQUIRE(cond, ...)             \
    do {                                  \
        if (!(cond)) {                    \
            set_error(__VA_ARGS__);       \
            return HC_ERR_INVALID_ARG;    \
        }                                 \
    } while (0)

extern "C" {

const char* hc_last_error_string(void) {
    return t_last_error;
}

const char* hc_version(void) {
    return "0.1.0";
}

hc_status hc_mask_compact(const uint8_t* mask, int B, int V, int32_t* coords, int32_t* row_of,
                          int32_t* batch_offsets, int32_t* count, hc_stream_t stream) {
    t_last_error[0] = 0;
    HC_REQUIRE(B >= 0 && V >= 0, "hc_mask_compact: B=%d V=%d must be >= 0", B, V);
    HC_REQUIRE((long long)B * V < (1ll << 31), "hc_mask_compact: B*V must be < 2^31");
    HC_REQUIRE(count != nullptr, "hc_mask_compact: count is NULL");
    HC_REQUIRE((long long)B * V == 0 || (mask && coords),
               "hc_mask_compact: mask and coords are required");
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_compact(ctx, mask, B, V, coords, row_of, batch_offsets, count,
                          (cudaStream_t)stream);
}

static hc_status check_conv_common(const char* fn, hc_dtype dt, int L, int C_in, int C_out,
                                   hc_act act, const void* x, const void* W, void* y) {
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(act == HC_ACT_NONE || act == HC_ACT_ELU || act == HC_ACT_RELU,
               "%s: unknown activation %d", fn, (int)act);
    HC_REQUIRE(C_in >= 1 && C_out >= 1, "%s: C_in=%d C_out=%d must be >= 1", fn, C_in, C_out);
    HC_REQUIRE(L >= 1, "%s: L=%d must be >= 1", fn, L);
    if (L > HC_MAX_SPIRAL) {
        set_error("%s: L=%d exceeds HC_MAX_SPIRAL=%d", fn, L, HC_MAX_SPIRAL);
        return HC_ERR_UNSUPPORTED;
    }
    HC_REQUIRE((long long)L * C_in < (1ll << 31), "%s: L*C_in too large", fn);
    HC_REQUIRE(x && W && y, "%s: x, W and y are required", fn);
    size_t eb = dt == HC_F32 ? 4 : 2;
    HC_REQUIRE(!misaligned(x, eb) && !misaligned(W, eb) && !misaligned(y, eb),
               "%s: x, W, y must be aligned to the element size", fn);
    return HC_OK;
}

hc_status hc_sparse_spiral_conv_fwd(const void* x, hc_layout x_layout, hc_dtype dt,
                                    const int32_t* coords, const int32_t* row_of,
                                    const int32_t* count, const int32_t* spiral, int B, int V,
                                    int L, int C_in, int C_out, const void* W, const float* bias,
                                    hc_act act, void* y, hc_stream_t stream) {
    const char* fn = "hc_sparse_spiral_conv_fwd";
    t_last_error[0] = 0;
    hc_status st = check_conv_common(fn, dt, L, C_in, C_out, act, x, W, y);
    if (st != HC_OK) return st;
    HC_REQUIRE(x_layout == HC_LAYOUT_DENSE || x_layout == HC_LAYOUT_COMPACT,
               "%s: unknown layout %d", fn, (int)x_layout);
    HC_REQUIRE(B >= 0 && V >= 0, "%s: B=%d V=%d must be >= 0", fn, B, V);
    HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
    HC_REQUIRE(coords && row_of && count && spiral, "%s: coords, row_of, count, spiral required",
               fn);
    if ((long long)B * V == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    ConvArgs a{};
    a.x = x;
    a.coords = coords;
    a.row_of = row_of;
    a.count = count;
    a.spiral = spiral;
    a.W = W;
    a.bias = bias;
    a.y = y;
    a.capacity = (long long)B * V;
    a.x_rows = (long long)B * V;
    a.B = B;
    a.V = V;
    a.L = L;
    a.C_in = C_in;
    a.C_out = C_out;
    a.K = L * C_in;
    a.mode = x_layout == HC_LAYOUT_DENSE ? kSparseDenseX : kSparseCompactX;
    a.act = act;
    return dispatch_conv(ctx, a, dt, (cudaStream_t)stream);
}

hc_status hc_sparse_linear_fwd(const void* x, hc_dtype dt, const int32_t* count, int capacity,
                               int C_in, int C_out, const void* W, const float* bias, hc_act act,
                               void* y, hc_stream_t stream) {
    const char* fn = "hc_sparse_linear_fwd";
    t_last_error[0] = 0;
    hc_status st = check_conv_common(fn, dt, 1, C_in, C_out, act, x, W, y);
    if (st != HC_OK) return st;
    HC_REQUIRE(capacity >= 0, "%s: capacity=%d must be >= 0", fn, capacity);
    HC_REQUIRE(count != nullptr, "%s: count is NULL", fn);
    if (capacity == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    ConvArgs a{};
    a.x = x;
    a.count = count;
    a.W = W;
    a.bias = bias;
    a.y = y;
    a.capacity = capacity;
    a.x_rows = capacity;
    a.B = 1;
    a.V = capacity;
    a.L = 1;
    a.C_in = C_in;
    a.C_out = C_out;
    a.K = C_in;
    a.mode = kLinear;
    a.act = act;
    return dispatch_conv(ctx, a, dt, (cudaStream_t)stream);
}

hc_status hc_spiral_conv_fwd(const void* x, hc_dtype dt, const int32_t* spiral, int B, int V,
                             int L, int C_in, int C_out, const void* W, const float* bias,
                             hc_act act, void* y, hc_stream_t stream) {
    const char* fn = "hc_spiral_conv_fwd";
    t_last_error[0] = 0;
    hc_status st = check_conv_common(fn, dt, L, C_in, C_out, act, x, W, y);
    if (st != HC_OK) return st;
    HC_REQUIRE(B >= 0 && V >= 0, "%s: B=%d V=%d must be >= 0", fn, B, V);
    HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
    HC_REQUIRE(spiral != nullptr, "%s: spiral is NULL", fn);
    if ((long long)B * V == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    ConvArgs a{};
    a.x = x;
    a.spiral = spiral;
    a.W = W;
    a.bias = bias;
    a.y = y;
    a.capacity = (long long)B * V;
    a.x_rows = (long long)B * V;
    a.B = B;
    a.V = V;
    a.L = L;
    a.C_in = C_in;
    a.C_out = C_out;
    a.K = L * C_in;
    a.mode = kDense;
    a.act = act;
    return dispatch_conv(ctx, a, dt, (cudaStream_t)stream);
}

hc_status hc_conv_rulebook(const int32_t* coords, const int32_t* row_of, const int32_t* count,
                           const int32_t* spiral, int B, int V, int L, hc_layout x_layout,
                           int32_t* rulebook, hc_stream_t stream) {
    const char* fn = "hc_conv_rulebook";
    t_last_error[0] = 0;
    HC_REQUIRE(B >= 0 && V >= 0, "%s: B=%d V=%d must be >= 0", fn, B, V);
    HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
    HC_REQUIRE(L >= 1, "%s: L=%d must be >= 1", fn, L);
    if (L > HC_MAX_SPIRAL) {
        set_error("%s: L=%d exceeds HC_MAX_SPIRAL=%d", fn, L, HC_MAX_SPIRAL);
        return HC_ERR_UNSUPPORTED;
    }
    HC_REQUIRE(x_layout == HC_LAYOUT_DENSE || x_layout == HC_LAYOUT_COMPACT,
               "%s: unknown layout %d", fn, (int)x_layout);
    HC_REQUIRE(coords && row_of && count && spiral && rulebook,
               "%s: coords, row_of, count, spiral and rulebook are required", fn);
    if ((long long)B * V == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_rulebook(ctx, coords, row_of, count, spiral, B, V, L, (int)x_layout, rulebook,
                           (cudaStream_t)stream);
}

hc_status hc_mask_compact_rulebook(const uint8_t* mask, int B, int V, const int32_t* spiral, int L,
                                   hc_layout x_layout, int32_t* coords, int32_t* row_of,
                                   int32_t* batch_offsets, int32_t* count, int32_t* rulebook,
                                   hc_stream_t stream) {
    const char* fn = "hc_mask_compact_rulebook";
    t_last_error[0] = 0;
    HC_REQUIRE(B >= 0 && V >= 0, "%s: B=%d V=%d must be >= 0", fn, B, V);
    HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
    HC_REQUIRE(L >= 1, "%s: L=%d must be >= 1", fn, L);
    if (L > HC_MAX_SPIRAL) {
        set_error("%s: L=%d exceeds HC_MAX_SPIRAL=%d", fn, L, HC_MAX_SPIRAL);
        return HC_ERR_UNSUPPORTED;
    }
    HC_REQUIRE(x_layout == HC_LAYOUT_DENSE || x_layout == HC_LAYOUT_COMPACT,
               "%s: unknown layout %d", fn, (int)x_layout);
    HC_REQUIRE(count != nullptr, "%s: count is NULL", fn);
    HC_REQUIRE((long long)B * V == 0 || (mask && spiral && coords && row_of && rulebook),
               "%s: mask, spiral, coords, row_of and rulebook are required", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    const cudaStream_t s = (cudaStream_t)stream;
    if ((long long)B * V > 0 && compact_map_supported(B, V, L))
        return launch_compact_map(ctx, mask, B, V, spiral, L, (int)x_layout, coords, row_of,
                                  batch_offsets, count, rulebook, s);
    hc_status st = launch_compact(ctx, mask, B, V, coords, row_of, batch_offsets, count, s);
    if (st != HC_OK || (long long)B * V == 0) return st;
    return launch_rulebook(ctx, coords, row_of, count, spiral, B, V, L, (int)x_layout, rulebook, s);
}

}  // extern "C"

static hc_status conv_rulebook(const char* fn, const void* x, hc_dtype dt, int x_rows,
                               const int32_t* rulebook, const int32_t* count, int capacity, int L,
                               int C_in, int C_out, const void* W, const float* bias, hc_act act,
                               void* y, const int32_t* coords, int B, int V, void* out,
                               long long rows_hint, cudaStream_t stream) {
    HC_REQUIRE(y || out, "%s: at least one of y and out is required", fn);
    hc_status st = check_conv_common(fn, dt, L, C_in, C_out, act, x, W, y ? y : out);
    if (st != HC_OK) return st;
    HC_REQUIRE(x_rows >= 1 && capacity >= 0, "%s: x_rows=%d capacity=%d", fn, x_rows, capacity);
    HC_REQUIRE(rulebook && count, "%s: rulebook and count are required", fn);
    if (out) {
        HC_REQUIRE(coords && B >= 1 && V >= 1, "%s: out needs coords, B >= 1 and V >= 1", fn);
        HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
        HC_REQUIRE(!misaligned(out, dt == HC_F32 ? 4 : 2), "%s: misaligned out", fn);
    }
    if (capacity == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    ConvArgs a{};
    a.x = x;
    a.count = count;
    a.rulebook = rulebook;
    a.W = W;
    a.bias = bias;
    a.y = y;
    a.capacity = capacity;
    a.x_rows = x_rows;
    a.B = 1;
    a.V = capacity;
    a.L = L;
    a.C_in = C_in;
    a.C_out = C_out;
    a.K = L * C_in;
    a.mode = kRulebook;
    a.act = act;
    a.out_dense = out;
    a.out_coords = coords;
    a.out_B = B;
    a.out_V = V;
    a.rows_hint = rows_hint;
    return dispatch_conv(ctx, a, dt, stream);
}

extern "C" {

hc_status hc_sparse_conv_rulebook_fwd(const void* x, hc_dtype dt, int x_rows,
                                      const int32_t* rulebook, const int32_t* count, int capacity,
                                      int L, int C_in, int C_out, const void* W, const float* bias,
                                      hc_act act, void* y, const int32_t* coords, int B, int V,
                                      void* out, hc_stream_t stream) {
    t_last_error[0] = 0;
    return conv_rulebook("hc_sparse_conv_rulebook_fwd", x, dt, x_rows, rulebook, count, capacity,
                         L, C_in, C_out, W, bias, act, y, coords, B, V, out, 0,
                         (cudaStream_t)stream);
}

hc_status hc_sparse_conv_rulebook_fwd_hint(const void* x, hc_dtype dt, int x_rows,
                                           const int32_t* rulebook, const int32_t* count,
                                           int capacity, int L, int C_in, int C_out,
                                           const void* W, const float* bias, hc_act act, void* y,
                                           const int32_t* coords, int B, int V, void* out,
                                           long long rows_hint, hc_stream_t stream) {
    const char* fn = "hc_sparse_conv_rulebook_fwd_hint";
    t_last_error[0] = 0;
    HC_REQUIRE(rows_hint >= 0, "%s: rows_hint=%lld must be >= 0", fn, rows_hint);
    return conv_rulebook(fn, x, dt, x_rows, rulebook, count, capacity, L, C_in, C_out, W, bias,
                         act, y, coords, B, V, out, rows_hint, (cudaStream_t)stream);
}

hc_status hc_sparse_group_norm_fwd(const void* x, hc_dtype dt, const int32_t* batch_offsets, int B,
                                   int capacity, int C, int G, float eps, const float* gamma,
                                   const float* beta, hc_act act, void* y, hc_stream_t stream) {
    const char* fn = "hc_sparse_group_norm_fwd";
    t_last_error[0] = 0;
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(act == HC_ACT_NONE || act == HC_ACT_ELU || act == HC_ACT_RELU,
               "%s: unknown activation %d", fn, (int)act);
    HC_REQUIRE(B >= 0 && capacity >= 0, "%s: B=%d capacity=%d must be >= 0", fn, B, capacity);
    HC_REQUIRE(C >= 1 && G >= 1 && C % G == 0, "%s: C=%d must be a multiple of G=%d >= 1", fn, C,
               G);
    HC_REQUIRE((long long)B * G < (1ll << 31), "%s: B*G=%lld too large", fn, (long long)B * G);
    HC_REQUIRE(eps >= 0.f, "%s: eps must be >= 0", fn);
    HC_REQUIRE(batch_offsets != nullptr, "%s: batch_offsets is NULL", fn);
    if (B == 0 || capacity == 0) return HC_OK;
    HC_REQUIRE(x && y, "%s: x and y are required", fn);
    const int eb = dt == HC_F32 ? 4 : 2;
    HC_REQUIRE(!misaligned(x, eb) && !misaligned(y, eb), "%s: misaligned x/y", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_group_norm(ctx, x, dt, batch_offsets, B, capacity, C, G, eps, gamma, beta,
                             (int)act, y, (cudaStream_t)stream);
}

hc_status hc_sparse_conv_gn_fwd(const void* x, hc_dtype dt, int x_rows, const int32_t* rulebook,
                                const int32_t* count, int capacity, int L, int C_in, int C_out,
                                const void* W, const float* bias, const int32_t* coords,
                                const int32_t* batch_offsets, int B, int G, float eps,
                                const float* gamma, const float* beta, hc_act act, void* y,
                                hc_stream_t stream) {
    const char* fn = "hc_sparse_conv_gn_fwd";
    t_last_error[0] = 0;
    hc_status st = check_conv_common(fn, dt, L, C_in, C_out, act, x, W, y);
    if (st != HC_OK) return st;
    HC_REQUIRE(x_rows >= 1 && capacity >= 0, "%s: x_rows=%d capacity=%d", fn, x_rows, capacity);
    HC_REQUIRE(rulebook && count && coords && batch_offsets,
               "%s: rulebook, count, coords and batch_offsets are required", fn);
    HC_REQUIRE(B >= 1 && G >= 1 && C_out % G == 0, "%s: B=%d >= 1 and C_out=%d a multiple of G=%d",
               fn, B, C_out, G);
    HC_REQUIRE((long long)B * G < (1ll << 31), "%s: B*G=%lld too large", fn, (long long)B * G);
    HC_REQUIRE(eps >= 0.f, "%s: eps must be >= 0", fn);
    if (capacity == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    ConvArgs a{};
    a.x = x;
    a.count = count;
    a.rulebook = rulebook;
    a.W = W;
    a.bias = bias;
    a.y = y;
    a.capacity = capacity;
    a.x_rows = x_rows;
    a.B = 1;
    a.V = capacity;
    a.L = L;
    a.C_in = C_in;
    a.C_out = C_out;
    a.K = L * C_in;
    a.mode = kRulebook;
    a.act = HC_ACT_NONE;  // the activation follows the normalisation
    a.status = ctx->status;
    const int cpg = C_out / G;
    // channels per group a power of two from 8 to the tile's width
    if (conv_tc_supported(a, dt) && cpg >= 8 && (cpg & (cpg - 1)) == 0 && cpg <= conv_tc_tile_n(a) &&
        group_norm_parts_supported(dt, C_out, G, y)) {
        // statistics from the convolution's epilogue: one partial per
        // (frame, 32-row block inside it) in slot frame + block, one per row
        // of the blocks that straddle a frame boundary
        const size_t slots = (size_t)B + ((size_t)capacity + 31) / 32;
        const size_t part_bytes = (16 * slots * (size_t)G + 255) / 256 * 256;
        const size_t rows_bytes = (8 * (size_t)capacity * (size_t)G + 255) / 256 * 256;
        const size_t pad_bytes = conv_tc_pad_bytes(a);
        char* ws = (char*)stream_workspace(s, part_bytes + rows_bytes + pad_bytes);
        if (!ws) return HC_ERR_CUDA;
        float* part = (float*)ws;
        float* rows = (float*)(ws + part_bytes);
        if (pad_bytes) a.pad_ws = ws + part_bytes + rows_bytes;
        a.gn_part = part;
        a.gn_rows = rows;
        a.gn_coords = coords;
        a.gn_G = G;
        a.gn_B = B;
        a.gn_cpg = cpg;
        st = launch_conv_tc(ctx, a, s);
        if (st != HC_OK) return st;
        return launch_group_norm_apply(ctx, y, batch_offsets, B, capacity, C_out, G, part, rows,
                                       32, count, eps, gamma, beta, (int)act, s);
    }
    st = dispatch_conv(ctx, a, dt, s);
    if (st != HC_OK) return st;
    return launch_group_norm(ctx, y, dt, batch_offsets, B, capacity, C_out, G, eps, gamma, beta,
                             (int)act, y, s);
}

hc_status hc_conv_rulebook_transpose(const int32_t* rulebook, const int32_t* count, int capacity,
                                     int L, int x_rows, int32_t* row_ptr, int32_t* taps,
                                     hc_stream_t stream) {
    const char* fn = "hc_conv_rulebook_transpose";
    t_last_error[0] = 0;
    HC_REQUIRE(L >= 1 && L <= HC_MAX_SPIRAL, "%s: L=%d must be in [1, %d]", fn, L, HC_MAX_SPIRAL);
    HC_REQUIRE(capacity >= 0 && x_rows >= 0, "%s: capacity=%d x_rows=%d must be >= 0", fn,
               capacity, x_rows);
    HC_REQUIRE((long long)capacity * L < (1ll << 31), "%s: capacity*L must be < 2^31", fn);
    HC_REQUIRE(rulebook && count && row_ptr && (taps || capacity == 0),
               "%s: rulebook, count, row_ptr and taps are required", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    if (x_rows == 0)
        return check_cuda(cudaMemsetAsync(row_ptr, 0, sizeof(int32_t), (cudaStream_t)stream),
                          "cudaMemsetAsync(row_ptr)");
    return launch_rulebook_transpose(ctx, rulebook, count, capacity, L, x_rows, row_ptr, taps,
                                     (cudaStream_t)stream);
}

hc_status hc_sparse_conv_rulebook_bwd(const void* x, hc_dtype dt, int x_rows,
                                      const int32_t* rulebook, const int32_t* count, int capacity,
                                      int L, int C_in, int C_out, const void* W, const void* y,
                                      const void* dy, hc_act act, const int32_t* row_ptr,
                                      const int32_t* taps, void* dx, float* dW, float* dbias,
                                      hc_stream_t stream) {
    const char* fn = "hc_sparse_conv_rulebook_bwd";
    t_last_error[0] = 0;
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(act == HC_ACT_NONE || act == HC_ACT_ELU || act == HC_ACT_RELU,
               "%s: unknown activation %d", fn, (int)act);
    HC_REQUIRE(C_in >= 1 && C_out >= 1 && L >= 1, "%s: L=%d C_in=%d C_out=%d must be >= 1", fn, L,
               C_in, C_out);
    if (L > HC_MAX_SPIRAL) {
        set_error("%s: L=%d exceeds HC_MAX_SPIRAL=%d", fn, L, HC_MAX_SPIRAL);
        return HC_ERR_UNSUPPORTED;
    }
    HC_REQUIRE(capacity >= 0 && x_rows >= 0, "%s: capacity=%d x_rows=%d must be >= 0", fn,
               capacity, x_rows);
    HC_REQUIRE((long long)capacity * L < (1ll << 31) && (long long)L * C_in < (1ll << 31),
               "%s: capacity*L and L*C_in must be < 2^31", fn);
    HC_REQUIRE(rulebook && count && y && dy, "%s: rulebook, count, y and dy are required", fn);
    HC_REQUIRE(!dW || x, "%s: x is required for dW", fn);
    HC_REQUIRE(!dx || (W && row_ptr && taps), "%s: W, row_ptr and taps are required for dx", fn);
    const size_t eb = dt == HC_F32 ? 4 : 2;
    HC_REQUIRE(!misaligned(x, eb) && !misaligned(W, eb) && !misaligned(y, eb) &&
                   !misaligned(dy, eb) && !misaligned(dx, eb),
               "%s: x, W, y, dy, dx must be aligned to the element size", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    if (capacity == 0) {  // no output rows: every gradient is zero
        hc_status st = HC_OK;
        if (dx && x_rows > 0)
            st = check_cuda(cudaMemsetAsync(dx, 0, eb * (size_t)x_rows * C_in, s), "cudaMemsetAsync");
        if (st == HC_OK && dW)
            st = check_cuda(cudaMemsetAsync(dW, 0, sizeof(float) * (size_t)L * C_in * C_out, s),
                            "cudaMemsetAsync");
        if (st == HC_OK && dbias)
            st = check_cuda(cudaMemsetAsync(dbias, 0, sizeof(float) * (size_t)C_out, s),
                            "cudaMemsetAsync");
        return st;
    }
    BwdArgs b{};
    b.x = x;
    b.dt = dt;
    b.x_rows = x_rows;
    b.rulebook = rulebook;
    b.count = count;
    b.capacity = capacity;
    b.L = L;
    b.C_in = C_in;
    b.C_out = C_out;
    b.W = W;
    b.y = y;
    b.dy = dy;
    b.act = (int)act;
    b.row_ptr = row_ptr;
    b.taps = taps;
    b.dx = x_rows > 0 ? dx : nullptr;
    b.dW = dW;
    b.dbias = dbias;
    return launch_conv_bwd(ctx, b, s);
}

hc_status hc_mask_score_update(const void* O, hc_dtype dt, int K, int N, int D,
                               const float* alpha_in, float* alpha_out, float* sim,
                               hc_stream_t stream) {
    const char* fn = "hc_mask_score_update";
    t_last_error[0] = 0;
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(K >= 1 && D >= 1 && N >= 0, "%s: K=%d D=%d must be >= 1, N=%d >= 0", fn, K, D, N);
    if ((long long)K * D > HC_MASK_SCORE_MAX_FEATURES) {
        set_error("%s: K*D=%lld above the supported %d", fn, (long long)K * D,
                  HC_MASK_SCORE_MAX_FEATURES);
        return HC_ERR_UNSUPPORTED;
    }
    HC_REQUIRE(alpha_in && alpha_out, "%s: alpha_in and alpha_out are required", fn);
    HC_REQUIRE(N == 0 || O != nullptr, "%s: O is NULL", fn);
    HC_REQUIRE(!misaligned(O, dt == HC_F32 ? 4 : 2), "%s: misaligned O", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_mask_score(ctx, O, dt, K, N, D, alpha_in, alpha_out, sim, (cudaStream_t)stream);
}

hc_status hc_mask_select_topk(const float* alpha, int K, int kappa, int32_t* selected,
                              hc_stream_t stream) {
    const char* fn = "hc_mask_select_topk";
    t_last_error[0] = 0;
    HC_REQUIRE(K >= 1 && K <= HC_TOPK_MAX_MASKS, "%s: K=%d must be in [1, %d]", fn, K,
               HC_TOPK_MAX_MASKS);
    HC_REQUIRE(kappa >= 0 && kappa <= K, "%s: kappa=%d must be in [0, K=%d]", fn, kappa, K);
    HC_REQUIRE(alpha && selected, "%s: alpha and selected are required", fn);
    if (kappa == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_topk(ctx, alpha, K, kappa, selected, (cudaStream_t)stream);
}

hc_status hc_kappa_masks(const uint8_t* masks, int K, int V, const int32_t* selected, int kappa,
                         int B, uint8_t* out, hc_stream_t stream) {
    const char* fn = "hc_kappa_masks";
    t_last_error[0] = 0;
    HC_REQUIRE(K >= 1 && V >= 0 && kappa >= 0 && B >= 0, "%s: K=%d V=%d kappa=%d B=%d", fn, K,
               V, kappa, B);
    HC_REQUIRE((long long)B * kappa * V < (1ll << 31), "%s: B*kappa*V must be < 2^31", fn);
    if ((long long)B * kappa * V == 0) return HC_OK;
    HC_REQUIRE(masks && selected && out, "%s: masks, selected and out are required", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_kappa_masks(ctx, masks, K, V, selected, kappa, B, out, (cudaStream_t)stream);
}

hc_status hc_gather_rows(const void* x, hc_dtype dt, int B_in, int V, int C, const int32_t* coords,
                         const int32_t* count, int capacity, int frames_per_sample, void* y,
                         hc_stream_t stream) {
    const char* fn = "hc_gather_rows";
    t_last_error[0] = 0;
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(B_in >= 0 && V >= 0 && C >= 1 && capacity >= 0 && frames_per_sample >= 1,
               "%s: B_in=%d V=%d C=%d capacity=%d frames_per_sample=%d", fn, B_in, V, C, capacity,
               frames_per_sample);
    HC_REQUIRE(count != nullptr, "%s: count is NULL", fn);
    if (capacity == 0) return HC_OK;
    HC_REQUIRE(x && y, "%s: x and y are required", fn);
    const int eb = dt == HC_F32 ? 4 : 2;
    HC_REQUIRE(!misaligned(x, eb) && !misaligned(y, eb), "%s: misaligned x/y", fn);
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_gather_rows(ctx, x, eb, B_in, V, C, coords, count, capacity, frames_per_sample,
                              y, (cudaStream_t)stream);
}

hc_status hc_scatter_dense(const void* y, hc_dtype dt, const int32_t* coords,
                           const int32_t* row_of, const int32_t* count, int B, int V, int C,
                           int zero_fill, void* out, hc_stream_t stream) {
    const char* fn = "hc_scatter_dense";
    t_last_error[0] = 0;
    HC_REQUIRE(dt == HC_F32 || dt == HC_BF16, "%s: unknown dtype %d", fn, (int)dt);
    HC_REQUIRE(B >= 0 && V >= 0 && C >= 1, "%s: B=%d V=%d C=%d", fn, B, V, C);
    HC_REQUIRE((long long)B * V < (1ll << 31), "%s: B*V must be < 2^31", fn);
    HC_REQUIRE(y && count && out, "%s: y, count and out are required", fn);
    HC_REQUIRE(coords != nullptr || (zero_fill && row_of != nullptr),
               "%s: coords are required (zero_fill may use row_of instead)", fn);
    int eb = dt == HC_F32 ? 4 : 2;
    HC_REQUIRE(!misaligned(y, eb) && !misaligned(out, eb), "%s: misaligned y/out", fn);
    if ((long long)B * V == 0) return HC_OK;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    return launch_scatter(ctx, y, eb, coords, row_of, count, B, V, C, zero_fill, out,
                          (cudaStream_t)stream);
}

hc_status hc_test_set_option(int option, long long value) {
    t_last_error[0] = 0;
    if (option == HC_TEST_GROUP_NORM_PATH) {
        HC_REQUIRE(value >= 0 && value <= 2, "hc_test_set_option: group-norm path %lld", value);
        g_test_gn_path.store((int)value, std::memory_order_relaxed);
        return HC_OK;
    }
    if (option == HC_TEST_WAIT_LIMIT_NS) {
        HC_REQUIRE(value >= 0, "hc_test_set_option: wait limit %lld ns", value);
        const DeviceCtx* ctx = device_ctx();
        if (!ctx) return HC_ERR_CUDA;
        const unsigned long long ns = value == 0 ? kWaitLimitNs : (unsigned long long)value;
        DeviceWord* word = reinterpret_cast<DeviceWord*>(ctx->status);
        return check_cuda(cudaMemcpy(&word->wait_limit_ns, &ns, sizeof ns, cudaMemcpyHostToDevice),
                          "set wait limit");
    }
    set_error("hc_test_set_option: unknown option %d", option);
    return HC_ERR_INVALID_ARG;
}

hc_status hc_get_device_status(hc_stream_t stream) {
    t_last_error[0] = 0;
    const DeviceCtx* ctx = device_ctx();
    if (!ctx) return HC_ERR_CUDA;
    if (check_cuda(cudaStreamSynchronize((cudaStream_t)stream), "cudaStreamSynchronize") != HC_OK)
        return HC_ERR_CUDA;
    unsigned word = 0, zero = 0;
    if (check_cuda(cudaMemcpy(&word, ctx->status, sizeof word, cudaMemcpyDeviceToHost),
                   "read device status") != HC_OK)
        return HC_ERR_CUDA;
    if (word == 0) return HC_OK;
    if (check_cuda(cudaMemcpy(ctx->status, &zero, sizeof zero, cudaMemcpyHostToDevice),
                   "clear device status") != HC_OK)
        return HC_ERR_CUDA;
    for (int code = HC_ERR_CAPACITY; code <= HC_ERR_TIMEOUT; ++code)
        if (word & (1u << code)) {
            set_error("device reported status word 0x%x", word);
            return (hc_status)code;
        }
    set_error("device reported unknown status word 0x%x", word);
    return HC_ERR_CUDA;
}

}  // extern "C"
