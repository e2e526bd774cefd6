// Internal declarations shared by the libhc translation units: the device
// status word, the per-device context, the row/neighbour index logic of the
// sparse operators, and thin inline-PTX wrappers for sm_103a (cp.async,
// mbarrier, tcgen05). Nothing here is part of the public ABI (include/hc.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "hc.h"

namespace hc {

// ------------------------------------------------------------ status bits
// Device kernels OR one of these into the per-device status word.
enum : unsigned {
    kErrCapacity = 1u << HC_ERR_CAPACITY,
    kErrIndex = 1u << HC_ERR_INVALID_INDEX,
    kErrTimeout = 1u << HC_ERR_TIMEOUT,
};

// Longest a kernel waits on any one barrier before it gives up, records
// HC_ERR_TIMEOUT and unwinds (nanoseconds of %globaltimer). A test may lower
// the limit of the pipeline waits on a device (hc_test_set_option); the
// waits of an unwind, for copies and MMAs already issued, always keep it.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// The per-device word kernels report into (`status` in every kernel's
// arguments points at its first member), with the pipeline-wait limit
// beside it so that kernels read it through the same pointer.
struct DeviceWord {
    unsigned status;                   // sticky kErr* bits
    unsigned reserved;
    unsigned long long wait_limit_ns;  // kWaitLimitNs unless a test lowered it
};

// Path choices that only the library's tests override (hc_test_set_option).
int test_group_norm_path();  // 0 automatic, 1 per-(frame, group) kernel, 2 row ranges

// ------------------------------------------------------------ host context
struct DeviceCtx {
    int device;
    int num_sms;
    unsigned* status;  // device address of the sticky status word
};

// Context of the current device (cached); nullptr after recording an error.
const DeviceCtx* device_ctx();
void set_error(const char* fmt, ...);
hc_status check_cuda(cudaError_t e, const char* what);
// Per-(device, stream) scratch of at least `bytes`, grown on demand and kept
// until exit. nullptr after recording an error.
void* stream_workspace(cudaStream_t s, size_t bytes);

// ------------------------------------------------------------ operator modes
enum RowMode : int {
    kSparseDenseX = 0,    // rows = coords[0..count); input rows at b*V+u
    kSparseCompactX = 1,  // rows = coords[0..count); input rows at row_of[b*V+u]
    kDense = 2,           // rows = all b*V+v; input rows at b*V+u
    kLinear = 3,          // rows = 0..count; input row = output row; L = 1
    kRulebook = 4,        // rows = 0..count; input rows from a precomputed rulebook
};

struct ConvArgs {
    const void* x;
    const int32_t* coords;
    const int32_t* row_of;
    const int32_t* count;  // device N' (sparse/linear), unused for dense
    const int32_t* spiral;
    const void* W;
    const float* bias;
    void* y;
    unsigned* status;
    long long capacity;  // upper bound on rows (B*V, or the linear capacity)
    long long x_rows;    // rows of the input x (valid input row indices are < x_rows)
    const int32_t* rulebook;  // kRulebook: [L, capacity] slot-major tap rows, -1 = absent
    // Optional fused scatter (Eq. 2 inverse): row n is also written to
    // out_dense[(b*out_V + v)*C_out ...] with (b, v) = out_coords[n].
    void* out_dense;
    const int32_t* out_coords;
    int out_B, out_V;
    int B, V, L, C_in, C_out, K;  // K = L*C_in
    int mode;
    int act;
    int stages;  // pipeline depth chosen by the launcher (tensor-core kernel)
    int stages_tr;  // the row-count-dispatched kernel's depth for two-half items
    int w3d;     // tensor-core kernel: W's tensor map is the 3-D view (one box per stage)
    // Optional group-norm statistics of the stored output (Eqs. 7-9,
    // tensor-core kernel): every block c of 32 output rows writes, for each
    // frame b among its rows (b = gn_coords[2n]) and each channel group g of
    // gn_G, the (count, mean, M2) of its stored values to
    // gn_part[4 * ((b + c) * gn_G + g)].
    // Blocks whose rows are not all active and in one frame write, instead,
    // every active row's (mean, M2) of each group (gn_C / gn_G values) to
    // gn_rows[2 * (row * gn_G + g)].
    float* gn_part;
    float* gn_rows;
    const int32_t* gn_coords;
    int gn_G, gn_B;
    int gn_cpg;  // channels per group, C_out / gn_G: 8, 16, 32, 64 or 128
    // Host-side estimate of the active row count (rulebook mode; 0 =
    // unknown): it only chooses the tensor-core kernel's item shape.
    long long rows_hint;
    // Tensor-core kernel with C_in not a multiple of 8: workspace of at
    // least conv_tc_pad_bytes(a) bytes (256-byte aligned) for x and W with
    // zero channels appended up to a multiple of 8.
    void* pad_ws;
};

// Launchers (each in its own translation unit). All return HC_OK or an
// error already recorded with set_error().
hc_status launch_compact(const DeviceCtx* ctx, const uint8_t* mask, int B, int V, int32_t* coords,
                         int32_t* row_of, int32_t* offsets, int32_t* count, cudaStream_t s);
hc_status launch_conv_simt(const DeviceCtx* ctx, const ConvArgs& a, hc_dtype dt, cudaStream_t s);
hc_status launch_conv_tc(const DeviceCtx* ctx, const ConvArgs& a, cudaStream_t s);
bool conv_tc_supported(const ConvArgs& a, hc_dtype dt);
int conv_tc_tile_n(const ConvArgs& a);  // output channels per tensor-core tile
size_t conv_tc_pad_bytes(const ConvArgs& a);  // 0 when C_in % 8 == 0
// Compaction fused with the Eq. 4 mapping (frames of at most 65535 vertices).
bool compact_map_supported(int B, int V, int L);
hc_status launch_compact_map(const DeviceCtx* ctx, const uint8_t* mask, int B, int V,
                             const int32_t* spiral, int L, int x_layout, int32_t* coords,
                             int32_t* row_of, int32_t* offsets, int32_t* count, int32_t* rulebook,
                             cudaStream_t s);
hc_status launch_rulebook(const DeviceCtx* ctx, const int32_t* coords, const int32_t* row_of,
                          const int32_t* count, const int32_t* spiral, int B, int V, int L,
                          int x_layout, int32_t* rulebook, cudaStream_t s);
hc_status launch_group_norm(const DeviceCtx* ctx, const void* x, hc_dtype dt,
                            const int32_t* offsets, int B, long long capacity, int C, int G,
                            float eps, const float* gamma, const float* beta, int act, void* y,
                            cudaStream_t s);
// The normalising pass alone, in place on bf16 y, from the partials the
// convolution wrote for the rows [0, *count): one per (frame, part_rows-row
// block lying inside the frame, group) in part, and one per (row, group) in
// rows for the other rows. The frame table must start at 0 and end at *count.
bool group_norm_parts_supported(hc_dtype dt, int C, int G, const void* y);
hc_status launch_group_norm_apply(const DeviceCtx* ctx, void* y, const int32_t* offsets, int B,
                                  long long capacity, int C, int G, const float* part,
                                  const float* rows, int part_rows, const int32_t* count,
                                  float eps, const float* gamma, const float* beta, int act,
                                  cudaStream_t s);
// Backward of the sparse conv through a rulebook (see bwd.cu).
struct BwdArgs {
    const void* x;
    hc_dtype dt;
    int x_rows;
    const int32_t* rulebook;  // [L, capacity]
    const int32_t* count;
    int capacity;
    int L, C_in, C_out;
    const void* W;
    const void* y;
    const void* dy;
    int act;
    const int32_t* row_ptr;  // transposed mapping (needed for dx)
    const int32_t* taps;
    void* dx;
    float* dW;
    float* dbias;
};
hc_status dispatch_conv(const DeviceCtx* ctx, ConvArgs& a, hc_dtype dt, cudaStream_t s);
hc_status launch_conv_bwd(const DeviceCtx* ctx, const BwdArgs& b, cudaStream_t s);
hc_status launch_rulebook_transpose(const DeviceCtx* ctx, const int32_t* rb, const int32_t* count,
                                    int capacity, int L, int x_rows, int32_t* ptr, int32_t* taps,
                                    cudaStream_t s);
hc_status launch_mask_score(const DeviceCtx* ctx, const void* O, hc_dtype dt, int K, long long N,
                            int D, const float* alpha_in, float* alpha_out, float* sim,
                            cudaStream_t s);
hc_status launch_topk(const DeviceCtx* ctx, const float* alpha, int K, int kappa, int32_t* selected,
                      cudaStream_t s);
hc_status launch_kappa_masks(const DeviceCtx* ctx, const uint8_t* masks, int K, int V,
                             const int32_t* selected, int kappa, int B, uint8_t* out,
                             cudaStream_t s);
hc_status launch_gather_rows(const DeviceCtx* ctx, const void* x, int elem_bytes, int B_in, int V,
                             int C, const int32_t* coords, const int32_t* count, int capacity,
                             int frames_per_sample, void* y, cudaStream_t s);
hc_status launch_scatter(const DeviceCtx* ctx, const void* y, int elem_bytes, const int32_t* coords,
                         const int32_t* row_of, const int32_t* count, int B, int V, int C,
                         int zero_fill, void* out, cudaStream_t s);

// ------------------------------------------------------------ launches
// Every kernel of the library is launched with programmatic stream
// serialisation: it may be scheduled while the previous kernel on the stream
// is still finishing, runs its on-chip prologue, and waits (pdl_wait) for
// the previous grid to complete before its first global-memory access.
#if defined(__CUDACC__)
template <typename... KArgs, typename... Args>
hc_status launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t s, const char* what, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return check_cuda(cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...), what);
}
#endif

// ------------------------------------------------------------ device helpers
#if defined(__CUDACC__)

// Wait until the previous grid on the stream has completed and its writes are
// visible (a no-op without a programmatic dependency), then allow the next
// grid to be scheduled early.
__device__ __forceinline__ void pdl_wait() {
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
}
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

__device__ __forceinline__ void report(unsigned* status, unsigned bit) {
    atomicOr(status, bit);
}

// Number of output rows of this call: N' from the device count (clamped to
// the capacity, which is reported), or every grid row for the dense layer.
__device__ __forceinline__ long long active_rows(const ConvArgs& a) {
    if (a.mode == kDense) return (long long)a.B * a.V;
    long long n = *a.count;
    if (n < 0) {
        report(a.status, kErrIndex);
        return 0;
    }
    if (n > a.capacity) {
        report(a.status, kErrCapacity);
        n = a.capacity;
    }
    return n;
}

// The helpers below never write memory: they return an error bit instead
// (kErrIndex), which callers OR together and report once. A global atomic
// between loads would stop the compiler from issuing the loads of many taps
// back to back.

// Activation of Eq. 10. ELU(z) = z for z > 0, else exp(z) - 1, written
// without a branch as max(z, 0) + (exp(min(z, 0)) - 1): for z > 0 the second
// term is exp(0) - 1 = 0 exactly. The fast exponential's absolute error is a
// few 1e-7, far inside the fp32 (1e-4 absolute) and bf16 (2e-2 relative)
// tolerances of this library.
template <int ACT>
__device__ __forceinline__ float act_fixed(float z) {
    if (ACT == HC_ACT_ELU) return fmaxf(z, 0.f) + (__expf(fminf(z, 0.f)) - 1.0f);
    if (ACT == HC_ACT_RELU) return fmaxf(z, 0.f);
    return z;
}
__device__ __forceinline__ float act_apply(float z, int act) {
    if (act == HC_ACT_ELU) return act_fixed<HC_ACT_ELU>(z);
    if (act == HC_ACT_RELU) return act_fixed<HC_ACT_RELU>(z);
    return z;
}

// Explicit shared-memory accesses (32-bit shared addresses).
__device__ __forceinline__ int lds_s32(uint32_t addr) {
    int v;
    asm volatile("ld.shared.b32 %0, [%1];\n" : "=r"(v) : "r"(addr));
    return v;
}
__device__ __forceinline__ void sts_s32(uint32_t addr, int v) {
    asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(addr), "r"(v) : "memory");
}

// q = a / d and r = a - q * d for a >= 0, d > 0: 32-bit division when a
// fits (a 64-bit division is a long subroutine), 64-bit otherwise.
__device__ __forceinline__ long long div32(long long a, int d, int& r) {
    if (a < (1ll << 31)) {
        const unsigned q = (unsigned)a / (unsigned)d;
        r = (int)((unsigned)a - q * (unsigned)d);
        return q;
    }
    const long long q = a / d;
    r = (int)(a - q * d);
    return q;
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

// ---- cp.async (16 bytes, zero-filled when !valid)
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src, bool valid) {
    uint32_t n = valid ? 16u : 0u;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(n)
                 : "memory");
}
// 4 bytes, zero-filled when !valid (both addresses 4-byte aligned).
__device__ __forceinline__ void cp_async_4(uint32_t dst, const void* src, bool valid) {
    uint32_t n = valid ? 4u : 0u;
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(dst), "l"(src), "r"(n)
                 : "memory");
}
// Arrive on `bar` once every cp.async issued so far by this thread has
// completed (the arrival is not counted in advance: the barrier's expected
// count includes it).
__device__ __forceinline__ void cp_async_arrive_noinc(uint32_t bar) {
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.wait_all;\n" ::: "memory");
}

// Make this thread's generic-proxy shared-memory writes visible to the
// async proxy (tcgen05.mma operand reads).
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}

// ---- mbarrier
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n"
        " mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase with the given parity for at most `limit` ns. On
// timeout (or, with an abort flag, when another role already gave up) it
// records HC_ERR_TIMEOUT, raises the flag and returns false.
__device__ __forceinline__ bool mbar_wait_for(uint32_t bar, uint32_t parity,
                                              volatile int* abort_flag, unsigned* status,
                                              unsigned long long limit) {
    // try_wait itself may suspend the thread for a while, so the clock and
    // the abort flag are read after every unsuccessful try
    const unsigned long long t0 = globaltimer_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (abort_flag && *abort_flag) return false;
        if (globaltimer_ns() - t0 > limit) {
            if (abort_flag) *abort_flag = 1;
            report(status, kErrTimeout);
            return false;
        }
    }
}
// A pipeline wait: bounded by the device's wait limit (kWaitLimitNs unless a
// test lowered it), abandoned when another role of the CTA gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned* status) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long limit =
        reinterpret_cast<const volatile DeviceWord*>(status)->wait_limit_ns;
    return mbar_wait_for(bar, parity, abort_flag, status, limit);
}
// A wait of the unwind, for copies or MMAs already issued: always the full
// limit, regardless of the abort flag.
__device__ __forceinline__ bool mbar_wait_drain(uint32_t bar, uint32_t parity, unsigned* status) {
    if (mbar_try_wait(bar, parity)) return true;
    return mbar_wait_for(bar, parity, nullptr, status, kWaitLimitNs);
}

// ---- TMA (bulk tensor copies global -> shared, completion on an mbarrier)
// Arrive on `bar` and add `bytes` to the transaction count its phase waits for.
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes)
                 : "memory");
}
// 2-D tiled load of the tensor map's box at (c0 = inner, c1 = outer).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int c0, int c1,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];\n" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}
// 3-D tiled load of the tensor map's box at (c0, c1, c2), innermost first.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tmap, int c0, int c1, int c2,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];\n" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void prefetch_tensormap(const void* tmap) {
    asm volatile("prefetch.tensormap [%0];\n" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}
__device__ __forceinline__ void sts_v4(uint32_t addr, uint4 v) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ uint4 lds_u4(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}

// ---- tcgen05 (5th-generation tensor cores, accumulators in TMEM)
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(dst_smem),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem], kind::f16 (bf16 inputs, fp32 accumulate).
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive once on `bar` when every tcgen05 op issued so far by this thread
// has completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
        : "memory");
}
// 32 lanes x 32 consecutive fp32 columns: thread i of the warp receives
// lane (base lane + i), columns [col, col+32).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
}
// Lane i writes its 32 registers to TMEM lane (warp's quarter) + i,
// columns taddr.col .. + 31.
__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),
          "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]),
          "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]),
          "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
          "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

#endif  // __CUDACC__

}  // namespace hc
