// Inference with kappa kept masks (Sec. 3.1, Sparse Mask Selection):
//   topk_kernel         the kappa masks with the highest score alpha
//                       (highest first; equal scores lowest index first; a
//                       NaN score ranks below every number)
//   kappa_masks_kernel  every kept mask applied to every sample: frame
//                       f = b * kappa + j is sample b under mask selected[j]
//   gather_rows_kernel  the feature matrix S' of Eq. 2: the input row of
//                       every active coordinate (f, v), frame f reading
//                       sample f / frames_per_sample; without coordinates,
//                       the first N' rows in order (a copy sized on the
//                       device)
#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kTopkThreads = 1024;

// a ranks before b (a at index ia, b at ib).
__device__ __forceinline__ bool ranks_before(float a, int ia, float b, int ib) {
    const bool na = a != a, nb = b != b;
    if (na != nb) return nb;          // a number ranks before NaN
    if (!na && a != b) return a > b;  // higher score first
    return ia < ib;                   // equal (or both NaN): lower index first
}

__global__ void __launch_bounds__(kTopkThreads)
    topk_kernel(const float* __restrict__ alpha, int K, int kappa, int32_t* __restrict__ selected) {
    extern __shared__ uint8_t taken[];  // K bytes
    __shared__ float s_v[kTopkThreads / 32];
    __shared__ int s_i[kTopkThreads / 32];
    pdl_wait();
    pdl_trigger();
    for (int k = threadIdx.x; k < K; k += kTopkThreads) taken[k] = 0;
    __syncthreads();
    for (int j = 0; j < kappa; ++j) {
        float bv = 0.f;
        int bi = -1;
        for (int k = threadIdx.x; k < K; k += kTopkThreads) {
            if (taken[k]) continue;
            const float v = alpha[k];
            if (bi < 0 || ranks_before(v, k, bv, bi)) {
                bv = v;
                bi = k;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (oi >= 0 && (bi < 0 || ranks_before(ov, oi, bv, bi))) {
                bv = ov;
                bi = oi;
            }
        }
        if ((threadIdx.x & 31) == 0) {
            s_v[threadIdx.x >> 5] = bv;
            s_i[threadIdx.x >> 5] = bi;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            float v = 0.f;
            int b = -1;
            for (int w = 0; w < kTopkThreads / 32; ++w)
                if (s_i[w] >= 0 && (b < 0 || ranks_before(s_v[w], s_i[w], v, b))) {
                    v = s_v[w];
                    b = s_i[w];
                }
            selected[j] = b;
            taken[b] = 1;
        }
        __syncthreads();
    }
}

__global__ void kappa_masks_kernel(const uint8_t* __restrict__ masks, int K, int V,
                                   const int32_t* __restrict__ selected, int kappa, long long B,
                                   uint8_t* __restrict__ out, unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long total = B * kappa * (long long)V;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        int v, j;
        const long long f = div32(e, V, v);
        div32(f, kappa, j);
        const int sel = __ldg(selected + j);
        uint8_t m = 0;
        if (sel >= 0 && sel < K)
            m = masks[(long long)sel * V + v];
        else if (v == 0)
            report(status, kErrIndex);
        out[e] = m;
    }
}

// Rows move in U-sized chunks (16, 4 or 2 bytes), cpr chunks per row.
template <typename U>
__global__ void gather_rows_kernel(const U* __restrict__ x, long long B_in, int V, int cpr,
                                   const int32_t* __restrict__ coords,
                                   const int32_t* __restrict__ count, long long capacity,
                                   int frames_per_sample, U* __restrict__ y, unsigned* status) {
    pdl_wait();
    pdl_trigger();
    long long rows = *count;
    if (rows < 0) {
        if (blockIdx.x == 0 && threadIdx.x == 0) report(status, kErrIndex);
        return;
    }
    if (rows > capacity) {
        if (blockIdx.x == 0 && threadIdx.x == 0) report(status, kErrCapacity);
        rows = capacity;
    }
    const long long total = rows * cpr;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        int c;
        const long long n = div32(i, cpr, c);
        if (!coords) {
            // rows in order: x viewed as B_in * V rows
            if (n >= B_in * V) {
                if (c == 0) report(status, kErrIndex);
                continue;
            }
            y[i] = x[i];
            continue;
        }
        const int f = __ldg(coords + 2 * n), v = __ldg(coords + 2 * n + 1);
        const long long b = f >= 0 ? f / frames_per_sample : -1;
        if (b < 0 || b >= B_in || v < 0 || v >= V) {
            if (c == 0) report(status, kErrIndex);
            continue;
        }
        y[i] = x[(b * V + v) * cpr + c];
    }
}

template <typename U>
hc_status launch_gather_typed(const DeviceCtx* ctx, const void* x, long long B_in, int V, int cpr,
                              const int32_t* coords, const int32_t* count, long long capacity,
                              int fps, void* y, cudaStream_t s) {
    long long blocks = (capacity * cpr + 255) / 256;
    const long long cap = (long long)ctx->num_sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    return launch_pdl(gather_rows_kernel<U>, dim3((unsigned)blocks), dim3(256), 0, s,
                      "gather_rows_kernel", (const U*)x, B_in, V, cpr, coords, count, capacity,
                      fps, (U*)y, ctx->status);
}

}  // namespace

hc_status launch_topk(const DeviceCtx* ctx, const float* alpha, int K, int kappa, int32_t* selected,
                      cudaStream_t s) {
    (void)ctx;
    return launch_pdl(topk_kernel, dim3(1), dim3(kTopkThreads), (size_t)K, s, "topk_kernel", alpha,
                      K, kappa, selected);
}

hc_status launch_kappa_masks(const DeviceCtx* ctx, const uint8_t* masks, int K, int V,
                             const int32_t* selected, int kappa, int B, uint8_t* out,
                             cudaStream_t s) {
    const long long total = (long long)B * kappa * V;
    long long blocks = (total + 255) / 256;
    const long long cap = (long long)ctx->num_sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    return launch_pdl(kappa_masks_kernel, dim3((unsigned)blocks), dim3(256), 0, s,
                      "kappa_masks_kernel", masks, K, V, selected, kappa, (long long)B, out,
                      ctx->status);
}

hc_status launch_gather_rows(const DeviceCtx* ctx, const void* x, int elem_bytes, int B_in, int V,
                             int C, const int32_t* coords, const int32_t* count, int capacity,
                             int frames_per_sample, void* y, cudaStream_t s) {
    const long long row_bytes = (long long)C * elem_bytes;
    const uintptr_t al = (uintptr_t)x | (uintptr_t)y;
    if (row_bytes % 16 == 0 && al % 16 == 0)
        return launch_gather_typed<uint4>(ctx, x, B_in, V, (int)(row_bytes / 16), coords, count,
                                          capacity, frames_per_sample, y, s);
    if (row_bytes % 4 == 0 && al % 4 == 0)
        return launch_gather_typed<uint32_t>(ctx, x, B_in, V, (int)(row_bytes / 4), coords, count,
                                             capacity, frames_per_sample, y, s);
    return launch_gather_typed<uint16_t>(ctx, x, B_in, V, (int)(row_bytes / 2), coords, count,
                                         capacity, frames_per_sample, y, s);
}

}  // namespace hc
