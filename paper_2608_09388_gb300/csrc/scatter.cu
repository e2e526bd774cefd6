// Scatter of compact rows back into a dense [B, V, C] tensor (the inverse of
// the decomposition, Eq. 2). Rows are moved in 16-, 4- or 2-byte chunks
// (the widest the row size and pointer alignment allow), bit for bit.
//   scatter:      out[coords[n]] = y[n]           for n < N'
//   scatter+fill: out[r] = row_of[r] >= 0 ? y[row_of[r]] : 0   for every r
// With row_of, the fill variant writes every dense row exactly once (one
// pass over the output instead of a memset followed by a scatter); without
// it, a zero pass over the output is followed by the scatter.
#include "hc_internal.cuh"

namespace hc {
namespace {

template <typename U>
__device__ __forceinline__ U zero_chunk();
template <>
__device__ __forceinline__ uint4 zero_chunk<uint4>() {
    return make_uint4(0, 0, 0, 0);
}
template <>
__device__ __forceinline__ uint32_t zero_chunk<uint32_t>() {
    return 0u;
}
template <>
__device__ __forceinline__ uint16_t zero_chunk<uint16_t>() {
    return (uint16_t)0;
}

__device__ __forceinline__ long long clamp_count(const int32_t* count, long long capacity,
                                                 unsigned* status) {
    long long n = *count;
    if (n < 0) {
        report(status, kErrIndex);
        return 0;
    }
    if (n > capacity) {
        report(status, kErrCapacity);
        return capacity;
    }
    return n;
}

template <typename U>
__global__ void scatter_kernel(const U* __restrict__ y, const int32_t* __restrict__ coords,
                               const int32_t* __restrict__ count, int B, int V, int cpr,
                               U* __restrict__ out, unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_count(count, (long long)B * V, status);
    const long long total = rows * cpr;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        int c;
        const long long n = div32(i, cpr, c);
        const int b = __ldg(coords + 2 * n), v = __ldg(coords + 2 * n + 1);
        if (b < 0 || b >= B || v < 0 || v >= V) {
            report(status, kErrIndex);
            continue;
        }
        out[((long long)b * V + v) * cpr + c] = y[i];
    }
}

template <typename U>
__global__ void zero_kernel(long long total, U* __restrict__ out) {
    pdl_wait();
    pdl_trigger();
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x)
        out[i] = zero_chunk<U>();
}

template <typename U>
__global__ void scatter_fill_kernel(const U* __restrict__ y, const int32_t* __restrict__ row_of,
                                    const int32_t* __restrict__ count, long long dense_rows,
                                    int cpr, U* __restrict__ out, unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_count(count, dense_rows, status);
    const long long total = dense_rows * cpr;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        int c;
        const long long r = div32(i, cpr, c);
        const int j = __ldg(row_of + r);
        U val = zero_chunk<U>();
        if (j >= 0 && j < rows)
            val = y[(long long)j * cpr + c];
        else if (j != -1)
            report(status, kErrIndex);
        out[i] = val;
    }
}

template <typename U>
hc_status launch_typed(const DeviceCtx* ctx, const void* y, const int32_t* coords,
                       const int32_t* row_of, const int32_t* count, int B, int V, int cpr,
                       int zero_fill, void* out, cudaStream_t s) {
    const long long dense_rows = (long long)B * V;
    const long long work = dense_rows * cpr;
    long long blocks = (work + 255) / 256;
    const long long cap = (long long)ctx->num_sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (zero_fill && !row_of) {
        // no inverse map: zero every row, then scatter the active ones
        hc_status st = launch_pdl(zero_kernel<U>, dim3((unsigned)blocks), dim3(256), 0, s,
                                  "zero_kernel", work, (U*)out);
        if (st != HC_OK) return st;
    } else if (zero_fill) {
        return launch_pdl(scatter_fill_kernel<U>, dim3((unsigned)blocks), dim3(256), 0, s,
                          "scatter_fill_kernel", (const U*)y, row_of, count, dense_rows, cpr,
                          (U*)out, ctx->status);
    }
    return launch_pdl(scatter_kernel<U>, dim3((unsigned)blocks), dim3(256), 0, s, "scatter_kernel",
                      (const U*)y, coords, count, B, V, cpr, (U*)out, ctx->status);
}

}  // namespace

hc_status launch_scatter(const DeviceCtx* ctx, const void* y, int elem_bytes, const int32_t* coords,
                         const int32_t* row_of, const int32_t* count, int B, int V, int C,
                         int zero_fill, void* out, cudaStream_t s) {
    const long long row_bytes = (long long)C * elem_bytes;
    const uintptr_t align = (uintptr_t)y | (uintptr_t)out;
    if (row_bytes % 16 == 0 && align % 16 == 0)
        return launch_typed<uint4>(ctx, y, coords, row_of, count, B, V, (int)(row_bytes / 16),
                                   zero_fill, out, s);
    if (row_bytes % 4 == 0 && align % 4 == 0)
        return launch_typed<uint32_t>(ctx, y, coords, row_of, count, B, V, (int)(row_bytes / 4),
                                      zero_fill, out, s);
    return launch_typed<uint16_t>(ctx, y, coords, row_of, count, B, V, (int)(row_bytes / 2),
                                  zero_fill, out, s);
}

}  // namespace hc
