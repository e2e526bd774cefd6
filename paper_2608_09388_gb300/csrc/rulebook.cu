// The indexing matrix of the sparse convolution (Eq. 4) for the spiral
// neighbourhood, materialised once per mask: for every active row n and
// spiral slot l, the input row that feeds the tap, or -1 when the tap is
// absent (no neighbour in that slot, or the neighbour is not an active row).
// The coordinates do not change from layer to layer (Eq. 5 keeps the centre
// coordinates), so one rulebook serves every conv layer of a network.
//
// Layout: [L, capacity] int32, slot-major (entry (l, n) at l*capacity + n),
// so that a tile of consecutive rows reads each slot as one contiguous run.
// One thread per active row; its coordinate, spiral entries and row_of
// lookups are each issued together from clamped, always-valid addresses:
// the first row's coordinate together with the row count, then up to
// kChunk spiral slots, then their row_of entries (three round trips for
// L <= kChunk); a thread with more rows fetches the next row's coordinate
// during the current row's lookups.
#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kChunk = 16;

__global__ void __launch_bounds__(256, 3) rulebook_kernel(const int32_t* __restrict__ coords,
                                                       const int32_t* __restrict__ row_of,
                                                       const int32_t* __restrict__ count,
                                                       const int32_t* __restrict__ spiral, int B,
                                                       int V, int L, int x_layout,
                                                       int32_t* __restrict__ rulebook,
                                                       unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long cap = (long long)B * V;
    const long long n0 = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    // every n < capacity indexes coords: the first row's coordinate is
    // fetched with the row count, before it is known to be active
    int b0 = 0, v0 = 0;
    if (n0 < cap) {
        b0 = __ldg(coords + 2 * n0);
        v0 = __ldg(coords + 2 * n0 + 1);
    }
    long long rows = *count;
    unsigned err = 0;
    if (rows < 0) {
        err |= kErrIndex;
        rows = 0;
    }
    if (rows > cap) {
        err |= kErrCapacity;
        rows = cap;
    }
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long n = n0; n < rows; n += stride) {
        int b = b0, v = v0;
        // the next row's coordinate, fetched while this row's lookups run
        if (n + stride < rows) {
            b0 = __ldg(coords + 2 * (n + stride));
            v0 = __ldg(coords + 2 * (n + stride) + 1);
        }
        const bool ok = b >= 0 && b < B && v >= 0 && v < V;
        if (!ok) {
            err |= kErrIndex;
            b = v = 0;
        }
        for (int l0 = 0; l0 < L; l0 += kChunk) {
            int u[kChunk], dr[kChunk], j[kChunk];
#pragma unroll
            for (int d = 0; d < kChunk; ++d)
                u[d] = __ldg(spiral + (long long)v * L + (l0 + d < L ? l0 + d : L - 1));
#pragma unroll
            for (int d = 0; d < kChunk; ++d) {
                const bool live = ok && l0 + d < L;
                if (live && (u[d] < -1 || u[d] >= V)) err |= kErrIndex;
                dr[d] = (live && u[d] >= 0 && u[d] < V) ? b * V + u[d] : -1;
            }
#pragma unroll
            for (int d = 0; d < kChunk; ++d) j[d] = __ldg(row_of + (dr[d] >= 0 ? dr[d] : 0));
#pragma unroll
            for (int d = 0; d < kChunk; ++d) {
                if (l0 + d >= L) continue;
                int e = -1;
                if (dr[d] >= 0) {
                    if (j[d] < -1 || j[d] >= rows) err |= kErrIndex;
                    if (j[d] >= 0 && j[d] < rows) e = x_layout == HC_LAYOUT_DENSE ? dr[d] : j[d];
                }
                rulebook[(long long)(l0 + d) * cap + n] = e;
            }
        }
    }
    if (err) report(status, err);
}

}  // namespace

hc_status launch_rulebook(const DeviceCtx* ctx, const int32_t* coords, const int32_t* row_of,
                          const int32_t* count, const int32_t* spiral, int B, int V, int L,
                          int x_layout, int32_t* rulebook, cudaStream_t s) {
    const long long cap = (long long)B * V;
    long long blocks = (cap + 255) / 256;
    // up to 8 blocks per SM: beyond the resident ones (3 per SM) they cost
    // the row count's round trip per wave when rows are few, but keep more
    // lookups in flight when most rows are active
    const long long lim = (long long)ctx->num_sms * 8;
    if (blocks > lim) blocks = lim;
    if (blocks < 1) blocks = 1;
    return launch_pdl(rulebook_kernel, dim3((unsigned)blocks), dim3(256), 0, s, "rulebook_kernel",
                      coords, row_of, count, spiral, B, V, L, x_layout, rulebook, ctx->status);
}

}  // namespace hc
