// Row order for the rulebook convolution (an execution schedule; the paper
// has no counterpart, and the results do not depend on it).
//
// Under the Eq. 4 mapping a row's tap l contributes only when its rulebook
// entry (l, n) is present; at low mask density most entries are absent, yet
// a tile of 128 consecutive rows almost always has every tap present in some
// row, so the conv multiplies all L taps of every tile. Sorting the active
// rows by their presence pattern (bit l set when tap l is present) puts rows
// with the same taps into the same tiles, and the union of a tile's patterns
// names the only taps its MMAs need. Like the rulebook, the order depends on
// the mask only, so one pass serves every conv layer of a network.
//
//   keys      key of every active row (its presence pattern), and the count
//             of each bin (the low min(L, 12) bits of the key);
//   scan      exclusive prefix of the bin counts (one block);
//   scatter   every row to its bin's next positions, and its rulebook column
//             to the same position of the sorted rulebook (so that the conv
//             reads a tile's columns contiguously, as without an order);
//   unions    the OR of the keys of each 128-row tile of the order.
// Counting is aggregated per block (lanes of equal bin matched in a warp,
// per-block counts in shared memory) so that one global atomic serves every
// row of a bin in a block: with few distinct keys (dense masks) per-row
// atomics on one counter would serialise the whole pass. Rows of equal bin
// land in an unspecified order (a row's result does not depend on the rows
// sharing its tile).
#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kOrderTile = 128;  // rows per conv tile
constexpr int kSortBits = 12;    // bins = 2^min(L, kSortBits)
constexpr int kMaxBins = 1 << kSortBits;
constexpr int kBlock = 256;
constexpr int kScanThreads = 1024;

__device__ __forceinline__ long long clamp_rows(const int32_t* count, long long capacity,
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

// Key of row n: bit l set when rulebook entry (l, n) is present.
__device__ __forceinline__ uint32_t row_key(const int32_t* __restrict__ rulebook,
                                            long long capacity, int L, long long n) {
    int e[HC_MAX_SPIRAL];
#pragma unroll
    for (int l = 0; l < HC_MAX_SPIRAL; ++l)
        e[l] = l < L ? __ldg(rulebook + (long long)l * capacity + n) : -1;
    uint32_t key = 0;
#pragma unroll
    for (int l = 0; l < HC_MAX_SPIRAL; ++l) key |= (e[l] >= 0 ? 1u : 0u) << l;
    return key;
}

// Rank of this lane among the active lanes of the warp with the same bin,
// the number of such lanes, and whether this lane is their leader.
__device__ __forceinline__ void bin_peers(uint32_t active, uint32_t bin, int& rank, int& n,
                                          bool& leader) {
    const uint32_t peers = __match_any_sync(active, bin);
    const int lane = threadIdx.x & 31;
    rank = __popc(peers & ((1u << lane) - 1u));
    n = __popc(peers);
    leader = rank == 0;
}

__global__ void __launch_bounds__(kBlock) order_keys_kernel(const int32_t* __restrict__ rulebook,
                                                            const int32_t* __restrict__ count,
                                                            long long capacity, int L, int bins,
                                                            uint32_t* __restrict__ keys,
                                                            int32_t* __restrict__ hist,
                                                            unsigned* status) {
    __shared__ int32_t cnt[kMaxBins];
    for (int i = threadIdx.x; i < bins; i += kBlock) cnt[i] = 0;
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    __syncthreads();
    for (long long base = blockIdx.x * (long long)kBlock; base < rows;
         base += (long long)gridDim.x * kBlock) {
        const long long n = base + threadIdx.x;
        const bool in = n < rows;
        const uint32_t active = __ballot_sync(0xffffffffu, in);
        if (in) {
            const uint32_t key = row_key(rulebook, capacity, L, n);
            keys[n] = key;
            const uint32_t bin = key & (uint32_t)(bins - 1);
            int rank, k;
            bool leader;
            bin_peers(active, bin, rank, k, leader);
            if (leader) atomicAdd(cnt + bin, k);
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < bins; i += kBlock)
        if (cnt[i]) atomicAdd(hist + i, cnt[i]);
}

// Exclusive prefix of the bin counts into cursor (bins <= 4096, one block).
__global__ void __launch_bounds__(kScanThreads) order_scan_kernel(const int32_t* __restrict__ hist,
                                                                  int bins,
                                                                  int32_t* __restrict__ cursor) {
    pdl_wait();
    pdl_trigger();
    __shared__ int32_t warp_sums[kScanThreads / 32];
    const int per = (bins + kScanThreads - 1) / kScanThreads;
    const int b0 = threadIdx.x * per;
    int32_t local = 0;
    for (int i = 0; i < per; ++i)
        if (b0 + i < bins) local += hist[b0 + i];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t v = local;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int32_t u = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += u;
    }
    if (lane == 31) warp_sums[warp] = v;
    __syncthreads();
    if (warp == 0) {
        int32_t s = warp_sums[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t u = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += u;
        }
        warp_sums[lane] = s;  // inclusive over warps
    }
    __syncthreads();
    int32_t run = v - local + (warp > 0 ? warp_sums[warp - 1] : 0);
    for (int i = 0; i < per; ++i)
        if (b0 + i < bins) {
            cursor[b0 + i] = run;
            run += hist[b0 + i];
        }
}

// Every row (and its rulebook column) to a position of its bin. Per chunk of
// kBlock rows: ranks within the block's bins (warp match + shared counts),
// one global reservation per bin present, then the writes.
__global__ void __launch_bounds__(kBlock) order_scatter_kernel(
    const uint32_t* __restrict__ keys, const int32_t* __restrict__ rulebook,
    const int32_t* __restrict__ count, long long capacity, int L, int bins,
    int32_t* __restrict__ cursor, int32_t* __restrict__ order, int32_t* __restrict__ sorted_rb,
    unsigned* status) {
    __shared__ int32_t cnt[kMaxBins];
    __shared__ int32_t start[kMaxBins];
    for (int i = threadIdx.x; i < bins; i += kBlock) cnt[i] = 0;
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    __syncthreads();
    for (long long base = blockIdx.x * (long long)kBlock; base < rows;
         base += (long long)gridDim.x * kBlock) {
        const long long n = base + threadIdx.x;
        const bool in = n < rows;
        const uint32_t active = __ballot_sync(0xffffffffu, in);
        uint32_t bin = 0;
        int rank = 0;
        bool first = false;  // the block's first row of its bin
        if (in) {
            bin = keys[n] & (uint32_t)(bins - 1);
            int k;
            bool leader;
            bin_peers(active, bin, rank, k, leader);
            int b = 0;
            if (leader) b = atomicAdd(cnt + bin, k);
            b = __shfl_sync(active, b, __ffs(__match_any_sync(active, bin)) - 1);
            rank += b;
            first = rank == 0;
        }
        __syncthreads();
        if (first) start[bin] = atomicAdd(cursor + bin, cnt[bin]);
        __syncthreads();
        if (in) {
            const int pos = start[bin] + rank;
            order[pos] = (int32_t)n;
            for (int l = 0; l < L; ++l)
                sorted_rb[(long long)l * capacity + pos] = __ldg(rulebook + (long long)l * capacity + n);
        }
        __syncthreads();
        if (first) cnt[bin] = 0;  // ready for the next chunk
        __syncthreads();
    }
}

// One warp per tile of the order: the OR of its rows' keys.
__global__ void __launch_bounds__(kBlock) order_unions_kernel(const uint32_t* __restrict__ keys,
                                                              const int32_t* __restrict__ order,
                                                              const int32_t* __restrict__ count,
                                                              long long capacity,
                                                              uint32_t* __restrict__ tile_taps,
                                                              unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    const long long tiles = (rows + kOrderTile - 1) / kOrderTile;
    const int lane = threadIdx.x & 31;
    for (long long t = (blockIdx.x * (long long)kBlock + threadIdx.x) / 32; t < tiles;
         t += (long long)gridDim.x * kBlock / 32) {
        uint32_t u = 0;
#pragma unroll
        for (int i = 0; i < kOrderTile / 32; ++i) {
            const long long p = t * kOrderTile + lane + 32 * i;
            if (p < rows) {
                const int32_t n = order[p];
                if (n >= 0 && n < rows) u |= keys[n];
                else report(status, kErrIndex);
            }
        }
        u = __reduce_or_sync(0xffffffffu, u);
        if (lane == 0) tile_taps[t] = u;
    }
}

}  // namespace

hc_status launch_rulebook_order(const DeviceCtx* ctx, const int32_t* rulebook,
                                const int32_t* count, long long capacity, int L, int32_t* order,
                                uint32_t* tile_taps, int32_t* sorted_rb, cudaStream_t s) {
    const int bits = L < kSortBits ? L : kSortBits;
    const int bins = 1 << bits;
    // workspace: keys [capacity], bin counts [bins], cursor [bins]
    const size_t key_bytes = ((size_t)capacity * 4 + 255) / 256 * 256;
    char* ws = static_cast<char*>(stream_workspace(s, key_bytes + 8 * (size_t)bins));
    if (!ws) return HC_ERR_CUDA;
    uint32_t* keys = reinterpret_cast<uint32_t*>(ws);
    int32_t* hist = reinterpret_cast<int32_t*>(ws + key_bytes);
    int32_t* cursor = hist + bins;
    hc_status st = check_cuda(cudaMemsetAsync(hist, 0, sizeof(int32_t) * (size_t)bins, s),
                              "cudaMemsetAsync(order bin counts)");
    if (st != HC_OK) return st;
    long long blocks = (capacity + kBlock - 1) / kBlock;
    const long long cap = (long long)ctx->num_sms * 4;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    st = launch_pdl(order_keys_kernel, dim3((unsigned)blocks), dim3(kBlock), 0, s,
                    "order_keys_kernel", rulebook, count, capacity, L, bins, keys, hist,
                    ctx->status);
    if (st != HC_OK) return st;
    st = launch_pdl(order_scan_kernel, dim3(1), dim3(kScanThreads), 0, s, "order_scan_kernel",
                    (const int32_t*)hist, bins, cursor);
    if (st != HC_OK) return st;
    st = launch_pdl(order_scatter_kernel, dim3((unsigned)blocks), dim3(kBlock), 0, s,
                    "order_scatter_kernel", (const uint32_t*)keys, rulebook, count, capacity, L,
                    bins, cursor, order, sorted_rb, ctx->status);
    if (st != HC_OK) return st;
    const long long tiles = (capacity + kOrderTile - 1) / kOrderTile;
    long long ublocks = (tiles * 32 + kBlock - 1) / kBlock;
    if (ublocks > cap) ublocks = cap;
    if (ublocks < 1) ublocks = 1;
    return launch_pdl(order_unions_kernel, dim3((unsigned)ublocks), dim3(kBlock), 0, s,
                      "order_unions_kernel", (const uint32_t*)keys, (const int32_t*)order, count,
                      capacity, tile_taps, ctx->status);
}

}  // namespace hc
