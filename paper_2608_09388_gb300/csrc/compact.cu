// Mask compaction: the decomposition of the masked tensor into coordinates
// C' (Eq. 2) together with the inverse map idx() of Eq. 4 and per-frame
// offsets. The output is the stable (ascending b*V + v) list of active rows,
// so it is unique and bit-exact.
//
// Two passes over tiles of 4096 mask bytes (256 threads x 16 bytes):
//   1. count   - every CTA counts the nonzero bytes of its tile;
//   2. write   - every CTA sums the counts of the tiles before it (or reads
//                a pre-scanned offset when there are many tiles), scans its
//                own 16-byte chunks across the block, and writes coords,
//                row_of and the per-frame offsets.
// Neither pass waits on another CTA, so there is no inter-CTA spin. The
// mask is read with 16-byte loads; HBM traffic is 2 reads of the mask plus
// the writes (8 B per active row, 4 B per row_of entry).
#include <mutex>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kThreads = 256;
constexpr int kItems = 16;
constexpr int kTile = kThreads * kItems;  // 4096 mask bytes per CTA
constexpr int kMaxDirectTiles = 1024;     // above this, pre-scan the tile counts

// High bit of each byte of the result is set iff that byte of w is nonzero.
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t w) {
    return (((w & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | w) & 0x80808080u;
}

// Loads this thread's 16 mask bytes (zeros past n) as a 16-bit flag set.
__device__ __forceinline__ uint32_t load_flags(const uint8_t* mask, long long n, long long base) {
    uint32_t flags = 0;
    if (base + kItems <= n && ((reinterpret_cast<uintptr_t>(mask + base) & 15u) == 0)) {
        uint4 q = __ldg(reinterpret_cast<const uint4*>(mask + base));
        uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            uint32_t m = nonzero_bytes(w[k]);
            // bytes 0..3 of word k -> flag bits 4k..4k+3
            flags |= ((m >> 7) & 1u) << (4 * k + 0);
            flags |= ((m >> 15) & 1u) << (4 * k + 1);
            flags |= ((m >> 23) & 1u) << (4 * k + 2);
            flags |= ((m >> 31) & 1u) << (4 * k + 3);
        }
    } else {
        for (int k = 0; k < kItems; ++k) {
            long long i = base + k;
            if (i < n && __ldg(mask + i) != 0) flags |= 1u << k;
        }
    }
    return flags;
}

__device__ __forceinline__ int block_sum(int v, int* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w) t += red[w];
    return t;
}

__global__ void __launch_bounds__(kThreads) compact_count_kernel(const uint8_t* __restrict__ mask,
                                                                 long long n,
                                                                 int32_t* __restrict__ tile_counts) {
    __shared__ int red[kThreads / 32];
    pdl_wait();
    pdl_trigger();
    long long base = (long long)blockIdx.x * kTile + (long long)threadIdx.x * kItems;
    int c = __popc(load_flags(mask, n, base));
    int t = block_sum(c, red);
    if (threadIdx.x == 0) tile_counts[blockIdx.x] = t;
}

// Exclusive scan of the tile counts in place (one CTA), for many tiles.
__global__ void __launch_bounds__(1024) compact_scan_kernel(int32_t* __restrict__ tile_counts,
                                                            int num_tiles) {
    __shared__ int warp_tot[32];
    __shared__ int carry;
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int base = 0; base < num_tiles; base += 1024) {
        int i = base + threadIdx.x;
        int v = i < num_tiles ? tile_counts[i] : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) warp_tot[warp] = x;
        __syncthreads();
        if (warp == 0) {
            int w = warp_tot[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            warp_tot[lane] = w;  // inclusive over warps
        }
        __syncthreads();
        int excl = carry + (warp ? warp_tot[warp - 1] : 0) + x - v;
        if (i < num_tiles) tile_counts[i] = excl;
        __syncthreads();
        if (threadIdx.x == 1023) carry = excl + v;
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kThreads)
    compact_write_kernel(const uint8_t* __restrict__ mask, long long n, int B, int V,
                         const int32_t* __restrict__ tile_counts, int num_tiles, int prescanned,
                         int32_t* __restrict__ coords, int32_t* __restrict__ row_of,
                         int32_t* __restrict__ offsets, int32_t* __restrict__ count) {
    __shared__ int red[kThreads / 32];
    __shared__ int warp_excl[kThreads / 32];
    __shared__ int tile_base_s;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int tile = blockIdx.x;
    // The mask is read before waiting on the count pass: that pass started
    // only after everything before it on the stream had finished, so the
    // mask is complete; its load overlaps the wait and the tile-count read.
    long long base = (long long)tile * kTile + (long long)tid * kItems;
    uint32_t flags = load_flags(mask, n, base);
    pdl_wait();
    pdl_trigger();

    // Rows before this tile.
    int tile_base;
    if (prescanned) {
        if (tid == 0) tile_base_s = tile_counts[tile];
        __syncthreads();
        tile_base = tile_base_s;
    } else {
        int part = 0;
        for (int t = tid; t < tile; t += kThreads) part += tile_counts[t];
        tile_base = block_sum(part, red);
    }

    int c = __popc(flags);

    // Block-wide exclusive scan of c.
    int x = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();  // every thread is done reading red[] from block_sum
    if (lane == 31) red[warp] = x;
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int w = 0; w < kThreads / 32; ++w) {
            warp_excl[w] = run;
            run += red[w];
        }
    }
    __syncthreads();
    int row = tile_base + warp_excl[warp] + x - c;

    // coords and row_of for this thread's 16 positions.
    if (base < n) {
        int v;
        int b = (int)div32(base, V, v);  // base < B*V < 2^31
        const int b_first = b, v_first = v;  // frame and vertex of base
        int r = row;
        int ro[kItems];
#pragma unroll
        for (int k = 0; k < kItems; ++k) {
            bool on = (flags >> k) & 1u;
            ro[k] = on ? r : -1;
            if (on) {
                coords[2LL * r + 0] = b;
                coords[2LL * r + 1] = v;
                ++r;
            }
            if (++v == V) {
                v = 0;
                ++b;
            }
        }
        if (row_of) {
            if (base + kItems <= n && ((reinterpret_cast<uintptr_t>(row_of + base) & 15u) == 0)) {
                int4* dst = reinterpret_cast<int4*>(row_of + base);
#pragma unroll
                for (int k = 0; k < kItems / 4; ++k)
                    dst[k] = make_int4(ro[4 * k], ro[4 * k + 1], ro[4 * k + 2], ro[4 * k + 3]);
            } else {
#pragma unroll
                for (int k = 0; k < kItems; ++k)
                    if (base + k < n) row_of[base + k] = ro[k];
            }
        }
        // Frame offsets: offsets[b] = rows before position b*V, for every
        // frame boundary b*V that falls in [base, base+16).
        if (offsets) {
            long long end = base + kItems < n ? base + kItems : n;
            // first frame boundary at or after base: the frame of base, plus
            // one unless base starts that frame
            long long bb = b_first + (v_first != 0 ? 1 : 0);
            for (; bb * V < end; ++bb) {
                int before = __popc(flags & ((1u << (int)(bb * V - base)) - 1u));
                offsets[bb] = row + before;
            }
        }
    }

    // The last tile knows the total.
    if (tile == num_tiles - 1) {
        int tot = block_sum(c, red);
        if (tid == 0) {
            *count = tile_base + tot;
            if (offsets) offsets[B] = tile_base + tot;
        }
    }
}

__global__ void compact_empty_kernel(int B, int32_t* offsets, int32_t* count) {
    pdl_wait();
    pdl_trigger();
    for (int i = threadIdx.x; i <= B; i += blockDim.x)
        if (offsets) offsets[i] = 0;
    if (threadIdx.x == 0) *count = 0;
}

}  // namespace

hc_status launch_compact(const DeviceCtx* ctx, const uint8_t* mask, int B, int V, int32_t* coords,
                         int32_t* row_of, int32_t* offsets, int32_t* count, cudaStream_t s) {
    (void)ctx;
    long long n = (long long)B * V;
    if (n == 0) {
        return launch_pdl(compact_empty_kernel, dim3(1), dim3(256), 0, s, "compact_empty_kernel", B,
                          offsets, count);
    }
    int num_tiles = (int)((n + kTile - 1) / kTile);
    int32_t* tile_counts = (int32_t*)stream_workspace(s, sizeof(int32_t) * (size_t)num_tiles);
    if (!tile_counts) return HC_ERR_CUDA;
    hc_status st = launch_pdl(compact_count_kernel, dim3(num_tiles), dim3(kThreads), 0, s,
                              "compact_count_kernel", mask, n, tile_counts);
    if (st != HC_OK) return st;
    int prescanned = num_tiles > kMaxDirectTiles;
    if (prescanned) {
        st = launch_pdl(compact_scan_kernel, dim3(1), dim3(1024), 0, s, "compact_scan_kernel",
                        tile_counts, num_tiles);
        if (st != HC_OK) return st;
    }
    return launch_pdl(compact_write_kernel, dim3(num_tiles), dim3(kThreads), 0, s,
                      "compact_write_kernel", mask, n, B, V, tile_counts, num_tiles, prescanned,
                      coords, row_of, offsets, count);
}

}  // namespace hc

// ---------------------------------------------------------------------------
// hc_mask_compact_static: the same compaction for callers that cannot
// allocate device memory. Its scratch (one int32 per 4096-byte mask tile) is
// a fixed array in the library's device image instead of a cudaMalloc'd
// workspace, so it serves masks of at most kStaticMaxTiles * 4096 bytes.
// ---------------------------------------------------------------------------
namespace hc {
namespace {

constexpr int kStaticMaxTiles = 4096;  // 16 KiB of scratch per device
static_assert((long long)kStaticMaxTiles * kTile == HC_STATIC_MAX_MASK_BYTES,
              "header limit and scratch size disagree");

// Every GPU that loads the library holds this array until the process exits.
// All calls on a device share it: it keeps the previous call's tile counts,
// and two calls whose kernels overlap on the GPU would race on it.
static __device__ __align__(256) int32_t g_static_tile_counts[kStaticMaxTiles];

constexpr int kMaxStaticDevices = 64;
int32_t* g_static_ptr[kMaxStaticDevices];
std::mutex g_static_mutex;

// Device address of the array for the current device. In host code the
// array's name is only a host-side stand-in, so the address is looked up
// once per device (with that device current) and cached.
hc_status static_scratch(int32_t** out) {
    int dev = -1;
    hc_status st = check_cuda(cudaGetDevice(&dev), "cudaGetDevice");
    if (st != HC_OK) return st;
    if (dev < 0 || dev >= kMaxStaticDevices) {
        set_error("device ordinal %d out of range", dev);
        return HC_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(g_static_mutex);
    if (!g_static_ptr[dev]) {
        void* p = nullptr;
        st = check_cuda(cudaGetSymbolAddress(&p, g_static_tile_counts),
                        "cudaGetSymbolAddress(static compaction scratch)");
        if (st != HC_OK) return st;
        g_static_ptr[dev] = static_cast<int32_t*>(p);
    }
    *out = g_static_ptr[dev];
    return HC_OK;
}

// The count / (scan) / write passes into caller-chosen scratch. Every tile's
// count is rewritten before it is read, so nothing has to be cleared first.
hc_status launch_compact_into(const uint8_t* mask, int B, int V, int32_t* coords,
                              int32_t* row_of, int32_t* offsets, int32_t* count,
                              int32_t* tile_counts, cudaStream_t s) {
    long long n = (long long)B * V;
    if (n == 0) {
        return launch_pdl(compact_empty_kernel, dim3(1), dim3(256), 0, s, "compact_empty_kernel", B,
                          offsets, count);
    }
    int num_tiles = (int)((n + kTile - 1) / kTile);
    hc_status st = launch_pdl(compact_count_kernel, dim3(num_tiles), dim3(kThreads), 0, s,
                              "compact_count_kernel", mask, n, tile_counts);
    if (st != HC_OK) return st;
    int prescanned = num_tiles > kMaxDirectTiles;
    if (prescanned) {
        st = launch_pdl(compact_scan_kernel, dim3(1), dim3(1024), 0, s, "compact_scan_kernel",
                        tile_counts, num_tiles);
        if (st != HC_OK) return st;
    }
    return launch_pdl(compact_write_kernel, dim3(num_tiles), dim3(kThreads), 0, s,
                      "compact_write_kernel", mask, n, B, V, tile_counts, num_tiles, prescanned,
                      coords, row_of, offsets, count);
}

}  // namespace
}  // namespace hc

extern "C" hc_status hc_mask_compact_static(const uint8_t* mask, int B, int V, int32_t* coords,
                                            int32_t* row_of, int32_t* batch_offsets,
                                            int32_t* count, hc_stream_t stream) {
    using namespace hc;
    set_error("%s", "");
    if (B < 0 || V < 0) {
        set_error("hc_mask_compact_static: B=%d V=%d must be >= 0", B, V);
        return HC_ERR_INVALID_ARG;
    }
    if (count == nullptr) {
        set_error("hc_mask_compact_static: count is NULL");
        return HC_ERR_INVALID_ARG;
    }
    const long long n = (long long)B * V;
    if (n > 0 && (mask == nullptr || coords == nullptr)) {
        set_error("hc_mask_compact_static: mask and coords are required");
        return HC_ERR_INVALID_ARG;
    }
    if (n > HC_STATIC_MAX_MASK_BYTES) {
        set_error("hc_mask_compact_static: B*V = %lld exceeds the fixed scratch limit of %d mask "
                  "bytes; use hc_mask_compact",
                  n, HC_STATIC_MAX_MASK_BYTES);
        return HC_ERR_UNSUPPORTED;
    }
    int32_t* scratch = nullptr;
    hc_status st = static_scratch(&scratch);
    if (st != HC_OK) return st;
    return launch_compact_into(mask, B, V, coords, row_of, batch_offsets, count, scratch,
                               (cudaStream_t)stream);
}
