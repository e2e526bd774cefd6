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

// The 16 nonzero-byte flags of a 16-byte piece of the mask.
__device__ __forceinline__ uint32_t flags_of(uint4 q) {
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
    uint32_t flags = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t m = nonzero_bytes(w[k]);
        flags |= ((m >> 7) & 1u) << (4 * k + 0);
        flags |= ((m >> 15) & 1u) << (4 * k + 1);
        flags |= ((m >> 23) & 1u) << (4 * k + 2);
        flags |= ((m >> 31) & 1u) << (4 * k + 3);
    }
    return flags;
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

template <int NT>
__device__ __forceinline__ int block_sum(int v, int* red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) t += red[w];
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
    int t = block_sum<kThreads>(c, red);
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
        tile_base = block_sum<kThreads>(part, red);
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
        int tot = block_sum<kThreads>(c, red);
        if (tid == 0) {
            *count = tile_base + tot;
            if (offsets) offsets[B] = tile_base + tot;
        }
    }
}

// ---------------------------------------------------------------- compaction + Eq. 4 mapping
// The write pass fused with the mapping (the rulebook of hc_conv_rulebook):
// CTA (b, s) rebuilds frame b's activity and ranks in shared memory, per
// 16-byte chunk of the mask bytes from the aligned byte below b*V: the
// chunk's 16 activity flags and the frame's active rows before it, so that
// the rank of vertex p (active rows of the frame before p) is the chunk's
// count plus a popcount. It then writes row_of, coords and the rulebook
// columns of the active vertices in its portion [s*kMapPortion,
// (s+1)*kMapPortion); every tap lookup row_of[b, u] of Eq. 4 is a
// shared-memory read. The mask, the ranks and the first spiral entries of
// the portion's active vertices do not depend on the count pass and are
// read before waiting on it (the count pass lets this one start only after
// its own wait, so whatever wrote the mask and the spiral table before it
// has finished); after the wait only the tile counts before the frame are
// read (frame offset = those counts + the active bytes of the frame's own
// 4096-byte tile before b*V, counted here). Shared memory stays small (6
// bytes per 16 vertices + 2 per portion vertex); it is the registers (a
// CTA's 12k beside a conv CTA's 59k) that keep the conv that follows off an
// SM until the SM's mapping CTAs have finished.
constexpr int kMapThreads = 256;
constexpr int kMapPortion = 1024;
constexpr int kMapMaxV = 65535;
constexpr int kMapMaxL = HC_MAX_SPIRAL;
constexpr int kMapPre = 4;  // tap entries per thread read before the wait

struct MapArgs {
    const uint8_t* mask;
    long long n;  // B * V
    int B, V, L, x_layout, S, nch;
    const int32_t* spiral;
    const int32_t* tile_counts;
    int num_tiles, prescanned;
    int32_t* coords;
    int32_t* row_of;
    int32_t* offsets;
    int32_t* count;
    int32_t* rulebook;
    unsigned* status;
};

size_t map_smem_bytes(int nch) {
    return ((size_t)nch * 4 + (size_t)nch * 2 + 15) / 16 * 16 + sizeof(uint16_t) * kMapPortion;
}

// Exclusive block scan of v (kMapThreads threads); total in *tot.
__device__ __forceinline__ int block_excl_scan(int v, int* red, int* tot) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();  // red[] is free
    if (lane == 31) red[warp] = x;
    __syncthreads();
    int before = 0, all = 0;
#pragma unroll
    for (int w = 0; w < kMapThreads / 32; ++w) {
        before += w < warp ? red[w] : 0;
        all += red[w];
    }
    *tot = all;
    return before + x - v;
}

__global__ void __launch_bounds__(kMapThreads) compact_map_kernel(const MapArgs a) {
    extern __shared__ __align__(16) uint8_t map_smem[];
    __shared__ int red[kMapThreads / 32];
    const int V = a.V, L = a.L;
    int32_t* s_rank = reinterpret_cast<int32_t*>(map_smem);           // [nch]
    uint16_t* s_flag = reinterpret_cast<uint16_t*>(s_rank + a.nch);    // [nch]
    uint16_t* act_v = reinterpret_cast<uint16_t*>(map_smem + ((size_t)a.nch * 6 + 15) / 16 * 16);
    const int tid = threadIdx.x;
    const int b = blockIdx.x / a.S, s = blockIdx.x - b * a.S;
    const long long fb = (long long)b * V;  // the frame's first mask byte
    const long long a0 = fb & ~15ll;
    const int sh = (int)(fb - a0);  // vertex p is bit (p + sh) of the chunk list
    const int nch = (int)((fb + V - a0 + 15) >> 4);

    // active bytes of the frame's 4096-byte tile before fb (loaded with the
    // frame's own chunks)
    const int tb = (int)(fb / kTile);
    uint32_t pf = 0;
    {
        const long long g = (long long)tb * kTile + 16ll * tid;
        if (g < fb) {
            pf = load_flags(a.mask, a.n, g);
            const long long hi = fb - g;
            if (hi < kItems) pf &= (1u << hi) - 1u;
        }
    }
    // thread t takes chunks t*m .. t*m + m - 1: their flags, one block scan of
    // the per-thread counts, then the chunks' ranks
    const int m = (nch + kMapThreads - 1) / kMapThreads;
    const int cb0 = tid * m;
    int cnt = 0;
    // the chunks' loads in batches of kBatch, all in flight before any is used
    constexpr int kBatch = 4;
    const bool vec_ok = (reinterpret_cast<uintptr_t>(a.mask + a0) & 15u) == 0;
    for (int j0 = 0; j0 < m; j0 += kBatch) {
        uint4 q[kBatch];
#pragma unroll
        for (int jj = 0; jj < kBatch; ++jj) {
            const int c = cb0 + j0 + jj;
            const long long g = a0 + 16ll * c;
            q[jj] = (j0 + jj < m && c < nch && vec_ok && g + kItems <= a.n)
                        ? __ldg(reinterpret_cast<const uint4*>(a.mask + g))
                        : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int jj = 0; jj < kBatch; ++jj) {
            const int c = cb0 + j0 + jj;
            if (j0 + jj < m && c < nch) {
                const long long g = a0 + 16ll * c;
                uint32_t f = (vec_ok && g + kItems <= a.n) ? flags_of(q[jj])
                                                          : load_flags(a.mask, a.n, g);
                const long long lo = fb - g, hi = fb + V - g;  // in-frame bytes lo .. hi-1
                if (lo > 0) f &= 0xFFFFu << lo;
                if (hi < kItems) f &= (1u << hi) - 1u;
                s_flag[c] = (uint16_t)f;
                cnt += __popc(f);
            }
        }
    }
    int fc;  // active rows of frame b
    int r = block_excl_scan(cnt, red, &fc);
    for (int j = 0; j < m; ++j) {
        const int c = cb0 + j;
        if (c < nch) {
            s_rank[c] = r;
            r += __popc((uint32_t)s_flag[c]);
        }
    }
    const int part = block_sum<kMapThreads>(__popc(pf), red);  // synchronises: the chunk tables are complete
    // rank of vertex p (active rows of the frame before it) and its activity
    auto rank_of = [&](int p, bool& on) {
        const int q = p + sh, c = q >> 4, k = q & 15;
        const uint32_t f = s_flag[c];
        on = (f >> k) & 1u;
        return s_rank[c] + __popc(f & ((1u << k) - 1u));
    };
    const int v0 = s * kMapPortion, v1 = v0 + kMapPortion < V ? v0 + kMapPortion : V;
    bool on;
    const int R0 = rank_of(v0, on);  // v0 < V
    const int R1 = v1 < V ? rank_of(v1, on) : fc;
    const int nact = R1 - R0;
    for (int p = v0 + tid; p < v1; p += kMapThreads) {
        const int r = rank_of(p, on);
        if (on) act_v[r - R0] = (uint16_t)(p - v0);
    }
    __syncthreads();
    // the first tap entries of this thread (item i: slot l = i / nact,
    // active vertex k = i % nact of the portion)
    const int items = nact * L;
    int u_pre[kMapPre];
#pragma unroll
    for (int q = 0; q < kMapPre; ++q) {
        const int i = tid + q * kMapThreads;
        u_pre[q] = -1;
        if (i < items) {
            int k;
            const int l = (int)div32(i, nact, k);
            u_pre[q] = __ldg(a.spiral + (long long)(v0 + act_v[k]) * L + l);
        }
    }

    pdl_wait();  // the tile counts come from the count pass
    pdl_trigger();
    int before;
    if (a.prescanned) {
        before = a.tile_counts[tb];
    } else {
        int acc = 0;
        for (int t = tid; t < tb; t += kMapThreads) acc += a.tile_counts[t];
        before = block_sum<kMapThreads>(acc, red);
    }
    const int off = before + part;  // rows before frame b
    if (tid == 0 && s == 0) {
        if (a.offsets) a.offsets[b] = off;
        if (b == a.B - 1) {
            *a.count = off + fc;
            if (a.offsets) a.offsets[a.B] = off + fc;
        }
    }
    const long long n0 = (long long)off + R0;  // first row of the portion
    unsigned err = 0;
    for (int i = tid; i < items; i += kMapThreads) {
        int k;
        const int l = (int)div32(i, nact, k);
        const int q = (i - tid) / kMapThreads;
        int u = -1;
#pragma unroll
        for (int j = 0; j < kMapPre; ++j)
            if (q == j) u = u_pre[j];
        if (q >= kMapPre) u = __ldg(a.spiral + (long long)(v0 + act_v[k]) * L + l);
        int e = -1;
        if (u < -1 || u >= V) {
            err |= kErrIndex;
        } else if (u >= 0) {
            bool hit;
            const int r = rank_of(u, hit);
            if (hit) e = a.x_layout == HC_LAYOUT_DENSE ? (int)(fb + u) : off + r;
        }
        a.rulebook[(long long)l * a.n + n0 + k] = e;
    }
    if (a.row_of)
        for (int p = v0 + tid; p < v1; p += kMapThreads) {
            const int r = rank_of(p, on);
            a.row_of[fb + p] = on ? off + r : -1;
        }
    for (int k = tid; k < nact; k += kMapThreads) {
        a.coords[2 * (n0 + k)] = b;
        a.coords[2 * (n0 + k) + 1] = v0 + act_v[k];
    }
    if (err) report(a.status, err);
}

__global__ void compact_empty_kernel(int B, int32_t* offsets, int32_t* count) {
    pdl_wait();
    pdl_trigger();
    for (int i = threadIdx.x; i <= B; i += blockDim.x)
        if (offsets) offsets[i] = 0;
    if (threadIdx.x == 0) *count = 0;
}

}  // namespace

bool compact_map_supported(int B, int V, int L) {
    return B >= 1 && V >= 1 && V <= kMapMaxV && L >= 1 && L <= kMapMaxL &&
           map_smem_bytes(V / 16 + 2) <= 48 * 1024;
}

// Count pass (and the tile pre-scan when there are many tiles), then the
// fused write + mapping pass.
hc_status launch_compact_map(const DeviceCtx* ctx, const uint8_t* mask, int B, int V,
                             const int32_t* spiral, int L, int x_layout, int32_t* coords,
                             int32_t* row_of, int32_t* offsets, int32_t* count, int32_t* rulebook,
                             cudaStream_t s) {
    const long long n = (long long)B * V;
    const int num_tiles = (int)((n + kTile - 1) / kTile);
    int32_t* tile_counts = (int32_t*)stream_workspace(s, sizeof(int32_t) * (size_t)num_tiles);
    if (!tile_counts) return HC_ERR_CUDA;
    hc_status st = launch_pdl(compact_count_kernel, dim3(num_tiles), dim3(kThreads), 0, s,
                              "compact_count_kernel", mask, n, tile_counts);
    if (st != HC_OK) return st;
    const int prescanned = num_tiles > kMaxDirectTiles;
    if (prescanned) {
        st = launch_pdl(compact_scan_kernel, dim3(1), dim3(1024), 0, s, "compact_scan_kernel",
                        tile_counts, num_tiles);
        if (st != HC_OK) return st;
    }
    const int nch = V / 16 + 2;  // 16-byte chunks covering a frame, any alignment
    const size_t smem = map_smem_bytes(nch);
    MapArgs a{};
    a.nch = nch;
    a.mask = mask;
    a.n = n;
    a.B = B;
    a.V = V;
    a.L = L;
    a.x_layout = x_layout;
    a.S = (V + kMapPortion - 1) / kMapPortion;
    a.spiral = spiral;
    a.tile_counts = tile_counts;
    a.num_tiles = num_tiles;
    a.prescanned = prescanned;
    a.coords = coords;
    a.row_of = row_of;
    a.offsets = offsets;
    a.count = count;
    a.rulebook = rulebook;
    a.status = ctx->status;
    return launch_pdl(compact_map_kernel, dim3((unsigned)((long long)B * a.S)), dim3(kMapThreads),
                      smem, s, "compact_map_kernel", a);
}

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
