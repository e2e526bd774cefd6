// Sparse group normalisation (Eqs. 7-9): for every frame b and channel group
// g, mean and variance over the frame's active rows [offsets[b], offsets[b+1])
// and the group's C/G channels only, then (x - mean) / sqrt(var + eps),
// optional per-channel affine, and the activation of Eq. 10 fused.
//
// Statistics. Values are read in chunks; per chunk its mean (shifted by the
// chunk's first value) and centred sum of squares, merged into a running
// (count, mean, M2) by the pairwise update of Chan, Golub and LeVeque, and
// partial results merged the same way. The variance is never formed as
// E[x^2] - mean^2, and a group of equal values gets exactly that mean and
// M2 = 0, so it normalises to exactly 0. All in fp32: GB300's fp64 rate is
// far too low for a bandwidth-bound kernel.
//
// Fast path (rows in 16-byte chunks, C/VEC a power of two <= 256, and either
// VEC | C/G or C/G | VEC): the compact rows [offsets[0], offsets[B]) are cut
// into gridDim.x equal contiguous ranges, one per CTA, independent of frame
// boundaries. That balances the load whatever the frame sizes, and whole
// rows are read with coalesced 16-byte loads; each thread owns one chunk
// column, hence a fixed set of groups and fixed gamma/beta values.
//   gn_stats_kernel: per frame segment of its range, a block merge per group
//     and one partial (n, mean, M2) per (frame b, CTA c), written to slot
//     b + c of the workspace. Frames are contiguous and in order, so the
//     slots of frame b, b + [first CTA, last CTA], end before those of frame
//     b + 1 begin: slots never collide and (B + gridDim.x) * G suffice.
//   gn_apply_kernel: same ranges; per frame segment, merge the partials of
//     the CTAs that hold the frame, normalise and store. Segments and rows
//     are walked in reverse, so the most recently read rows, still in L2,
//     are consumed first, and its loads and stores carry an L2 evict-first
//     policy (last use), which keeps the rest of the input in L2.
// Frames are located by a kThreads-ary block search of the frame table and
// read a window of kThreads frames at a time into shared memory; loads are
// issued a batch ahead of the arithmetic.
// The general path (one CTA per (frame, group)) serves every other layout,
// and small frames (a group slice within its register cache), where one
// launch beats the two latency-bound row-range launches.
// Partials from the convolution: the tensor-core convolution can write the
// (n, mean, M2) partials of its stored output itself, one per (frame b,
// 32-row block c lying inside the frame) in slot b + c (the slot argument
// above with ranges of 32 rows), and one per row for the rows of blocks that
// straddle a frame boundary, so that gn_apply_kernel alone finishes the
// layer.
// The output may alias the input in both paths. Deterministic, no atomics.
#include <cuda_bf16.h>

#include <cstdlib>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kThreads = 256;
constexpr int kBatch = 4;
constexpr int kMaxGroupsFast = 2048;
constexpr int kMergeBatch = 4;  // partials a lane loads before merging them

// VEC consecutive elements as one raw chunk (16 bytes when VEC > 1).
template <typename T, int VEC>
struct Chunk;
template <>
struct Chunk<float, 1> {
    using Raw = float;
    static __device__ __forceinline__ Raw load(const float* p) { return *p; }
    static __device__ __forceinline__ void unpack(Raw r, float* v) { v[0] = r; }
    static __device__ __forceinline__ void store(float* p, const float* v) { *p = v[0]; }
};
template <>
struct Chunk<float, 4> {
    using Raw = float4;
    static __device__ __forceinline__ Raw load(const float* p) {
        return *reinterpret_cast<const float4*>(p);
    }
    static __device__ __forceinline__ void unpack(Raw r, float* v) {
        v[0] = r.x, v[1] = r.y, v[2] = r.z, v[3] = r.w;
    }
    static __device__ __forceinline__ void store(float* p, const float* v) {
        *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    }
};
template <>
struct Chunk<__nv_bfloat16, 1> {
    using Raw = __nv_bfloat16;
    static __device__ __forceinline__ Raw load(const __nv_bfloat16* p) { return *p; }
    static __device__ __forceinline__ void unpack(Raw r, float* v) { v[0] = __bfloat162float(r); }
    static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
        *p = __float2bfloat16_rn(v[0]);
    }
};
template <>
struct Chunk<__nv_bfloat16, 8> {
    using Raw = uint4;
    static __device__ __forceinline__ Raw load(const __nv_bfloat16* p) {
        return *reinterpret_cast<const uint4*>(p);
    }
    static __device__ __forceinline__ void unpack(Raw r, float* v) {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            v[2 * k] = __uint_as_float(w[k] << 16);
            v[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
        }
    }
    static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
        uint32_t w[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * k], v[2 * k + 1]);
            w[k] = *reinterpret_cast<const uint32_t*>(&h);
        }
        *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
    }
};

// 16-byte accesses with an L2 evict-first policy (last use of a line).
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ uint4 ld_ef(const void* p, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}
__device__ __forceinline__ void st_ef(void* p, uint4 v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "r"(v.x),
                 "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol)
                 : "memory");
}
template <typename Raw>
__device__ __forceinline__ Raw as_raw(uint4 v) {
    return *reinterpret_cast<const Raw*>(&v);
}
template <typename Raw>
__device__ __forceinline__ uint4 as_u4(const Raw& v) {
    return *reinterpret_cast<const uint4*>(&v);
}

// Running (count, mean, M2), fp32. Counts are exact integers below 2^24.
struct Stats {
    float n = 0.f, mean = 0.f, m2 = 0.f;
    template <int VEC>
    __device__ __forceinline__ void add_chunk(const float* v) {
        float s = 0.f;
#pragma unroll
        for (int k = 1; k < VEC; ++k) s += v[k] - v[0];
        const float cm = v[0] + s * (1.f / VEC);
        float q = 0.f;
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
            const float d = v[k] - cm;
            q = fmaf(d, d, q);
        }
        const float nn = n + (float)VEC;
        const float d = cm - mean;
        const float r = (float)VEC * __frcp_rn(nn);
        mean = fmaf(d, r, mean);
        m2 += q + d * d * n * r;
        n = nn;
    }
};

// Pairwise merge of (nb, mb, qb) into (n, mean, m2).
__device__ __forceinline__ void merge(float& n, float& mean, float& m2, float nb, float mb,
                                      float qb) {
    if (nb == 0.f) return;
    const float nn = n + nb;
    const float d = mb - mean;
    const float r = nb * __frcp_rn(nn);
    mean = fmaf(d, r, mean);
    m2 += qb + d * d * n * r;
    n = nn;
}

__device__ __forceinline__ void merge_xor(float& n, float& mean, float& m2, int o) {
    const float nb = __shfl_xor_sync(0xffffffffu, n, o);
    const float mb = __shfl_xor_sync(0xffffffffu, mean, o);
    const float qb = __shfl_xor_sync(0xffffffffu, m2, o);
    merge(n, mean, m2, nb, mb, qb);
}

// Merge over the whole block; every thread gets the result.
__device__ __forceinline__ void block_merge(float& n, float& mean, float& m2, float* red) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) merge_xor(n, mean, m2, o);
    if ((threadIdx.x & 31) == 0) {
        red[3 * (threadIdx.x >> 5)] = n;
        red[3 * (threadIdx.x >> 5) + 1] = mean;
        red[3 * (threadIdx.x >> 5) + 2] = m2;
    }
    __syncthreads();
    n = mean = m2 = 0.f;
#pragma unroll
    for (int w = 0; w < kThreads / 32; ++w)
        merge(n, mean, m2, red[3 * w], red[3 * w + 1], red[3 * w + 2]);
}

// ---- fast path: contiguous row ranges ------------------------------------
struct GnPart {
    float n, mean, m2, pad;
};

// Row range of CTA c over [off0, end): R = ceil((end - off0) / grid).
struct RangeMap {
    long long off0, end, R;
    __device__ __forceinline__ long long cta_of(long long row) const { return (row - off0) / R; }
};

// First frame b in [0, B] with offsets[b + 1] > row (B if none): a
// kThreads-ary search, every thread of the block taking part, so one round
// trip to the table per factor of kThreads frames. A malformed (unsorted)
// table yields some b in [0, B].
__device__ __forceinline__ int find_frame(const int32_t* offsets, int B, long long row) {
    long long wlo = 0, whi = B;
    while (whi > wlo) {
        const long long step = (whi - wlo + kThreads - 1) / kThreads;
        const long long p = wlo + (long long)threadIdx.x * step;
        const int before = p < whi && (long long)__ldg(offsets + p + 1) <= row;
        const int k = __syncthreads_count(before);
        if (step == 1) return (int)(wlo + k);
        const long long nlo = k == 0 ? wlo : wlo + (long long)(k - 1) * step + 1;
        const long long nhi = wlo + (long long)k * step < whi ? wlo + (long long)k * step : whi;
        wlo = nlo;
        whi = nhi;
    }
    __syncthreads();  // every exit path passes the same number of barriers
    return (int)wlo;
}

// offsets[wb + j] for j in [0, n] into s_off (n <= kThreads).
__device__ __forceinline__ void load_window(const int32_t* offsets, int wb, int n, int* s_off) {
    __syncthreads();  // the previous window is no longer read
    for (int j = threadIdx.x; j <= n; j += kThreads) s_off[j] = __ldg(offsets + wb + j);
    __syncthreads();
}

// Thread layout: cpr chunks per row; thread t owns chunk column t % cpr and
// rows rg, rg + rpp, ... of a segment (rg = t / cpr, rpp = kThreads / cpr).
// GPC groups per chunk when a group is narrower than a chunk, else 1 (the
// chunk lies in group col / cpc, cpc = chunks per group).
struct Layout {
    int cpr, rpp, col, rg, cpc;
};

template <int VEC, int GPC>
__device__ __forceinline__ Layout make_layout(int C, int G) {
    Layout l;
    l.cpr = C / VEC;
    l.rpp = kThreads / l.cpr;
    l.col = threadIdx.x % l.cpr;
    l.rg = threadIdx.x / l.cpr;
    l.cpc = GPC == 1 ? (C / G) / VEC : 1;
    return l;
}

// This CTA's row range [lo, hi); false if there is nothing to do or the
// frame table's span is unusable (reported).
__device__ __forceinline__ bool range_from(long long o0, long long oB, long long capacity,
                                           unsigned* status, RangeMap& m, long long& lo,
                                           long long& hi) {
    if (o0 < 0 || oB < o0 || oB > capacity) {
        if (threadIdx.x == 0 && blockIdx.x == 0) report(status, kErrIndex);
        return false;
    }
    const long long total = oB - o0;
    if (total == 0) return false;
    m.off0 = o0;
    m.end = oB;
    m.R = (total + gridDim.x - 1) / gridDim.x;
    lo = o0 + (long long)blockIdx.x * m.R;
    hi = lo + m.R < oB ? lo + m.R : oB;
    return lo < hi;
}

__device__ __forceinline__ bool range_setup(const int32_t* offsets, int B, long long capacity,
                                            unsigned* status, RangeMap& m, long long& lo,
                                            long long& hi) {
    return range_from(__ldg(offsets), __ldg(offsets + B), capacity, status, m, lo, hi);
}

template <typename T, int VEC, int GPC>
__global__ void __launch_bounds__(kThreads, 2)
    gn_stats_kernel(const T* x, const int32_t* __restrict__ offsets, int B, int C, int G,
                    long long capacity, GnPart* __restrict__ part, unsigned* status) {
    using CK = Chunk<T, VEC>;
    using Raw = typename CK::Raw;
    constexpr int SUB = VEC / GPC;  // elements of one group inside a chunk (GPC > 1)
    __shared__ float red[kThreads * GPC * 3];
    __shared__ int s_off[kThreads + 1];
    pdl_wait();
    pdl_trigger();
    // frames must be in order (each CTA checks a share of the table)
    for (long long i = (long long)blockIdx.x * kThreads + threadIdx.x; i < B;
         i += (long long)gridDim.x * kThreads)
        if (__ldg(offsets + i + 1) < __ldg(offsets + i)) report(status, kErrIndex);
    RangeMap m;
    long long lo, hi;
    if (!range_setup(offsets, B, capacity, status, m, lo, hi)) return;
    const Layout l = make_layout<VEC, GPC>(C, G);
    // after the warp merge: row slots (warps, or thread rows) x cpr columns
    const int nrs = l.cpr < 32 ? kThreads / 32 : kThreads / l.cpr;
    const long long step = (long long)kBatch * l.rpp;

    auto segment = [&](int b, long long s0, long long s1) {
        Stats st[GPC];
        Raw cur[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const long long r = s0 + l.rg + (long long)i * l.rpp;
            if (r < s1) cur[i] = CK::load(x + r * C + l.col * VEC);
        }
        for (long long r0 = s0 + l.rg; r0 < s1; r0 += step) {
            Raw nxt[kBatch];  // next batch in flight while this one is reduced
#pragma unroll
            for (int i = 0; i < kBatch; ++i) {
                const long long r = r0 + step + (long long)i * l.rpp;
                if (r < s1) nxt[i] = CK::load(x + r * C + l.col * VEC);
            }
#pragma unroll
            for (int i = 0; i < kBatch; ++i) {
                if (r0 + (long long)i * l.rpp < s1) {
                    float v[VEC];
                    CK::unpack(cur[i], v);
#pragma unroll
                    for (int q = 0; q < GPC; ++q) st[q].template add_chunk<SUB>(v + q * SUB);
                }
            }
#pragma unroll
            for (int i = 0; i < kBatch; ++i) cur[i] = nxt[i];
        }
        // lanes holding the same column: merge across the warp
#pragma unroll
        for (int q = 0; q < GPC; ++q)
            for (int o = l.cpr; o < 32; o <<= 1) merge_xor(st[q].n, st[q].mean, st[q].m2, o);
        const int lane = threadIdx.x & 31;
        __syncthreads();  // red[] of the previous segment has been read
        if (l.cpr >= 32 || lane < l.cpr) {
            const int slot = l.cpr < 32 ? (int)(threadIdx.x >> 5) : l.rg;
#pragma unroll
            for (int q = 0; q < GPC; ++q) {
                float* e = red + 3 * ((slot * l.cpr + l.col) * GPC + q);
                e[0] = st[q].n, e[1] = st[q].mean, e[2] = st[q].m2;
            }
        }
        __syncthreads();
        GnPart* out = part + (long long)(b + blockIdx.x) * G;
        for (int g = threadIdx.x; g < G; g += kThreads) {
            const int c0 = GPC == 1 ? g * l.cpc : g / GPC, nc = GPC == 1 ? l.cpc : 1;
            const int q = GPC == 1 ? 0 : g % GPC;
            float n = 0.f, mean = 0.f, m2 = 0.f;
            for (int rs = 0; rs < nrs; ++rs)
                for (int c = c0; c < c0 + nc; ++c) {
                    const float* e = red + 3 * ((rs * l.cpr + c) * GPC + q);
                    merge(n, mean, m2, e[0], e[1], e[2]);
                }
            out[g] = GnPart{n, mean, m2, 0.f};
        }
    };

    // frames overlapping [lo, hi), a window of kThreads frames at a time
    for (int wb = find_frame(offsets, B, lo); wb < B; wb += kThreads) {
        const int nw = B - wb < kThreads ? B - wb : kThreads;
        load_window(offsets, wb, nw, s_off);
        bool past = false;
        for (int j = 0; j < nw; ++j) {
            const long long f0 = s_off[j], f1 = s_off[j + 1];
            if (f0 >= hi) {
                past = true;
                break;
            }
            const long long s0 = f0 > lo ? f0 : lo, s1 = f1 < hi ? f1 : hi;
            if (s0 < s1) segment(wb + j, s0, s1);  // f1 < f0 is reported above
        }
        if (past || (long long)s_off[nw] >= hi) break;
    }
}

template <typename T, int VEC, int GPC>
__global__ void __launch_bounds__(kThreads, 2)
    gn_apply_kernel(const T* x, const int32_t* __restrict__ offsets, int B, int C, int G,
                    long long capacity, const GnPart* __restrict__ part, float eps,
                    const float* __restrict__ gamma, const float* __restrict__ beta, int act, T* y,
                    int part_rows, const float2* __restrict__ row_part,
                    const int32_t* __restrict__ count, unsigned* status) {
    using CK = Chunk<T, VEC>;
    using Raw = typename CK::Raw;
    static_assert(sizeof(Raw) == 16, "the row-range path moves 16-byte chunks");
    constexpr int SUB = VEC / GPC;
    __shared__ float s_mu[kMaxGroupsFast], s_inv[kMaxGroupsFast];
    __shared__ int s_off[kThreads + 1];
    // part_rows > 0: the partials come from the convolution (the kernel
    // before this one) over the rows [0, *count): one per (frame b, block c
    // of part_rows rows inside the frame) in slot b + c, one per row
    // (row_part, C/G values each) for the frame's other rows. The frame table
    // must cover exactly those rows, in order (checked here, as the
    // statistics kernel does otherwise). The table, count, gamma and
    // beta were written before that convolution started, so they are read
    // before waiting for it: the set-up overlaps its last blocks.
    __shared__ int s_count;
    const bool early = part_rows > 0;
    if (!early) pdl_wait();
    pdl_trigger();
    const Layout l = make_layout<VEC, GPC>(C, G);
    float ga[VEC], be[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) {
        ga[k] = gamma ? __ldg(gamma + l.col * VEC + k) : 1.f;
        be[k] = beta ? __ldg(beta + l.col * VEC + k) : 0.f;
    }
    // B <= kThreads: the whole frame table (and the row count) in one round
    // trip; the checks and the row range then come from shared memory
    const bool small = B <= kThreads;
    if (small) {
        for (int j = threadIdx.x; j <= B; j += kThreads) s_off[j] = __ldg(offsets + j);
        if (threadIdx.x == 0) s_count = early ? __ldg(count) : 0;
        __syncthreads();
    }
    if (early) {
        if (small) {
            if (threadIdx.x < B && s_off[threadIdx.x + 1] < s_off[threadIdx.x])
                report(status, kErrIndex);
        } else {
            for (long long i = (long long)blockIdx.x * kThreads + threadIdx.x; i < B;
                 i += (long long)gridDim.x * kThreads)
                if (__ldg(offsets + i + 1) < __ldg(offsets + i)) report(status, kErrIndex);
        }
        const int o0 = small ? s_off[0] : __ldg(offsets), oB = small ? s_off[B] : __ldg(offsets + B);
        const int n = small ? s_count : __ldg(count);
        if (o0 != 0 || oB != n) {
            if (threadIdx.x == 0 && blockIdx.x == 0) report(status, kErrIndex);
            return;
        }
    }
    RangeMap m;
    long long lo, hi;
    if (small) {
        if (!range_from(s_off[0], s_off[B], capacity, status, m, lo, hi)) return;
    } else if (!range_setup(offsets, B, capacity, status, m, lo, hi)) {
        return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long step = (long long)kBatch * l.rpp;
    const uint64_t pol = l2_evict_first_policy();

    auto segment = [&](int b, long long f0, long long f1, long long s0, long long s1) {
        // partials of the CTAs that hold frame b: slots b + c, c in [c0, c1]
        // (clamped to the table's span, so a malformed table cannot index
        // outside the workspace)
        const long long p0 = f0 > m.off0 ? f0 : m.off0, p1 = (f1 < m.end ? f1 : m.end) - 1;
        const long long c0 = m.cta_of(p0), c1 = m.cta_of(p1);
        const GnPart* pb = part + (long long)b * G;
        // rows of the segment last to first (the statistics pass read them
        // first to last, so the most recent ones are still in L2); every
        // line is read and written here for the last time: evict first. The
        // first batch is issued before the partials are merged.
        auto row_at = [&](long long r) { return (s0 + r) * C + l.col * VEC; };
        const long long top = (s1 - s0) - 1 - l.rg;  // this thread's highest row offset
        Raw cur[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i)
            if (top - (long long)i * l.rpp >= 0)
                cur[i] = as_raw<Raw>(ld_ef(x + row_at(top - (long long)i * l.rpp), pol));
        __syncthreads();  // s_mu / s_inv of the previous segment have been read
        if (part_rows > 0) {
            // whole blocks [w0, w1) of the frame's rows [p0, p1], and its
            // other rows (at most 2 * part_rows - 2) [p0, h1) and [t0, p1]
            const long long P = part_rows, w0 = (p0 + P - 1) / P, w1 = (p1 + 1) / P;
            const bool any = w0 < w1;
            const long long nw = any ? w1 - w0 : 0;
            const long long h1 = any ? w0 * P : p1 + 1, t0 = any ? w1 * P : p1 + 1;
            const long long nh = h1 - p0, items = nw + nh + (p1 + 1 - t0);
            const float cpg = (float)(C / G);
            for (int g = warp; g < G; g += kThreads / 32) {
                float n = 0.f, mean = 0.f, m2 = 0.f;
                // kMergeBatch items per lane loaded together, then merged
                for (long long i0 = lane; i0 < items; i0 += 32 * kMergeBatch) {
                    float4 q[kMergeBatch];
#pragma unroll
                    for (int k = 0; k < kMergeBatch; ++k) {
                        const long long i = i0 + 32 * k;
                        q[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                        if (i < nw) {
                            const GnPart p = pb[(w0 + i) * G + g];
                            q[k] = make_float4(p.n, p.mean, p.m2, 0.f);
                        } else if (i < items) {
                            const long long r = i - nw < nh ? p0 + (i - nw) : t0 + (i - nw - nh);
                            const float2 v = row_part[r * G + g];
                            q[k] = make_float4(cpg, v.x, v.y, 0.f);
                        }
                    }
#pragma unroll
                    for (int k = 0; k < kMergeBatch; ++k) merge(n, mean, m2, q[k].x, q[k].y, q[k].z);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) merge_xor(n, mean, m2, o);
                if (lane == 0) {
                    s_mu[g] = mean;
                    s_inv[g] = 1.f / sqrtf(m2 / n + eps);
                }
            }
        } else if (c1 - c0 < 8) {
            for (int g = threadIdx.x; g < G; g += kThreads) {
                float n = 0.f, mean = 0.f, m2 = 0.f;
                for (long long c = c0; c <= c1; ++c) {
                    const GnPart q = pb[c * G + g];
                    merge(n, mean, m2, q.n, q.mean, q.m2);
                }
                s_mu[g] = mean;
                s_inv[g] = 1.f / sqrtf(m2 / n + eps);
            }
        } else {
            for (int g = warp; g < G; g += kThreads / 32) {
                float n = 0.f, mean = 0.f, m2 = 0.f;
                for (long long c = c0 + lane; c <= c1; c += 32) {
                    const GnPart q = pb[c * G + g];
                    merge(n, mean, m2, q.n, q.mean, q.m2);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) merge_xor(n, mean, m2, o);
                if (lane == 0) {
                    s_mu[g] = mean;
                    s_inv[g] = 1.f / sqrtf(m2 / n + eps);
                }
            }
        }
        __syncthreads();
        float mu[GPC], inv[GPC];
#pragma unroll
        for (int q = 0; q < GPC; ++q) {
            const int g = GPC == 1 ? l.col / l.cpc : l.col * GPC + q;
            mu[q] = s_mu[g];
            inv[q] = s_inv[g];
        }
        for (long long r0 = top; r0 >= 0; r0 -= step) {
            Raw nxt[kBatch];
#pragma unroll
            for (int i = 0; i < kBatch; ++i) {
                const long long r = r0 - step - (long long)i * l.rpp;
                if (r >= 0) nxt[i] = as_raw<Raw>(ld_ef(x + row_at(r), pol));
            }
#pragma unroll
            for (int i = 0; i < kBatch; ++i) {
                const long long r = r0 - (long long)i * l.rpp;
                if (r >= 0) {
                    float v[VEC];
                    CK::unpack(cur[i], v);
#pragma unroll
                    for (int k = 0; k < VEC; ++k) {
                        const int q = k / SUB;
                        const float z = fmaf((v[k] - mu[q]) * inv[q], ga[k], be[k]);
                        v[k] = act_apply(z, act);
                    }
                    T* dst = y + row_at(r);
                    Raw packed;
                    CK::store(reinterpret_cast<T*>(&packed), v);
                    st_ef(dst, as_u4(packed), pol);
                }
            }
#pragma unroll
            for (int i = 0; i < kBatch; ++i) cur[i] = nxt[i];
        }
    };

    // frames overlapping [lo, hi) of a window (frames wb .. wb + nw - 1, so
    // holding offsets[wb + j]), last to first; true when hi is reached
    auto walk = [&](int wb, int nw, const int* so) {
        int nf = 0;  // frames of the window that start before hi
        while (nf < nw && (long long)so[nf] < hi) ++nf;
        if (early) pdl_wait();  // x and the partials come from the convolution
        for (int j = nf - 1; j >= 0; --j) {
            const long long f0 = so[j], f1 = so[j + 1];
            if (f1 < f0) continue;  // reported by the statistics kernel
            const long long s0 = f0 > lo ? f0 : lo, s1 = f1 < hi ? f1 : hi;
            if (s0 < s1) segment(wb + j, f0, f1, s0, s1);
        }
        return nf < nw || (long long)so[nw] >= hi;
    };
    if (small) {
        // the first frame of the range (the number of frames ending at or
        // before lo), found in the table in shared memory
        const int wb =
            __syncthreads_count(threadIdx.x < B && (long long)s_off[threadIdx.x + 1] <= lo);
        if (wb < B) walk(wb, B - wb, s_off + wb);
        return;
    }
    // windows of kThreads frames
    for (int wb = find_frame(offsets, B, lo); wb < B; wb += kThreads) {
        const int nw = B - wb < kThreads ? B - wb : kThreads;
        load_window(offsets, wb, nw, s_off);
        if (walk(wb, nw, s_off)) break;
    }
}

// ---- general path: one CTA per (frame, group) ----------------------------
// Any C, G and alignment. The group's part of a row is read in chunks of VEC
// elements (16 bytes, or single elements); chunk e of the slice is at row
// r0 + e / vpr, channel c0 + (e % vpr) * VEC. The first batch of every
// thread stays in registers; pass 2 walks the other batches in reverse.
struct SliceMap {
    long long r0;
    int C, c0, vpr, VEC;
    bool narrow;  // 32-bit division suffices
    __device__ __forceinline__ long long at(long long e, int& c) const {
        long long q;
        int rem;
        if (narrow) {
            const unsigned qe = (unsigned)e / (unsigned)vpr;
            q = qe;
            rem = (int)((unsigned)e - qe * (unsigned)vpr);
        } else {
            q = e / vpr;
            rem = (int)(e - q * vpr);
        }
        c = c0 + rem * VEC;
        return (r0 + q) * C + c;
    }
};

template <typename T, int VEC>
__global__ void __launch_bounds__(kThreads, 4)
    group_norm_slice_kernel(const T* x, const int32_t* __restrict__ offsets, int C, int G,
                            long long capacity, float eps, const float* __restrict__ gamma,
                            const float* __restrict__ beta, int act, T* y, unsigned* status) {
    using CK = Chunk<T, VEC>;
    using Raw = typename CK::Raw;
    constexpr long long kStride = (long long)kThreads * kBatch;
    __shared__ float red[3 * (kThreads / 32)];
    pdl_wait();
    pdl_trigger();
    const int b = blockIdx.x / G, g = blockIdx.x - b * G;
    const long long r0 = __ldg(offsets + b), r1 = __ldg(offsets + b + 1);
    if (r0 < 0 || r1 < r0 || r1 > capacity) {
        if (threadIdx.x == 0) report(status, kErrIndex);
        return;
    }
    const int cpg = C / G;
    const SliceMap map{r0, C, g * cpg, cpg / VEC, VEC, (r1 - r0) * (cpg / VEC) < (1ll << 31)};
    const long long nv = (r1 - r0) * map.vpr;
    if (nv == 0) return;

    // pass 1: statistics
    Raw keep[kBatch];
    Stats st;
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
        const long long e = threadIdx.x + (long long)i * kThreads;
        int c;
        if (e < nv) keep[i] = CK::load(x + map.at(e, c));
    }
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
        if (threadIdx.x + (long long)i * kThreads < nv) {
            float v[VEC];
            CK::unpack(keep[i], v);
            st.add_chunk<VEC>(v);
        }
    }
    for (long long base = threadIdx.x + kStride; base < nv; base += kStride) {
        Raw t[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            int c;
            if (base + (long long)i * kThreads < nv)
                t[i] = CK::load(x + map.at(base + i * kThreads, c));
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            if (base + (long long)i * kThreads < nv) {
                float v[VEC];
                CK::unpack(t[i], v);
                st.add_chunk<VEC>(v);
            }
        }
    }
    float n = st.n, mean = st.mean, m2 = st.m2;
    block_merge(n, mean, m2, red);
    const float mu = mean;
    const float inv = 1.f / sqrtf(m2 / n + eps);

    // pass 2: normalise, affine, activation, store
    auto finish = [&](Raw r, long long off, int c) {
        float v[VEC];
        CK::unpack(r, v);
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
            float z = (v[k] - mu) * inv;
            if (gamma) z *= __ldg(gamma + c + k);
            if (beta) z += __ldg(beta + c + k);
            v[k] = act_apply(z, act);
        }
        CK::store(y + off, v);
    };
    for (long long j = (nv - 1) / kStride; j >= 1; --j) {
        const long long base = threadIdx.x + j * kStride;
        Raw t[kBatch];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            int c;
            if (base + (long long)i * kThreads < nv)
                t[i] = CK::load(x + map.at(base + i * kThreads, c));
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            if (base + (long long)i * kThreads < nv) {
                int c;
                const long long off = map.at(base + i * kThreads, c);
                finish(t[i], off, c);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
        const long long e = threadIdx.x + (long long)i * kThreads;
        if (e < nv) {
            int c;
            const long long off = map.at(e, c);
            finish(keep[i], off, c);
        }
    }
}

long long fast_grid(const DeviceCtx* ctx, long long capacity) {
    // ranges of at least ~64 rows; 2 CTAs per SM at most (the kernels' bound)
    long long grid = (capacity + 63) / 64;
    const long long cap = (long long)ctx->num_sms * 2;
    if (grid > cap) grid = cap;
    return grid < 1 ? 1 : grid;
}

template <typename T, int VEC, int GPC>
hc_status launch_fast(const DeviceCtx* ctx, const void* x, const int32_t* offsets, int B,
                      long long capacity, int C, int G, float eps, const float* gamma,
                      const float* beta, int act, void* y, cudaStream_t s) {
    const long long grid = fast_grid(ctx, capacity);
    GnPart* part = (GnPart*)stream_workspace(s, sizeof(GnPart) * (size_t)(B + grid) * G);
    if (!part) return HC_ERR_CUDA;
    hc_status st = launch_pdl(gn_stats_kernel<T, VEC, GPC>, dim3((unsigned)grid), dim3(kThreads),
                              0, s, "gn_stats_kernel", (const T*)x, offsets, B, C, G, capacity,
                              part, ctx->status);
    if (st != HC_OK) return st;
    return launch_pdl(gn_apply_kernel<T, VEC, GPC>, dim3((unsigned)grid), dim3(kThreads), 0, s,
                      "gn_apply_kernel", (const T*)x, offsets, B, C, G, capacity,
                      (const GnPart*)part, eps, gamma, beta, act, (T*)y, 0,
                      (const float2*)nullptr, (const int32_t*)nullptr, ctx->status);
}


template <typename T>
hc_status launch_typed(const DeviceCtx* ctx, const void* x, const int32_t* offsets, int B,
                       long long capacity, int C, int G, float eps, const float* gamma,
                       const float* beta, int act, void* y, cudaStream_t s) {
    constexpr int kVec = 16 / (int)sizeof(T);
    const int cpg = C / G;
    const uintptr_t al = (uintptr_t)x | (uintptr_t)y;
    const bool aligned = C % kVec == 0 && al % 16 == 0;
    const int cpr = C / kVec;
    // Small frames: when the average frame's group slice is within twice
    // the per-thread register cache of the per-(frame, group) kernel (the
    // rest re-read from L2) and there are enough (frame, group) blocks to
    // fill the GPU, that single launch beats the two latency-bound row-range
    // launches.
    const long long avg_chunks = (capacity + B - 1) / B * (long long)(cpg / kVec);
    const bool small_frames = cpg % kVec == 0 && aligned &&
                              avg_chunks <= 2ll * kThreads * kBatch &&
                              (long long)B * G >= ctx->num_sms;
    // a test may force the per-(frame, group) kernel (1) or the row-range
    // kernels where the layout allows (2), to cover both on any shape
    const int forced = test_group_norm_path();
    const bool force_slice = forced == 1;
    const bool force_rows = forced == 2;
    const bool fast_rows = aligned && cpr >= 1 && cpr <= kThreads && (cpr & (cpr - 1)) == 0 &&
                           G <= kMaxGroupsFast && !force_slice && (force_rows || !small_frames);
    if (fast_rows && cpg % kVec == 0)
        return launch_fast<T, kVec, 1>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta, act,
                                       y, s);
    if (fast_rows && kVec % cpg == 0) {
        if (kVec / cpg == 2)
            return launch_fast<T, kVec, 2>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta,
                                           act, y, s);
        if (kVec / cpg == 4)
            return launch_fast<T, kVec, 4>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta,
                                           act, y, s);
        if constexpr (kVec == 8)
            return launch_fast<T, kVec, 8>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta,
                                           act, y, s);
    }
    const dim3 grid((unsigned)((long long)B * G));
    if (cpg % kVec == 0 && aligned)
        return launch_pdl(group_norm_slice_kernel<T, kVec>, grid, dim3(kThreads), 0, s,
                          "group_norm_slice_kernel", (const T*)x, offsets, C, G, capacity, eps,
                          gamma, beta, act, (T*)y, ctx->status);
    return launch_pdl(group_norm_slice_kernel<T, 1>, grid, dim3(kThreads), 0, s,
                      "group_norm_slice_kernel", (const T*)x, offsets, C, G, capacity, eps, gamma,
                      beta, act, (T*)y, ctx->status);
}

}  // namespace

bool group_norm_parts_supported(hc_dtype dt, int C, int G, const void* y) {
    const int cpr = C / 8;
    return dt == HC_BF16 && C % 8 == 0 && (C / G) % 8 == 0 && (uintptr_t)y % 16 == 0 &&
           cpr >= 1 && cpr <= kThreads && (cpr & (cpr - 1)) == 0 && G <= kMaxGroupsFast;
}

hc_status launch_group_norm_apply(const DeviceCtx* ctx, void* y, const int32_t* offsets, int B,
                                  long long capacity, int C, int G, const float* part,
                                  const float* rows, int part_rows, const int32_t* count,
                                  float eps, const float* gamma, const float* beta, int act,
                                  cudaStream_t s) {
    using T = __nv_bfloat16;
    return launch_pdl(gn_apply_kernel<T, 8, 1>, dim3((unsigned)fast_grid(ctx, capacity)),
                      dim3(kThreads), 0, s, "gn_apply_kernel", (const T*)y, offsets, B, C, G,
                      capacity, (const GnPart*)part, eps, gamma, beta, act, (T*)y, part_rows,
                      (const float2*)rows, count, ctx->status);
}

hc_status launch_group_norm(const DeviceCtx* ctx, const void* x, hc_dtype dt,
                            const int32_t* offsets, int B, long long capacity, int C, int G,
                            float eps, const float* gamma, const float* beta, int act, void* y,
                            cudaStream_t s) {
    if (dt == HC_F32)
        return launch_typed<float>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta, act, y, s);
    return launch_typed<__nv_bfloat16>(ctx, x, offsets, B, capacity, C, G, eps, gamma, beta, act,
                                       y, s);
}

}  // namespace hc
