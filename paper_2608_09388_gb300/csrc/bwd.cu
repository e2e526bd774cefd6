// Backward of the sparse spiral convolution (the chain rule on Eqs. 4-5, 6
// and 10; the paper gives the forward only). Through the Eq. 4 mapping
// rulebook[l][n] = input row j read by tap l of output row n (or -1):
//   dz[n][o]  = dy[n][o] * act'(y[n][o])           act' read off the output
//   dbias[o]  = sum_n dz[n][o]
//   dW[l*C_in + c][o] = sum_n x[j(n,l)][c] * dz[n][o]
//   dx[j][c]  = sum over taps (n, l) reading j of (dz[n] W_l^T)[c]
// Kernels (every sum in a fixed order, no floating-point atomics):
//   act_bwd_kernel      dz (stored in the layer dtype) and per-block column
//                       sums of dz in fp32; dbias_kernel adds the blocks.
//   wgrad (tcgen05)     split-K [L*C_in] x [C_out] tiles: A = the gathered
//                       input rows (cp.async through the rulebook), B = dz,
//                       both MN-major, fp32 accumulators in TMEM; fp32 on
//                       CUDA cores otherwise. wgrad_reduce adds the splits.
//   dgrad               P = dz W^T by the linear conv kernels (W^T
//                       materialised once), then every input row sums the P
//                       slices of the taps that read it, in (n, l) order,
//                       from the transposed mapping (rb_* kernels: counts,
//                       exclusive scan, fill, per-row sort), a warp per 32
//                       rows where the channel chunks allow it.
#include <cuda_bf16.h>

#include "hc_internal.cuh"

namespace hc {
namespace {

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) {
    return v;
}
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) {
    return __bfloat162float(v);
}
template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) {
    return v;
}
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

__device__ __forceinline__ long long clamp_rows(const int32_t* count, long long capacity,
                                                unsigned* status) {
    long long n = *count;
    if (n < 0) {
        if (blockIdx.x == 0 && threadIdx.x == 0) report(status, kErrIndex);
        return 0;
    }
    if (n > capacity) {
        if (blockIdx.x == 0 && threadIdx.x == 0) report(status, kErrCapacity);
        return capacity;
    }
    return n;
}

// ---------------------------------------------------------------- dz, dbias
// Block (64, 4): thread (tx, ty) takes columns g*64 + tx of rows r0 + ty +
// 4 i of the block's row chunks (chunks blockIdx.x, + gridDim.x, ...); the
// four row lanes' sums meet in shared memory and the block writes one
// partial per column.
constexpr int kActRowsPerBlock = 16;

template <typename T>
__global__ void __launch_bounds__(256)
    act_bwd_kernel(const T* __restrict__ y, const T* __restrict__ dy, const int32_t* count,
                   long long capacity, int C_out, int act, T* __restrict__ dz,
                   float* __restrict__ bpart, unsigned* status) {
    __shared__ float red[4][64];
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    const int tx = threadIdx.x & 63, ty = threadIdx.x >> 6;
    for (int g0 = 0; g0 < C_out; g0 += 64) {
        const int o = g0 + tx;
        float sum = 0.f;
        if (o < C_out)
            for (long long r0 = (long long)blockIdx.x * kActRowsPerBlock; r0 < rows;
                 r0 += (long long)gridDim.x * kActRowsPerBlock) {
                const long long r1 = r0 + kActRowsPerBlock < rows ? r0 + kActRowsPerBlock : rows;
                for (long long rb0 = r0 + ty; rb0 < r1; rb0 += 16) {
                    // four rows' loads in flight, then their arithmetic
                    float yv[4], gv[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const long long r = rb0 + 4 * i;
                        yv[i] = r < r1 ? to_f(y[r * C_out + o]) : 0.f;
                        gv[i] = r < r1 ? to_f(dy[r * C_out + o]) : 0.f;
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const long long r = rb0 + 4 * i;
                        if (r >= r1) continue;
                        float d = 1.f;
                        if (act == HC_ACT_ELU) d = yv[i] > 0.f ? 1.f : yv[i] + 1.f;
                        else if (act == HC_ACT_RELU) d = yv[i] > 0.f ? 1.f : 0.f;
                        const float v = gv[i] * d;
                        dz[r * C_out + o] = from_f<T>(v);
                        sum += v;
                    }
                }
            }
        red[ty][tx] = sum;
        __syncthreads();
        if (ty == 0 && o < C_out)
            bpart[(long long)blockIdx.x * C_out + o] = ((red[0][tx] + red[1][tx]) + red[2][tx]) + red[3][tx];
        __syncthreads();
    }
}

// dbias: block (32, 32) per 32 columns; row lane ty adds partials ty,
// ty + 32, ... and the 32 lane sums are added in order.
__global__ void dbias_kernel(const float* __restrict__ bpart, int nblocks, int C_out,
                             float* __restrict__ dbias) {
    __shared__ float red[32][33];
    pdl_wait();
    pdl_trigger();
    const int o = blockIdx.x * 32 + threadIdx.x;
    float s = 0.f;
    if (o < C_out)
        for (int b = threadIdx.y; b < nblocks; b += 32) s += bpart[(long long)b * C_out + o];
    red[threadIdx.y][threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.y == 0 && o < C_out) {
        float t = 0.f;
#pragma unroll 8
        for (int i = 0; i < 32; ++i) t += red[i][threadIdx.x];
        dbias[o] = t;
    }
}

// W [K, C_out] -> W^T [C_out, K]
template <typename T>
__global__ void transpose_kernel(const T* __restrict__ W, int K, int C_out, T* __restrict__ Wt) {
    __shared__ T tile[32][33];
    pdl_wait();
    pdl_trigger();
    const int k0 = blockIdx.y * 32, o0 = blockIdx.x * 32;
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int k = k0 + i, o = o0 + threadIdx.x;
        if (k < K && o < C_out) tile[i][threadIdx.x] = W[(long long)k * C_out + o];
    }
    __syncthreads();
    for (int i = threadIdx.y; i < 32; i += blockDim.y) {
        const int o = o0 + i, k = k0 + threadIdx.x;
        if (k < K && o < C_out) Wt[(long long)o * K + k] = tile[threadIdx.x][i];
    }
}

// ---------------------------------------------------------------- transposed mapping
// taps of input row j: entries n*L + l with rulebook[l][n] == j, n < rows.
__global__ void rb_count_kernel(const int32_t* __restrict__ rb, const int32_t* count,
                                long long capacity, int L, int x_rows, int32_t* __restrict__ cnt,
                                unsigned* status) {
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    const long long total = rows * L;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        int n;
        const long long l = div32(e, (int)rows, n);  // rows <= capacity < 2^31
        const int j = __ldg(rb + l * capacity + n);
        if (j >= 0 && j < x_rows)
            atomicAdd(cnt + j, 1);
        else if (j < -1 || j >= x_rows)
            report(status, kErrIndex);
    }
}

// Exclusive scan of cnt[0..n) into ptr[0..n] (ptr[n] = total), in three
// passes over tiles of kScanTile: tile sums, a scan of the tile sums by one
// block, then each tile's scan plus its offset.
constexpr int kScanThreads = 1024;
constexpr int kScanTile = 4 * kScanThreads;

__device__ __forceinline__ int block_excl_scan(int v, int* sh, int& total) {
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += t;
    }
    if (lane == 31) sh[w] = x;
    __syncthreads();
    if (w == 0) {
        int s = lane < (int)(blockDim.x >> 5) ? sh[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += t;
        }
        sh[lane] = s;
    }
    __syncthreads();
    total = sh[(blockDim.x >> 5) - 1];
    const int before = w > 0 ? sh[w - 1] : 0;
    __syncthreads();
    return before + x - v;
}

__global__ void __launch_bounds__(kScanThreads)
    scan_tiles_kernel(const int32_t* __restrict__ cnt, int n, int32_t* __restrict__ tsum) {
    __shared__ int sh[32];
    pdl_wait();
    pdl_trigger();
    const long long base = (long long)blockIdx.x * kScanTile + threadIdx.x * 4;
    int v = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (base + i < n) v += cnt[base + i];
    int total;
    block_excl_scan(v, sh, total);
    if (threadIdx.x == 0) tsum[blockIdx.x] = total;
}

__global__ void __launch_bounds__(kScanThreads)
    scan_sums_kernel(int32_t* __restrict__ tsum, int ntiles) {
    __shared__ int sh[32];
    pdl_wait();
    pdl_trigger();
    int carry = 0;
    for (int b0 = 0; b0 < ntiles; b0 += kScanThreads) {
        const int i = b0 + threadIdx.x;
        const int v = i < ntiles ? tsum[i] : 0;
        int total;
        const int ex = block_excl_scan(v, sh, total);
        if (i < ntiles) tsum[i] = carry + ex;
        carry += total;
    }
}

__global__ void __launch_bounds__(kScanThreads)
    scan_apply_kernel(const int32_t* __restrict__ cnt, int n, const int32_t* __restrict__ toff,
                      int32_t* __restrict__ ptr, int32_t* __restrict__ fill) {
    __shared__ int sh[32];
    pdl_wait();
    pdl_trigger();
    const long long base = (long long)blockIdx.x * kScanTile + threadIdx.x * 4;
    int c[4], v = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        c[i] = base + i < n ? cnt[base + i] : 0;
        v += c[i];
    }
    int total;
    int run = toff[blockIdx.x] + block_excl_scan(v, sh, total);
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (base + i < n) {
            ptr[base + i] = run;
            fill[base + i] = 0;
            run += c[i];
        }
    if (base <= n - 1 && n - 1 < base + 4) ptr[n] = run;  // the total, by the holder of n - 1
}

__global__ void rb_fill_kernel(const int32_t* __restrict__ rb, const int32_t* count,
                               long long capacity, int L, int x_rows,
                               const int32_t* __restrict__ ptr, int32_t* __restrict__ fill,
                               int32_t* __restrict__ taps) {
    pdl_wait();
    pdl_trigger();
    long long rows = *count;
    rows = rows < 0 ? 0 : (rows > capacity ? capacity : rows);
    const long long total = rows * L;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        int n;
        const long long l = div32(e, (int)rows, n);  // rows <= capacity < 2^31
        const int j = __ldg(rb + l * capacity + n);
        if (j >= 0 && j < x_rows) {
            const int pos = atomicAdd(fill + j, 1);
            taps[ptr[j] + pos] = (int32_t)(n * L + l);
        }
    }
}

__device__ __forceinline__ void insertion_sort(int32_t* taps, int a, int b) {
    for (int i = a + 1; i < b; ++i) {
        const int key = taps[i];
        int k = i - 1;
        while (k >= a && taps[k] > key) {
            taps[k + 1] = taps[k];
            --k;
        }
        taps[k + 1] = key;
    }
}

// Within each row the fill order depends on timing: sort it. Warp w takes
// rows w, w + nwarps, ..., 32 at a time (row ranges in one load). A row of
// up to 32 keys (about L) is sorted by rank: lane i holds key i and counts
// the smaller keys by shuffles (keys are unique), then writes its key at
// that rank. Longer rows are insertion-sorted in place by one lane.
__global__ void rb_sort_kernel(const int32_t* __restrict__ ptr, int x_rows,
                               int32_t* __restrict__ taps) {
    pdl_wait();
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
    const long long w = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    for (long long q0 = 0; w + q0 * nwarps < x_rows; q0 += 32) {
        const long long jl = w + (q0 + lane) * nwarps;
        const bool have = jl < x_rows;
        const int pa = have ? ptr[jl] : 0, pb = have ? ptr[jl + 1] : 0;
        for (unsigned todo = __ballot_sync(0xffffffffu, have && pb - pa > 1); todo;
             todo &= todo - 1) {
            const int r = __ffs(todo) - 1;
            const int a = __shfl_sync(0xffffffffu, pa, r), b = __shfl_sync(0xffffffffu, pb, r);
            const int len = b - a;
            if (len <= 32) {
                const int key = lane < len ? taps[a + lane] : 0x7fffffff;
                int rank = 0;
#pragma unroll
                for (int k = 0; k < 32; ++k) rank += __shfl_sync(0xffffffffu, key, k) < key;
                if (lane < len) taps[a + rank] = key;
            } else if (lane == 0) {
                insertion_sort(taps, a, b);
            }
            __syncwarp();
        }
    }
}

// ---------------------------------------------------------------- dgrad gather-sum
// dx[j][c] = sum over the taps e of row j (ascending n*L + l) of
// P[n][l*C_in + c]; U-sized chunks of VEC elements; rows without taps get 0.
// Keys are checked against the P rows that exist (n < capacity) and the
// row ranges against the taps table (a malformed table is reported and its
// entries skipped).
template <typename T, typename U>
__global__ void dgrad_kernel(const T* __restrict__ P, const int32_t* __restrict__ ptr,
                             const int32_t* __restrict__ taps, int x_rows, int L, int C_in,
                             long long capacity, T* __restrict__ dx, unsigned* status) {
    constexpr int VEC = sizeof(U) / sizeof(T);
    pdl_wait();
    pdl_trigger();
    const int cpr = C_in / VEC;
    const long long total = (long long)x_rows * cpr;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        int ci;
        const long long j = div32(i, cpr, ci);
        const int c = ci * VEC;
        float acc[VEC];
#pragma unroll
        for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
        int a = __ldg(ptr + j), b = __ldg(ptr + j + 1);
        if (a < 0 || b < a || (long long)b > capacity * L) {
            if (c == 0) report(status, kErrIndex);
            b = a;
        }
        // a batch of keys, then all their P chunks in flight, then the sums
        // (in key order)
        constexpr int kBatchTaps = 4;
        for (int e0 = a; e0 < b; e0 += kBatchTaps) {
            int key[kBatchTaps];
#pragma unroll
            for (int i = 0; i < kBatchTaps; ++i) key[i] = e0 + i < b ? __ldg(taps + e0 + i) : -1;
            U raw[kBatchTaps];
#pragma unroll
            for (int i = 0; i < kBatchTaps; ++i) {
                if (e0 + i >= b) continue;
                if (key[i] < 0 || (long long)key[i] >= capacity * L) {
                    if (c == 0) report(status, kErrIndex);
                    key[i] = -1;
                    continue;
                }
                // key n*L + l: P's row n, slot l starts at (n*L + l)*C_in
                raw[i] = *reinterpret_cast<const U*>(P + (long long)key[i] * C_in + c);
            }
#pragma unroll
            for (int i = 0; i < kBatchTaps; ++i) {
                if (e0 + i >= b || key[i] < 0) continue;
                const T* v = reinterpret_cast<const T*>(&raw[i]);
#pragma unroll
                for (int k = 0; k < VEC; ++k) acc[k] += to_f(v[k]);
            }
        }
        U out;
        T* ov = reinterpret_cast<T*>(&out);
#pragma unroll
        for (int k = 0; k < VEC; ++k) ov[k] = from_f<T>(acc[k]);
        *reinterpret_cast<U*>(dx + j * C_in + c) = out;
    }
}

// ---------------------------------------------------------------- wgrad
constexpr int kTile = 128;
constexpr int kBK = 64;
constexpr int kStages = 6;
constexpr int kOpBytes = kBK * kTile * 2;
constexpr int kProducerWarps = 4, kEpilogueWarps = 4;
constexpr int kMmaWarp = kProducerWarps + kEpilogueWarps;
constexpr int kThreadsTc = (kMmaWarp + 1) * 32;
constexpr int kPartElems = kTile * kTile;
constexpr size_t kSmemTc = 1024 + (size_t)kStages * 2 * kOpBytes + 256;
// kind::f16: D fp32, A and B bf16, both MN-major, N = 128, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) |
                            ((uint32_t)(kTile >> 3) << 17) | ((uint32_t)(kTile >> 4) << 24);

struct WgradArgs {
    const void* x;
    const int32_t* rb;
    const int32_t* count;
    const void* dz;
    long long capacity;
    int x_rows, L, C_in, C_out, K;  // K = L * C_in
    int m_tiles, n_tiles, T, splits;  // rows split on the device, from *count
    float* part;                      // [splits * T][128][128]
    unsigned* status;
};

__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(lbo >> 4) << 16) |
           ((uint64_t)(sbo >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// Warps 0-3 load a stage: thread t owns 16-byte chunk column t % 16 of the
// tile's 128 columns (of the gathered rows for A, of dz for B) and rows
// t / 16 + 8 i; the rulebook entries of the next stage are loaded while the
// current stage's copies go out. Warp 8 issues the MMAs, warps 4-7 write
// the finished tile to the workspace.
__global__ void __launch_bounds__(kThreadsTc, 1) wgrad_tc_kernel(const WgradArgs a) {
    constexpr uint32_t kArrivals = kProducerWarps * 32;
    constexpr int kRowsPer = kBK / 8;  // rows of a stage per producer thread
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const base_ptr = smem_raw + (base - raw);
    const uint32_t sA = base, sB = base + kStages * kOpBytes;
    const uint32_t sBar = sB + kStages * kOpBytes;
    auto full_bar = [&](int s) { return sBar + 8u * s; };
    auto empty_bar = [&](int s) { return sBar + 8u * (kStages + s); };
    const uint32_t tfull_bar = sBar + 8u * (2 * kStages);
    const uint32_t fin_bar = sBar + 8u * (2 * kStages + 1);
    uint8_t* const misc = base_ptr + (sBar - base) + 8 * (2 * kStages + 2);
    volatile uint32_t* const tmem_holder = reinterpret_cast<volatile uint32_t*>(misc);
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(misc + 4);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(full_bar(s), kArrivals);
            mbar_init(empty_bar(s), 1);
        }
        mbar_init(tfull_bar, 1);
        mbar_init(fin_bar, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32((const void*)tmem_holder), kTile);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;
    pdl_wait();
    pdl_trigger();

    long long rows = *a.count;
    rows = rows < 0 ? 0 : (rows > a.capacity ? a.capacity : rows);
    const int item = blockIdx.x;
    const int split = item / a.T;
    const int tile = item - split * a.T;
    const int tm = tile / a.n_tiles, tn = tile - tm * a.n_tiles;
    // the active rows (known on the device) split evenly, in kBK blocks
    const long long rps = ((rows + a.splits - 1) / a.splits + kBK - 1) / kBK * kBK;
    const long long r_begin = (long long)split * rps;
    long long r_end = r_begin + rps;
    if (r_end > rows) r_end = rows;
    const int num_kb = r_end > r_begin ? (int)((r_end - r_begin + kBK - 1) / kBK) : 0;

    if (warp < kProducerWarps) {
        const __nv_bfloat16* __restrict__ x = static_cast<const __nv_bfloat16*>(a.x);
        const __nv_bfloat16* __restrict__ dz = static_cast<const __nv_bfloat16*>(a.dz);
        const int t = threadIdx.x;
        const int cc = t & 15, atom = cc >> 3, q = cc & 7;
        const int m = tm * kTile + cc * 8;  // A column: tap slot l, channel c
        const bool m_ok = m < a.K;
        const int l = m_ok ? m / a.C_in : 0, c = m - l * a.C_in;
        const int32_t* rbl = a.rb + (long long)l * a.capacity;
        const int o = tn * kTile + cc * 8;  // B column: output channel
        const bool o_ok = o < a.C_out;
        unsigned err = 0;
        int jn[kRowsPer];
        auto load_taps = [&](int kb, int (&j)[kRowsPer]) {
#pragma unroll
            for (int i = 0; i < kRowsPer; ++i) {
                const long long n = r_begin + (long long)kb * kBK + (t >> 4) + 8 * i;
                j[i] = (m_ok && n < r_end) ? __ldg(rbl + n) : -1;
            }
        };
        if (num_kb > 0) load_taps(0, jn);
        for (int kb = 0; kb < num_kb; ++kb) {
            int j[kRowsPer];
#pragma unroll
            for (int i = 0; i < kRowsPer; ++i) j[i] = jn[i];
            if (kb + 1 < num_kb) load_taps(kb + 1, jn);
            const int s = kb % kStages;
            const uint32_t ph = (uint32_t)((kb / kStages) & 1);
            if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, a.status)) break;
            const long long n0 = r_begin + (long long)kb * kBK;
            const uint32_t a_st = sA + s * kOpBytes + atom * (kBK * 128);
            const uint32_t b_st = sB + s * kOpBytes + atom * (kBK * 128);
#pragma unroll
            for (int i = 0; i < kRowsPer; ++i) {
                const int r = (t >> 4) + 8 * i;
                const long long n = n0 + r;
                const int ji = j[i];
                if (ji < -1 || ji >= a.x_rows) err |= kErrIndex;
                const bool av = ji >= 0 && ji < a.x_rows;
                cp_async_16(a_st + r * 128 + ((q ^ (r & 7)) << 4),
                            x + (av ? (long long)ji * a.C_in + c : 0), av);
                const bool bv = o_ok && n < r_end;
                cp_async_16(b_st + r * 128 + ((q ^ (r & 7)) << 4),
                            dz + (bv ? n * a.C_out + o : 0), bv);
            }
            cp_async_arrive_noinc(full_bar(s));
        }
        cp_async_wait_all();
        if (err) report(a.status, err);
    } else if (warp == kMmaWarp) {
        if (lane == 0) {
            bool ok = true;
            for (int kb = 0; kb < num_kb; ++kb) {
                const int s = kb % kStages;
                const uint32_t ph = (uint32_t)((kb / kStages) & 1);
                if (!mbar_wait(full_bar(s), ph, abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                fence_proxy_async_smem();  // operands written by cp.async
                const uint32_t a_st = sA + s * kOpBytes, b_st = sB + s * kOpBytes;
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k) {
                    const uint64_t ad = desc_sw128(a_st + k * 16 * 128, kBK * 128, 1024);
                    const uint64_t bd = desc_sw128(b_st + k * 16 * 128, kBK * 128, 1024);
                    tc_mma_bf16(tmem_base, ad, bd, kIdesc, (kb | k) != 0 ? 1u : 0u);
                }
                tc_commit(empty_bar(s));
            }
            if (ok && num_kb > 0) tc_commit(tfull_bar);
            tc_commit(fin_bar);
            int no_abort = 0;
            mbar_wait(fin_bar, 0, &no_abort, a.status);
            if (ok && num_kb == 0) mbar_arrive(tfull_bar);  // empty split: zeros
        }
        __syncwarp();
    } else {
        const int ew = warp - kProducerWarps;
        const int row = ew * 32 + lane;
        float* dst = a.part + (long long)item * kPartElems + (long long)row * kTile;
        if (mbar_wait(tfull_bar, 0, abort_flag, a.status)) {
            tc_fence_after();
#pragma unroll 1
            for (int cb = 0; cb < kTile / 32; ++cb) {
                uint32_t r[32];
                if (num_kb > 0) {
                    tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(ew * 32) << 16) + (uint32_t)(cb * 32),
                                       r);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int jj = 0; jj < 32; ++jj) r[jj] = 0u;
                }
                float4* d4 = reinterpret_cast<float4*>(dst + cb * 32);
#pragma unroll
                for (int jj = 0; jj < 8; ++jj)
                    d4[jj] = make_float4(__uint_as_float(r[4 * jj]), __uint_as_float(r[4 * jj + 1]),
                                         __uint_as_float(r[4 * jj + 2]),
                                         __uint_as_float(r[4 * jj + 3]));
            }
            tc_fence_before();
        }
    }
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, kTile);
    }
}

// fp32 (or unaligned bf16) on CUDA cores: 256 threads, 8 x 8 outputs each.
template <typename T>
__global__ void __launch_bounds__(256) wgrad_simt_kernel(const WgradArgs a) {
    constexpr int kBKs = 16;
    __shared__ float As[kBKs][kTile];
    __shared__ float Bs[kBKs][kTile];
    pdl_wait();
    pdl_trigger();
    const T* __restrict__ x = static_cast<const T*>(a.x);
    const T* __restrict__ dz = static_cast<const T*>(a.dz);
    long long rows = *a.count;
    rows = rows < 0 ? 0 : (rows > a.capacity ? a.capacity : rows);
    const int item = blockIdx.x;
    const int split = item / a.T;
    const int tile = item - split * a.T;
    const int tm = tile / a.n_tiles, tn = tile - tm * a.n_tiles;
    const long long rps = ((rows + a.splits - 1) / a.splits + kBKs - 1) / kBKs * kBKs;
    const long long r_begin = (long long)split * rps;
    long long r_end = r_begin + rps;
    if (r_end > rows) r_end = rows;
    const int t = threadIdx.x, ty = t >> 4, tx = t & 15;
    const int mm = t & (kTile - 1);
    const int m = tm * kTile + mm;
    const bool m_ok = m < a.K;
    const int l = m_ok ? m / a.C_in : 0, c = m - l * a.C_in;
    const int o = tn * kTile + mm;
    const bool o_ok = o < a.C_out;
    unsigned err = 0;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) acc[i][jj] = 0.f;
    for (long long n0 = r_begin; n0 < r_end; n0 += kBKs) {
#pragma unroll
        for (int i = 0; i < kBKs / 2; ++i) {
            const int r = (t >> 7) + 2 * i;
            const long long n = n0 + r;
            float av = 0.f, bv = 0.f;
            if (n < r_end) {
                if (m_ok) {
                    const int j = __ldg(a.rb + (long long)l * a.capacity + n);
                    if (j >= 0 && j < a.x_rows)
                        av = to_f(x[(long long)j * a.C_in + c]);
                    else if (j != -1)
                        err |= kErrIndex;
                }
                if (o_ok) bv = to_f(dz[n * a.C_out + o]);
            }
            As[r][mm] = av;
            Bs[r][mm] = bv;
        }
        __syncthreads();
#pragma unroll 4
        for (int k = 0; k < kBKs; ++k) {
            float avv[8], bvv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) avv[i] = As[k][ty * 8 + i];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) bvv[jj] = Bs[k][tx * 8 + jj];
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) acc[i][jj] = fmaf(avv[i], bvv[jj], acc[i][jj]);
        }
        __syncthreads();
    }
    if (err) report(a.status, err);
    float* dst = a.part + (long long)item * kPartElems;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float4* d4 = reinterpret_cast<float4*>(dst + (ty * 8 + i) * kTile + tx * 8);
        d4[0] = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        d4[1] = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
    }
}

// dW[m][o] = sum over splits (in order) of the partial tiles.
__global__ void wgrad_reduce_kernel(const float* __restrict__ part, int K, int C_out, int n_tiles,
                                    int T, int splits, float* __restrict__ dW) {
    pdl_wait();
    pdl_trigger();
    const long long total = (long long)K * C_out;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        int o;
        const int m = (int)div32(e, C_out, o);
        const int t = (m >> 7) * n_tiles + (o >> 7);
        const float* src = part + (long long)t * kPartElems + ((m & 127) << 7) + (o & 127);
        float s = 0.f;
        for (int sp = 0; sp < splits; ++sp) s += src[(long long)sp * T * kPartElems];
        dW[e] = s;
    }
}

// Rows whose 16-byte chunk count cpr divides 32: warp w takes rows w,
// w + nwarps, ..., 32 at a time. Their row ranges come in one load (lane r
// holds row r's); a ballot splits them into rows without taps, written as
// zeros G rows per store, and rows with taps, for which lane
// (g, c) = (lane / cpr, lane % cpr) sums chunk c of taps g, g + G, ...
// (G = 32 / cpr groups, keys then P chunks loaded four at a time) and the
// groups are added by a fixed shuffle tree.
template <typename T>
__global__ void __launch_bounds__(256)
    dgrad_warp_kernel(const T* __restrict__ P, const int32_t* __restrict__ ptr,
                      const int32_t* __restrict__ taps, int x_rows, int L, int C_in,
                      long long capacity, T* __restrict__ dx, unsigned* status) {
    constexpr int VEC = 16 / sizeof(T);
    pdl_wait();
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int cpr = C_in / VEC, G = 32 / cpr;
    const int g = lane / cpr, c = (lane - g * cpr) * VEC;
    const long long nwarps = (long long)gridDim.x * (blockDim.x >> 5);
    const long long w = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    // rows w, w + nwarps, w + 2 nwarps, ...: clustered active rows spread
    // over all warps instead of loading a few
    for (long long q0 = 0; w + q0 * nwarps < x_rows; q0 += 32) {
        const long long jl = w + (q0 + lane) * nwarps;
        const bool have = jl < x_rows;
        const int pa = have ? __ldg(ptr + jl) : 0;
        const int pb = have ? __ldg(ptr + jl + 1) : 0;
        const long long left = (x_rows - 1 - w) / nwarps + 1 - q0;  // rows left for this warp
        const int nr = left < 32 ? (int)left : 32;
        // rows without taps: zeros, G rows per store instruction
        const unsigned busy = __ballot_sync(0xffffffffu, have && pb != pa);
        for (int r0 = 0; r0 < nr; r0 += G) {
            const int r = r0 + g;
            if (r < nr && !((busy >> r) & 1u))
                *reinterpret_cast<uint4*>(dx + (w + (q0 + r) * nwarps) * C_in + c) =
                    make_uint4(0u, 0u, 0u, 0u);
        }
        // rows with taps
        for (unsigned todo = busy; todo; todo &= todo - 1) {
            const int r = __ffs(todo) - 1;
            const long long j = w + (q0 + r) * nwarps;
            int a = __shfl_sync(0xffffffffu, pa, r), b = __shfl_sync(0xffffffffu, pb, r);
            if (a < 0 || b < a || (long long)b > capacity * L) {
                if (lane == 0) report(status, kErrIndex);
                b = a;
            }
            float acc[VEC];
#pragma unroll
            for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
            for (int e0 = a + g; e0 < b; e0 += 4 * G) {
                int key[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = e0 + i * G;
                    key[i] = e < b ? __ldg(taps + e) : -1;
                    if (e < b && (key[i] < 0 || (long long)key[i] >= capacity * L)) {
                        report(status, kErrIndex);
                        key[i] = -1;
                    }
                }
                uint4 raw[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    if (key[i] < 0) continue;
                    // key n*L + l: P's row n, slot l starts at (n*L + l)*C_in
                    raw[i] = *reinterpret_cast<const uint4*>(P + (long long)key[i] * C_in + c);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    if (key[i] < 0) continue;
                    const T* v = reinterpret_cast<const T*>(&raw[i]);
#pragma unroll
                    for (int k = 0; k < VEC; ++k) acc[k] += to_f(v[k]);
                }
            }
            for (int o = cpr; o < 32; o <<= 1)
#pragma unroll
                for (int k = 0; k < VEC; ++k) acc[k] += __shfl_xor_sync(0xffffffffu, acc[k], o);
            if (g == 0) {
                uint4 out;
                T* ov = reinterpret_cast<T*>(&out);
#pragma unroll
                for (int k = 0; k < VEC; ++k) ov[k] = from_f<T>(acc[k]);
                *reinterpret_cast<uint4*>(dx + j * C_in + c) = out;
            }
        }
    }
}

template <typename T>
hc_status launch_dgrad_typed(const DeviceCtx* ctx, const void* P, const int32_t* ptr,
                             const int32_t* taps, int x_rows, int L, int C_in, long long capacity,
                             void* dx, cudaStream_t s) {
    const uintptr_t al = (uintptr_t)P | (uintptr_t)dx;
    const int vec16 = 16 / (int)sizeof(T);
    const bool wide = C_in % vec16 == 0 && al % 16 == 0;
    const int vec = wide ? vec16 : 1;
    const int cpr = C_in / vec16;
    if (wide && cpr <= 32 && (32 % cpr) == 0) {
        long long wblocks = ((long long)x_rows + 255) / 256;  // 8 warps x 32 rows per block
        if (wblocks > (long long)ctx->num_sms * 8) wblocks = (long long)ctx->num_sms * 8;
        if (wblocks < 1) wblocks = 1;
        return launch_pdl(dgrad_warp_kernel<T>, dim3((unsigned)wblocks), dim3(256), 0, s,
                          "dgrad_warp_kernel", (const T*)P, ptr, taps, x_rows, L, C_in, capacity,
                          (T*)dx, ctx->status);
    }
    long long blocks = ((long long)x_rows * (C_in / vec) + 255) / 256;
    const long long cap = (long long)ctx->num_sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (wide)
        return launch_pdl(dgrad_kernel<T, uint4>, dim3((unsigned)blocks), dim3(256), 0, s,
                          "dgrad_kernel", (const T*)P, ptr, taps, x_rows, L, C_in, capacity, (T*)dx,
                          ctx->status);
    return launch_pdl(dgrad_kernel<T, T>, dim3((unsigned)blocks), dim3(256), 0, s, "dgrad_kernel",
                      (const T*)P, ptr, taps, x_rows, L, C_in, capacity, (T*)dx, ctx->status);
}

}  // namespace

hc_status launch_rulebook_transpose(const DeviceCtx* ctx, const int32_t* rb, const int32_t* count,
                                    int capacity, int L, int x_rows, int32_t* ptr, int32_t* taps,
                                    cudaStream_t s) {
    const int ntiles = (x_rows + kScanTile - 1) / kScanTile;
    // workspace: per-row counts, fill cursors, tile sums
    int32_t* ws = (int32_t*)stream_workspace(s, sizeof(int32_t) * (2 * (size_t)x_rows + ntiles + 1));
    if (!ws) return HC_ERR_CUDA;
    int32_t* cnt = ws;
    int32_t* fill = ws + x_rows;
    int32_t* tsum = ws + 2 * (size_t)x_rows;
    hc_status st = check_cuda(cudaMemsetAsync(cnt, 0, sizeof(int32_t) * (size_t)x_rows, s),
                              "cudaMemsetAsync(counts)");
    if (st != HC_OK) return st;
    long long blocks = ((long long)capacity * L + 255) / 256;
    const long long cap = (long long)ctx->num_sms * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    st = launch_pdl(rb_count_kernel, dim3((unsigned)blocks), dim3(256), 0, s, "rb_count_kernel", rb,
                    count, (long long)capacity, L, x_rows, cnt, ctx->status);
    if (st != HC_OK) return st;
    st = launch_pdl(scan_tiles_kernel, dim3((unsigned)ntiles), dim3(kScanThreads), 0, s,
                    "scan_tiles_kernel", (const int32_t*)cnt, x_rows, tsum);
    if (st != HC_OK) return st;
    st = launch_pdl(scan_sums_kernel, dim3(1), dim3(kScanThreads), 0, s, "scan_sums_kernel", tsum,
                    ntiles);
    if (st != HC_OK) return st;
    st = launch_pdl(scan_apply_kernel, dim3((unsigned)ntiles), dim3(kScanThreads), 0, s,
                    "scan_apply_kernel", (const int32_t*)cnt, x_rows, (const int32_t*)tsum, ptr,
                    fill);
    if (st != HC_OK) return st;
    st = launch_pdl(rb_fill_kernel, dim3((unsigned)blocks), dim3(256), 0, s, "rb_fill_kernel", rb,
                    count, (long long)capacity, L, x_rows, (const int32_t*)ptr, fill, taps);
    if (st != HC_OK) return st;
    long long sblocks = ((long long)x_rows + 255) / 256;
    if (sblocks > cap) sblocks = cap;
    return launch_pdl(rb_sort_kernel, dim3((unsigned)sblocks), dim3(256), 0, s, "rb_sort_kernel",
                      (const int32_t*)ptr, x_rows, taps);
}

hc_status launch_conv_bwd(const DeviceCtx* ctx, const BwdArgs& b, cudaStream_t s) {
    const bool bf = b.dt == HC_BF16;
    const int eb = bf ? 2 : 4;
    const int K = b.L * b.C_in;
    // Work split of wgrad: 128 x 128 tiles of dW, rows split to fill the SMs.
    const int m_tiles = (K + kTile - 1) / kTile, n_tiles = (b.C_out + kTile - 1) / kTile;
    const int T = m_tiles * n_tiles;
    int splits = 1;
    {
        long long max_splits = ((long long)b.capacity + kBK - 1) / kBK;
        const long long cap_splits = 8ll * ctx->num_sms / T + 1;
        if (max_splits > cap_splits) max_splits = cap_splits;
        if (max_splits < 1) max_splits = 1;
        double best = 0.0;
        for (int sp = 1; sp <= max_splits; ++sp) {
            const long long items = (long long)sp * T;
            const long long waves = (items + ctx->num_sms - 1) / ctx->num_sms;
            const double eff = (double)items / (double)(waves * ctx->num_sms);
            if (eff > best + 1e-9) {
                best = eff;
                splits = sp;
            }
            if (eff >= 0.95) break;
        }
    }
    const long long items = (long long)splits * T;
    long long act_blocks_ll = ((long long)b.capacity + kActRowsPerBlock - 1) / kActRowsPerBlock;
    if (act_blocks_ll > 8ll * ctx->num_sms) act_blocks_ll = 8ll * ctx->num_sms;
    const int act_blocks = (int)(act_blocks_ll > 0 ? act_blocks_ll : 1);

    // workspace: dz | P | W^T | wgrad partials | dbias partials
    auto up = [](size_t v) { return (v + 255) / 256 * 256; };
    const size_t dz_bytes = up((size_t)b.capacity * b.C_out * eb);
    const size_t p_bytes = b.dx ? up((size_t)b.capacity * K * eb) : 0;
    const size_t wt_bytes = b.dx ? up((size_t)K * b.C_out * eb) : 0;
    const size_t part_bytes = b.dW ? up(sizeof(float) * (size_t)items * kPartElems) : 0;
    const size_t bp_bytes = up(sizeof(float) * (size_t)(act_blocks > 0 ? act_blocks : 1) * b.C_out);
    uint8_t* ws = (uint8_t*)stream_workspace(s, dz_bytes + p_bytes + wt_bytes + part_bytes + bp_bytes);
    if (!ws) return HC_ERR_CUDA;
    void* dz = ws;
    void* P = ws + dz_bytes;
    void* Wt = ws + dz_bytes + p_bytes;
    float* part = (float*)(ws + dz_bytes + p_bytes + wt_bytes);
    float* bpart = (float*)(ws + dz_bytes + p_bytes + wt_bytes + part_bytes);

    hc_status st;
    if (bf)
        st = launch_pdl(act_bwd_kernel<__nv_bfloat16>, dim3((unsigned)act_blocks), dim3(256), 0, s,
                        "act_bwd_kernel", (const __nv_bfloat16*)b.y, (const __nv_bfloat16*)b.dy,
                        b.count, (long long)b.capacity, b.C_out, b.act, (__nv_bfloat16*)dz, bpart,
                        ctx->status);
    else
        st = launch_pdl(act_bwd_kernel<float>, dim3((unsigned)act_blocks), dim3(256), 0, s,
                        "act_bwd_kernel", (const float*)b.y, (const float*)b.dy, b.count,
                        (long long)b.capacity, b.C_out, b.act, (float*)dz, bpart, ctx->status);
    if (st != HC_OK) return st;
    if (b.dbias) {
        st = launch_pdl(dbias_kernel, dim3((unsigned)((b.C_out + 31) / 32)), dim3(32, 32), 0, s,
                        "dbias_kernel", (const float*)bpart, act_blocks, b.C_out, b.dbias);
        if (st != HC_OK) return st;
    }

    if (b.dW) {
        WgradArgs w{};
        w.x = b.x;
        w.rb = b.rulebook;
        w.count = b.count;
        w.dz = dz;
        w.capacity = b.capacity;
        w.x_rows = b.x_rows;
        w.L = b.L;
        w.C_in = b.C_in;
        w.C_out = b.C_out;
        w.K = K;
        w.m_tiles = m_tiles;
        w.n_tiles = n_tiles;
        w.T = T;
        w.splits = splits;
        w.part = part;
        w.status = ctx->status;
        const bool tc = bf && b.C_in % 8 == 0 && b.C_out % 8 == 0 && (uintptr_t)b.x % 16 == 0;
        if (tc) {
            static bool attr_set[64] = {};
            if (!attr_set[ctx->device]) {
                st = check_cuda(cudaFuncSetAttribute(wgrad_tc_kernel,
                                                     cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                     (int)kSmemTc),
                                "cudaFuncSetAttribute(wgrad_tc_kernel)");
                if (st != HC_OK) return st;
                attr_set[ctx->device] = true;
            }
            st = launch_pdl(wgrad_tc_kernel, dim3((unsigned)items), dim3(kThreadsTc), kSmemTc, s,
                            "wgrad_tc_kernel", w);
        } else if (bf) {
            st = launch_pdl(wgrad_simt_kernel<__nv_bfloat16>, dim3((unsigned)items), dim3(256), 0, s,
                            "wgrad_simt_kernel", w);
        } else {
            st = launch_pdl(wgrad_simt_kernel<float>, dim3((unsigned)items), dim3(256), 0, s,
                            "wgrad_simt_kernel", w);
        }
        if (st != HC_OK) return st;
        long long rblocks = ((long long)K * b.C_out + 255) / 256;
        if (rblocks > (long long)ctx->num_sms * 8) rblocks = (long long)ctx->num_sms * 8;
        st = launch_pdl(wgrad_reduce_kernel, dim3((unsigned)rblocks), dim3(256), 0, s,
                        "wgrad_reduce_kernel", (const float*)part, K, b.C_out, n_tiles, T, splits,
                        b.dW);
        if (st != HC_OK) return st;
    }

    if (b.dx) {
        // W^T, then P = dz W^T through the linear conv path, then the gather-sum.
        const dim3 tg((unsigned)((b.C_out + 31) / 32), (unsigned)((K + 31) / 32)), tb(32, 8);
        st = bf ? launch_pdl(transpose_kernel<__nv_bfloat16>, tg, tb, 0, s, "transpose_kernel",
                             (const __nv_bfloat16*)b.W, K, b.C_out, (__nv_bfloat16*)Wt)
                : launch_pdl(transpose_kernel<float>, tg, tb, 0, s, "transpose_kernel",
                             (const float*)b.W, K, b.C_out, (float*)Wt);
        if (st != HC_OK) return st;
        ConvArgs c{};
        c.x = dz;
        c.count = b.count;
        c.W = Wt;
        c.bias = nullptr;
        c.y = P;
        c.capacity = b.capacity;
        c.x_rows = b.capacity;
        c.B = 1;
        c.V = b.capacity;
        c.L = 1;
        c.C_in = b.C_out;
        c.C_out = K;
        c.K = b.C_out;
        c.mode = kLinear;
        c.act = HC_ACT_NONE;
        st = dispatch_conv(ctx, c, b.dt, s);
        if (st != HC_OK) return st;
        st = bf ? launch_dgrad_typed<__nv_bfloat16>(ctx, P, b.row_ptr, b.taps, b.x_rows, b.L, b.C_in,
                                                    b.capacity, b.dx, s)
                : launch_dgrad_typed<float>(ctx, P, b.row_ptr, b.taps, b.x_rows, b.L, b.C_in,
                                            b.capacity, b.dx, s);
        if (st != HC_OK) return st;
    }
    return HC_OK;
}

}  // namespace hc
