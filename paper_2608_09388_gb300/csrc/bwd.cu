// Backward of the sparse spiral convolution (the chain rule on Eqs. 4-5, 6
// and 10; the paper gives the forward only). Through the Eq. 4 mapping
// rulebook[l][n] = input row j read by tap l of output row n (or -1):
//   dz[n][o]  = dy[n][o] * act'(y[n][o])           act' read off the output
//   dbias[o]  = sum_n dz[n][o]
//   dW[l*C_in + c][o] = sum_n x[j(n,l)][c] * dz[n][o]
//   dx[j][c]  = sum over taps (n, l) reading j of (dz[n] W_l^T)[c]
// Kernels (every sum in a fixed order, no floating-point atomics):
//   act_bwd_kernel      dz (stored in the layer dtype) and per-block column
//                       sums of dz in fp32 (act_bwd_vec_kernel: 16-byte
//                       chunks); dbias_kernel adds the blocks.
//   wgrad (tcgen05)     split-K [L*C_in] x [C_out] tiles: A = the gathered
//                       input rows (cp.async through the rulebook), B = dz,
//                       both MN-major, fp32 accumulators in TMEM; fp32 on
//                       CUDA cores otherwise. wgrad_reduce adds the splits.
//   dgrad               P = dz W^T by the linear conv kernels (W^T
//                       materialised once), then every input row sums the P
//                       slices of the taps that read it, in (n, l) order,
//                       from the transposed mapping (rb_* kernels: counts,
//                       exclusive scan, fill, per-row sort): a block per
//                       range of rows, their keys staged in shared memory,
//                       where rows are whole 16-byte chunks.
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

// Vectorised dz for rows of 16-byte chunks (cpr = C_out / VEC of them,
// cpr dividing 256): a block takes kActVecItems / cpr consecutive rows
// (ranges blockIdx.x, + gridDim.x, ...); thread t always holds chunk
// t % cpr, so it sums its VEC columns over its rows in registers, and the
// 256 / cpr row lanes of a column meet in shared memory in a fixed order.
constexpr int kActVecItems = 1024;

template <typename T>
__global__ void __launch_bounds__(256)
    act_bwd_vec_kernel(const T* __restrict__ y, const T* __restrict__ dy, const int32_t* count,
                       long long capacity, int C_out, int act, T* __restrict__ dz,
                       float* __restrict__ bpart, unsigned* status) {
    constexpr int VEC = 16 / sizeof(T);
    constexpr int kPer = kActVecItems / 256;
    __shared__ float red[256 * VEC];
    pdl_wait();
    pdl_trigger();
    const long long rows = clamp_rows(count, capacity, status);
    const int t = threadIdx.x;
    const int cpr = C_out / VEC, lanes = 256 / cpr;
    const int c = t % cpr, rl = t / cpr;
    const int R = kActVecItems / cpr;
    float sum[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) sum[k] = 0.f;
    for (long long r0 = (long long)blockIdx.x * R; r0 < rows; r0 += (long long)gridDim.x * R) {
        uint4 yv[kPer], gv[kPer];
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const long long r = r0 + rl + (long long)q * lanes;
            if (r < rows) {
                yv[q] = *reinterpret_cast<const uint4*>(y + r * C_out + c * VEC);
                gv[q] = *reinterpret_cast<const uint4*>(dy + r * C_out + c * VEC);
            }
        }
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const long long r = r0 + rl + (long long)q * lanes;
            if (r >= rows) continue;
            const T* yp = reinterpret_cast<const T*>(&yv[q]);
            const T* gp = reinterpret_cast<const T*>(&gv[q]);
            uint4 out;
            T* op = reinterpret_cast<T*>(&out);
#pragma unroll
            for (int k = 0; k < VEC; ++k) {
                const float yk = to_f(yp[k]);
                float d = 1.f;
                if (act == HC_ACT_ELU) d = yk > 0.f ? 1.f : yk + 1.f;
                else if (act == HC_ACT_RELU) d = yk > 0.f ? 1.f : 0.f;
                const float v = to_f(gp[k]) * d;
                op[k] = from_f<T>(v);
                sum[k] += v;
            }
            *reinterpret_cast<uint4*>(dz + r * C_out + c * VEC) = out;
        }
    }
#pragma unroll
    for (int k = 0; k < VEC; ++k) red[rl * C_out + c * VEC + k] = sum[k];
    __syncthreads();
    for (int o = t; o < C_out; o += 256) {
        float s = 0.f;
        for (int j = 0; j < lanes; ++j) s += red[j * C_out + o];
        bpart[(long long)blockIdx.x * C_out + o] = s;
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
#pragma unroll 4
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
            mbar_wait_drain(fin_bar, 0, a.status);
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

// Block-range gather-sum for rows of 16-byte chunks (cpr = C_in / VEC of
// them). A block takes R consecutive input rows r0 .. r0 + R - 1 (ranges
// blockIdx.x, + gridDim.x, ...). Their taps are one contiguous slice
// taps[ptr[r0] .. ptr[r0 + R]) of the transposed mapping, copied to shared
// memory in one coalesced pass (read from global memory instead when it does
// not fit or the table is malformed there). The block then writes zero
// chunks for the rows without taps and sums, for every (row with taps,
// chunk) item, the P chunks of the row's taps in ascending key order, eight
// loads in flight per thread. Every load of a round trip is issued by all
// threads at once: row ranges, keys, then P.
constexpr int kDgThreads = 256;
constexpr int kDgMaxRows = 1024;
constexpr int kDgKeys = 8192;

template <typename T>
__global__ void __launch_bounds__(kDgThreads, 4)
    dgrad_range_kernel(const T* __restrict__ P, const int32_t* __restrict__ ptr,
                       const int32_t* __restrict__ taps, int x_rows, int R, int C_in,
                       long long capL, T* __restrict__ dx, unsigned* status) {
    constexpr int VEC = 16 / sizeof(T);
    __shared__ int32_t s_ptr[kDgMaxRows + 1];
    __shared__ uint16_t s_busy[kDgMaxRows];
    __shared__ uint8_t s_on[kDgMaxRows];
    __shared__ int32_t s_keys[kDgKeys];
    __shared__ int s_nb;
    pdl_wait();
    pdl_trigger();
    const int t = threadIdx.x, lane = t & 31;
    const int cpr = C_in / VEC;
    for (long long r0 = (long long)blockIdx.x * R; r0 < x_rows; r0 += (long long)gridDim.x * R) {
        const int n = x_rows - r0 < R ? (int)(x_rows - r0) : R;
        for (int i = t; i <= n; i += kDgThreads) s_ptr[i] = __ldg(ptr + r0 + i);
        if (t == 0) s_nb = 0;
        __syncthreads();
        const int base = s_ptr[0], top = s_ptr[n];
        const bool in_smem = base >= 0 && top >= base && top - base <= kDgKeys && top <= capL;
        // the key slice, while the rows with taps are listed
        if (in_smem)
            for (int i = t; i < top - base; i += kDgThreads) s_keys[i] = __ldg(taps + base + i);
        for (int i0 = 0; i0 < n; i0 += kDgThreads) {
            const int i = i0 + t;
            bool on = false;
            if (i < n) {
                const int a = s_ptr[i], b = s_ptr[i + 1];
                const bool ok = a >= 0 && b >= a && b <= capL && (!in_smem || (a >= base && b <= top));
                if (!ok) report(status, kErrIndex);
                on = ok && b > a;
                s_on[i] = on ? 1 : 0;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, on);
            int wbase = 0;
            if (lane == 0 && bal) wbase = atomicAdd(&s_nb, __popc(bal));
            wbase = __shfl_sync(0xffffffffu, wbase, 0);
            if (on) s_busy[wbase + __popc(bal & ((1u << lane) - 1u))] = (uint16_t)i;
        }
        __syncthreads();
        // rows without taps: zeros, consecutive chunks per thread
        for (int f = t; f < n * cpr; f += kDgThreads) {
            int c;
            const int i = (int)div32(f, cpr, c);
            if (!s_on[i])
                *reinterpret_cast<uint4*>(dx + (r0 + i) * C_in + c * VEC) = make_uint4(0u, 0u, 0u, 0u);
        }
        // rows with taps
        const int nb = s_nb;
        const int32_t* kp = in_smem ? s_keys : taps;
        const int koff = in_smem ? base : 0;
        for (int f = t; f < nb * cpr; f += kDgThreads) {
            int c;
            const int bi = (int)div32(f, cpr, c);
            const int i = s_busy[bi];
            const int a = s_ptr[i] - koff, b = s_ptr[i + 1] - koff;
            float acc[VEC];
#pragma unroll
            for (int k = 0; k < VEC; ++k) acc[k] = 0.f;
            for (int e0 = a; e0 < b; e0 += 8) {
                uint4 raw[8];
                bool use[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const int key = e0 + q < b ? kp[e0 + q] : -1;
                    use[q] = key >= 0 && (long long)key < capL;
                    if (e0 + q < b && !use[q]) report(status, kErrIndex);
                    // key n*L + l: P's row n, slot l starts at (n*L + l)*C_in
                    if (use[q])
                        raw[q] = *reinterpret_cast<const uint4*>(P + (long long)key * C_in + c * VEC);
                }
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    if (!use[q]) continue;
                    const T* v = reinterpret_cast<const T*>(&raw[q]);
#pragma unroll
                    for (int k = 0; k < VEC; ++k) acc[k] += to_f(v[k]);
                }
            }
            uint4 out;
            T* ov = reinterpret_cast<T*>(&out);
#pragma unroll
            for (int k = 0; k < VEC; ++k) ov[k] = from_f<T>(acc[k]);
            *reinterpret_cast<uint4*>(dx + (r0 + i) * C_in + c * VEC) = out;
        }
        __syncthreads();  // the shared tables are reused by the next range
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
    if (wide && (long long)kDgMaxRows * (C_in / vec16) < (1ll << 31)) {
        // ranges of R rows, about one per resident block (4 per SM)
        const long long want = (long long)ctx->num_sms * 4;
        long long R = ((long long)x_rows + want - 1) / want;
        R = (R + 31) / 32 * 32;
        if (R < 256) R = 256;
        if (R > kDgMaxRows) R = kDgMaxRows;
        long long blocks = ((long long)x_rows + R - 1) / R;
        if (blocks > want) blocks = want;
        if (blocks < 1) blocks = 1;
        return launch_pdl(dgrad_range_kernel<T>, dim3((unsigned)blocks), dim3(kDgThreads), 0, s,
                          "dgrad_range_kernel", (const T*)P, ptr, taps, x_rows, (int)R, C_in,
                          capacity * L, (T*)dx, ctx->status);
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
    // dz: 16-byte chunks when a row is a whole number of them dividing 256
    const int act_vec = 16 / eb, act_cpr = b.C_out / act_vec;
    const bool act_wide = b.C_out % act_vec == 0 && 256 % act_cpr == 0 &&
                          ((uintptr_t)b.y | (uintptr_t)b.dy) % 16 == 0;
    const long long act_rows = act_wide ? kActVecItems / act_cpr : kActRowsPerBlock;
    long long act_blocks_ll = ((long long)b.capacity + act_rows - 1) / act_rows;
    const long long act_cap = (act_wide ? 4ll : 8ll) * ctx->num_sms;
    if (act_blocks_ll > act_cap) act_blocks_ll = act_cap;
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
    if (act_wide && bf)
        st = launch_pdl(act_bwd_vec_kernel<__nv_bfloat16>, dim3((unsigned)act_blocks), dim3(256), 0,
                        s, "act_bwd_vec_kernel", (const __nv_bfloat16*)b.y,
                        (const __nv_bfloat16*)b.dy, b.count, (long long)b.capacity, b.C_out, b.act,
                        (__nv_bfloat16*)dz, bpart, ctx->status);
    else if (act_wide)
        st = launch_pdl(act_bwd_vec_kernel<float>, dim3((unsigned)act_blocks), dim3(256), 0, s,
                        "act_bwd_vec_kernel", (const float*)b.y, (const float*)b.dy, b.count,
                        (long long)b.capacity, b.C_out, b.act, (float*)dz, bpart, ctx->status);
    else if (bf)
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
