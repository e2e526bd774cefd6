// Mask-score update (Eq. 3). With O_k the [N, D] output for mask k (masks
// stacked as [K, N, D]):
//   S[i][k]   = || O_i^T O_k ||_F^2
//   sim[i][k] = S[i][k] / sqrt(S[i][i] * S[k][k])   (0 where a norm is 0)
//   alpha'[k] = alpha[k] + 1/(K-1) * sum over i != k of (1 - sim[i][k])
//
// Every S entry is a block of one Gram matrix: with O_all = [N, K*D] (mask
// k's features in columns k*D .. k*D + D - 1), G = O_all^T O_all and S[i][k]
// is the sum of squares of G's (i, k) block. G is the only dense
// contraction here (2 * N * (K*D)^2 flops, symmetric, so only its
// upper-triangle tiles are computed), and a squared block norm needs the
// complete sum over N before squaring. So:
//   1. gram: split-K partial tiles of G, one work item per (row split,
//      upper tile), written to a workspace [item][tile][tile] fp32.
//      bf16: tcgen05 (both operands MN-major from shared memory, fp32
//      accumulators in TMEM); fp32: CUDA-core FFMA tiles.
//   2. pairs: blocks per pair i <= k and chunk of its D x D block sum the
//      splits of every entry (in a fixed order), square and reduce.
//   3. alpha: a thread per mask adds the chunks into S, forms sim and the
//      update (fp32; GB300's fp64 rate is far too low to be worth it here).
// Deterministic: no atomics, every sum in a fixed order.
//
// bf16 operands are read straight from [K, N, D] with cp.async: 16-byte
// pieces when D is a multiple of 8, 4-byte pieces when D is even (a piece
// never straddles two masks); odd D are first packed into a zero-padded
// [N, Mp] copy (Mp = K*D rounded up to the tile) in the workspace.
#include <cuda_bf16.h>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kBK = 64;  // rows of O per pipeline stage (the contraction dim)
// tcgen05 path: TILE x TILE tiles of G (TILE = 128 or 256); per K16 step
// TILE/128 MMAs of M=128 x N=TILE (the tile's row halves) into TILE/128
// accumulators (128 or all 512 TMEM columns). A stage holds both operands'
// TILE feature columns (TILE/64 64-column atoms each); 192 KB of stages, so
// a 256 tile moves 64 KB per 8.4 MFLOP and a 128 tile 32 KB per 2.1 MFLOP.
template <int TILE>
struct TcCfg {
    static constexpr int kHalves = TILE / 128;
    static constexpr int kOpBytes = kBK * TILE * 2;
    static constexpr int kStages = 196608 / (2 * kOpBytes);
    static constexpr uint32_t kTmemCols = kHalves * TILE;
    // kind::f16 instruction descriptor: D fp32 (bit 4), A and B bf16 (bits
    // 7, 10), A and B MN-major (bits 15, 16), N >> 3 at 17, M >> 4 at 24.
    static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) |
                                       (1u << 16) | ((uint32_t)(TILE >> 3) << 17) |
                                       ((uint32_t)(128 >> 4) << 24);
};
constexpr int kProducerWarps = 4, kEpilogueWarps = 4;
constexpr int kMmaWarp = kProducerWarps + kEpilogueWarps;
constexpr int kThreadsTc = (kMmaWarp + 1) * 32;
constexpr size_t kSmemTc = 1024 + 196608 + 256;
// CUDA-core path: 128 x 128 tiles.
constexpr int kTileSimt = 128;

struct GramArgs {
    const void* src;   // [Ksrc, N, Dsrc] (Ksrc = K, or 1 for the packed copy)
    long long N;       // rows
    int Dsrc;          // columns per source block
    int Mvalid;        // columns of O_all that exist (K*D); beyond: zeros
    int tile;          // tile edge (256 tensor cores, 128 CUDA cores)
    int nt;            // tiles per edge of G
    int T;             // upper-triangle tiles
    int splits;
    long long rows_per_split;  // multiple of kBK
    float* part;       // [splits * T][tile][tile]
    unsigned* status;
};

// Upper-triangle tile t -> (tm, tn), row-major over rows tm.
__device__ __forceinline__ void tile_of(int t, int nt, int& tm, int& tn) {
    tm = 0;
    while (t >= nt - tm) {
        t -= nt - tm;
        ++tm;
    }
    tn = tm + t;
}
__device__ __forceinline__ int tile_index(int tm, int tn, int nt) {
    return tm * nt - tm * (tm - 1) / 2 + (tn - tm);
}

// Shared-memory matrix descriptor, 128-byte swizzle, version bits 46-48 =
// 0b001 (the stage buffers are 1024-byte aligned).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(lbo >> 4) << 16) |
           ((uint64_t)(sbo >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// ---------------------------------------------------------------- bf16: tcgen05
// Warps 0-3 load both operand tiles of a stage: thread t owns 16-byte chunk
// column t % (TILE/8) of the TILE feature columns (atom cc / 8, chunk cc % 8
// in the 128-byte row) and rows t / (TILE/8) + (1024/TILE) i, so each row is
// read whole. In shared memory each operand is TILE/64 64-column atoms of
// kBK rows x 128 bytes, chunks XOR-swizzled by row (the layout a
// 128-byte-swizzled MN-major descriptor reads). Warp 8 issues the MMAs;
// warps 4-7 move the finished accumulators to the workspace.
template <int TILE, bool kWide>  // 16-byte source pieces (D % 8 == 0), else 4-byte (D even)
__global__ void __launch_bounds__(kThreadsTc, 1) gram_tc_kernel(const GramArgs a) {
    using Cf = TcCfg<TILE>;
    constexpr int kTileTc = TILE;
    constexpr int kStages = Cf::kStages;
    constexpr int kOpBytes = Cf::kOpBytes;
    constexpr uint32_t kIdesc = Cf::kIdesc;
    constexpr uint32_t kArrivals = kProducerWarps * 32;
    constexpr uint32_t kTmemCols = Cf::kTmemCols;
    constexpr int kCpr = TILE / 8;                        // 16-byte chunks per row
    constexpr int kRowsPerPass = kProducerWarps * 32 / kCpr;
    constexpr int kAtom = kBK * 128;  // bytes of one 64-column atom
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
        tmem_alloc(smem_u32((const void*)tmem_holder), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;
    pdl_wait();
    pdl_trigger();

    const int item = blockIdx.x;
    const int split = item / a.T;
    int tm, tn;
    tile_of(item - split * a.T, a.nt, tm, tn);
    const bool diag = tm == tn;
    const long long r_begin = (long long)split * a.rows_per_split;
    long long r_end = r_begin + a.rows_per_split;
    if (r_end > a.N) r_end = a.N;
    const int num_kb = r_end > r_begin ? (int)((r_end - r_begin + kBK - 1) / kBK) : 0;

    if (warp < kProducerWarps) {
        const __nv_bfloat16* __restrict__ src = static_cast<const __nv_bfloat16*>(a.src);
        const int cc = threadIdx.x % kCpr, rg = threadIdx.x / kCpr;
        const int atom = cc >> 3, q = cc & 7;
        // this thread's columns of each operand: source offset and validity
        // of each piece (one 8-column piece, or four 2-column pieces, which
        // never straddle two masks when D is even)
        constexpr int kPieces = kWide ? 1 : 4;
        long long col_off[2][kPieces];
        bool col_ok[2][kPieces];
#pragma unroll
        for (int op = 0; op < 2; ++op)
#pragma unroll
            for (int pc = 0; pc < kPieces; ++pc) {
                const int m = (op == 0 ? tm : tn) * kTileTc + cc * 8 + pc * 2;
                col_ok[op][pc] = m < a.Mvalid;
                const int blk = col_ok[op][pc] ? m / a.Dsrc : 0;
                col_off[op][pc] =
                    col_ok[op][pc] ? (long long)blk * a.N * a.Dsrc + (m - blk * a.Dsrc) : 0;
            }
        const int nops = diag ? 1 : 2;
        for (int kb = 0; kb < num_kb; ++kb) {
            const int s = kb % kStages;
            const uint32_t ph = (uint32_t)((kb / kStages) & 1);
            if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, a.status)) break;
            const long long n0 = r_begin + (long long)kb * kBK;
            for (int op = 0; op < nops; ++op) {
                const uint32_t st = (op == 0 ? sA : sB) + s * kOpBytes + atom * kAtom;
#pragma unroll 4
                for (int i = 0; i < kBK / kRowsPerPass; ++i) {
                    const int r = rg + kRowsPerPass * i;
                    const long long n = n0 + r;
                    const uint32_t dst = st + r * 128 + ((q ^ (r & 7)) << 4);
                    if constexpr (kWide) {
                        const bool valid = col_ok[op][0] && n < r_end;
                        const __nv_bfloat16* gp = src + (valid ? col_off[op][0] + n * a.Dsrc : 0);
                        cp_async_16(dst, gp, valid);
                    } else {
#pragma unroll
                        for (int pc = 0; pc < 4; ++pc) {
                            const bool valid = col_ok[op][pc] && n < r_end;
                            const __nv_bfloat16* gp =
                                src + (valid ? col_off[op][pc] + n * a.Dsrc : 0);
                            cp_async_4(dst + pc * 4, gp, valid);
                        }
                    }
                }
            }
            cp_async_arrive_noinc(full_bar(s));
        }
        cp_async_wait_all();
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
                // the operands were written by cp.async (generic proxy)
                fence_proxy_async_smem();
                const uint32_t a_st = sA + s * kOpBytes;
                const uint32_t b_st = diag ? a_st : sB + s * kOpBytes;
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k) {
                    const uint64_t bd = desc_sw128(b_st + k * 16 * 128, kAtom, 1024);
#pragma unroll
                    for (int h = 0; h < Cf::kHalves; ++h) {
                        const uint64_t ad = desc_sw128(a_st + h * 2 * kAtom + k * 16 * 128, kAtom, 1024);
                        tc_mma_bf16(tmem_base + h * TILE, ad, bd, kIdesc, (kb | k) != 0 ? 1u : 0u);
                    }
                }
                tc_commit(empty_bar(s));
            }
            if (ok && num_kb > 0) tc_commit(tfull_bar);
            // every MMA issued by this thread has completed once fin_bar fires
            tc_commit(fin_bar);
            mbar_wait_drain(fin_bar, 0, a.status);
            if (ok && num_kb == 0) mbar_arrive(tfull_bar);  // empty split: zeros
        }
        __syncwarp();
    } else {
        const int ew = warp - kProducerWarps;  // == warp % 4: TMEM lanes 32*ew..+32
        if (mbar_wait(tfull_bar, 0, abort_flag, a.status)) {
            tc_fence_after();
#pragma unroll 1
            for (int h = 0; h < Cf::kHalves; ++h) {
                const int row = h * 128 + ew * 32 + lane;
                float* dst = a.part + (long long)item * kTileTc * kTileTc + (long long)row * kTileTc;
#pragma unroll 1
                for (int cb = 0; cb < kTileTc / 32; ++cb) {
                    uint32_t r[32];
                    if (num_kb > 0) {
                        tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(ew * 32) << 16) +
                                               (uint32_t)(h * TILE + cb * 32),
                                           r);
                        tmem_ld_wait();
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) r[j] = 0u;
                    }
                    float4* d4 = reinterpret_cast<float4*>(dst + cb * 32);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        d4[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                            __uint_as_float(r[4 * j + 2]),
                                            __uint_as_float(r[4 * j + 3]));
                }
            }
            tc_fence_before();
        }
    }
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

// ---------------------------------------------------------------- fp32: CUDA cores
// 256 threads, 8 x 8 outputs each, rows of O staged 16 at a time.
constexpr int kSimtThreads = 256;
constexpr int kSimtBK = 16;

__global__ void __launch_bounds__(kSimtThreads) gram_simt_kernel(const GramArgs a) {
    __shared__ float As[kSimtBK][kTileSimt];
    __shared__ float Bs[kSimtBK][kTileSimt];
    pdl_wait();
    pdl_trigger();
    const float* __restrict__ src = static_cast<const float*>(a.src);
    const int item = blockIdx.x;
    const int split = item / a.T;
    int tm, tn;
    tile_of(item - split * a.T, a.nt, tm, tn);
    const bool diag = tm == tn;
    const long long r_begin = (long long)split * a.rows_per_split;
    long long r_end = r_begin + a.rows_per_split;
    if (r_end > a.N) r_end = a.N;
    const int t = threadIdx.x, ty = t >> 4, tx = t & 15;
    // columns this thread loads (fixed): mm = t % 128, rows t / 128 + 2 i
    const int mm = t & (kTileSimt - 1);
    long long off[2];
    bool okc[2];
#pragma unroll
    for (int op = 0; op < 2; ++op) {
        const int m = (op == 0 ? tm : tn) * kTileSimt + mm;
        okc[op] = m < a.Mvalid;
        const int blk = okc[op] ? m / a.Dsrc : 0;
        off[op] = okc[op] ? (long long)blk * a.N * a.Dsrc + (m - blk * a.Dsrc) : 0;
    }
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
    for (long long n0 = r_begin; n0 < r_end; n0 += kSimtBK) {
#pragma unroll
        for (int i = 0; i < kSimtBK / 2; ++i) {
            const int r = (t >> 7) + 2 * i;
            const long long n = n0 + r;
            As[r][mm] = (okc[0] && n < r_end) ? __ldg(src + off[0] + n * a.Dsrc) : 0.f;
            if (!diag) Bs[r][mm] = (okc[1] && n < r_end) ? __ldg(src + off[1] + n * a.Dsrc) : 0.f;
        }
        __syncthreads();
        const float(*Bp)[kTileSimt] = diag ? As : Bs;
#pragma unroll 4
        for (int k = 0; k < kSimtBK; ++k) {
            float av[8], bv[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) av[i] = As[k][ty * 8 + i];
#pragma unroll
            for (int j = 0; j < 8; ++j) bv[j] = Bp[k][tx * 8 + j];
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
    float* dst = a.part + (long long)item * kTileSimt * kTileSimt;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float4* d4 = reinterpret_cast<float4*>(dst + (ty * 8 + i) * kTileSimt + tx * 8);
        d4[0] = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        d4[1] = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
    }
}

// ---------------------------------------------------------------- pack (bf16, D % 8 != 0)
// opack[n][m] = O[m / D][n][m % D] for m < K*D, 0 for K*D <= m < Mp.
__global__ void pack_kernel(const __nv_bfloat16* __restrict__ O, long long N, int D, int KD,
                            int Mp, __nv_bfloat16* __restrict__ opack) {
    pdl_wait();
    pdl_trigger();
    const long long total = N * Mp;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        int m;
        const long long n = div32(e, Mp, m);
        __nv_bfloat16 v = __float2bfloat16_rn(0.f);
        if (m < KD) {
            const int k = m / D;
            v = O[((long long)k * N + n) * D + (m - k * D)];
        }
        opack[e] = v;
    }
}

// ---------------------------------------------------------------- pairs
// Block (p, c) <-> pair p = (i, k), i <= k (row-major over the upper
// triangle of the K x K matrix, diagonal included), and chunk c of
// kPairChunk entries of its D x D block, one entry per thread: the sum over
// the chunk of (sum over splits of G's entry)^2, written to P[p][c]. A
// thread issues its split loads kSplitBatch at a time (one round trip for
// up to kSplitBatch splits). Fixed orders.
constexpr int kPairThreads = 256;
constexpr int kPairChunk = kPairThreads;
constexpr int kSplitBatch = 16;

__device__ __forceinline__ int pair_of(int p, int K, int& k) {
    int i = 0;
    while (p >= K - i) {
        p -= K - i;
        ++i;
    }
    k = i + p;
    return i;
}
__device__ __forceinline__ int pair_index(int i, int k, int K) {  // i <= k
    return i * K - i * (i - 1) / 2 + (k - i);
}

__global__ void __launch_bounds__(kPairThreads)
    pair_kernel(const float* __restrict__ part, int K, int D, int tile_shift, int nt, int T,
                int splits, int nchunk, float* __restrict__ P) {
    __shared__ float red[kPairThreads / 32];
    pdl_wait();
    pdl_trigger();
    const int p = blockIdx.x / nchunk, chunk = blockIdx.x - p * nchunk;
    int k;
    const int i = pair_of(p, K, k);
    const int idx = chunk * kPairChunk + threadIdx.x;
    float acc = 0.f;
    if (idx < D * D) {
        const int d = idx / D, e = idx - d * D;
        int m = i * D + d, m2 = k * D + e;
        if (m > m2) {  // below the diagonal: the symmetric entry of an upper tile
            const int tmp = m;
            m = m2;
            m2 = tmp;
        }
        const int tmask = (1 << tile_shift) - 1;
        const long long tile_elems = 1ll << (2 * tile_shift);
        const long long split_stride = (long long)T * tile_elems;
        const float* src = part + tile_index(m >> tile_shift, m2 >> tile_shift, nt) * tile_elems +
                           ((long long)(m & tmask) << tile_shift) + (m2 & tmask);
        float g = 0.f;
        for (int sp0 = 0; sp0 < splits; sp0 += kSplitBatch) {
            float v[kSplitBatch];
#pragma unroll
            for (int j = 0; j < kSplitBatch; ++j)
                v[j] = sp0 + j < splits ? __ldg(src + (sp0 + j) * split_stride) : 0.f;
#pragma unroll
            for (int j = 0; j < kSplitBatch; ++j) g += v[j];
        }
        acc = g * g;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < kPairThreads / 32; ++w) tot += red[w];
        P[blockIdx.x] = tot;
    }
}

// ---------------------------------------------------------------- alpha
// Thread per mask k: S[i][k] = sum over chunks of P[pair(i, k)], the norms
// ||O_i^T O_i||_F = sqrt(S[i][i]), then sim and the update (fp32).
__device__ __forceinline__ float pair_sum(const float* P, int i, int k, int K, int nchunk) {
    const int p = i <= k ? pair_index(i, k, K) : pair_index(k, i, K);
    float s = 0.f;
    for (int c = 0; c < nchunk; ++c) s += __ldg(P + (long long)p * nchunk + c);
    return s;
}

// K <= kAlphaSmallK: one block; the pair sums S go to shared memory first,
// every pair's chunks loaded at once (one round trip), then thread k forms
// alpha_k from them (same arithmetic and order as alpha_kernel).
constexpr int kAlphaSmallK = 64;
constexpr int kAlphaThreads = 256;

__global__ void __launch_bounds__(kAlphaThreads)
    alpha_small_kernel(const float* __restrict__ P, int K, int nchunk, const float* alpha_in,
                       float* alpha_out, float* __restrict__ sim) {
    __shared__ float sS[kAlphaSmallK * (kAlphaSmallK + 1) / 2];
    pdl_wait();
    pdl_trigger();
    const int n_pairs = K * (K + 1) / 2;
    for (int p = threadIdx.x; p < n_pairs; p += kAlphaThreads) {
        float s = 0.f;
        for (int c0 = 0; c0 < nchunk; c0 += kSplitBatch) {
            float v[kSplitBatch];
#pragma unroll
            for (int j = 0; j < kSplitBatch; ++j)
                v[j] = c0 + j < nchunk ? __ldg(P + (long long)p * nchunk + c0 + j) : 0.f;
#pragma unroll
            for (int j = 0; j < kSplitBatch; ++j) s += v[j];
        }
        sS[p] = s;
    }
    __syncthreads();
    const int k = threadIdx.x;
    if (k >= K) return;
    const float nk = sqrtf(sS[pair_index(k, k, K)]);
    float sum = 0.f;
    for (int i = 0; i < K; ++i) {
        const float den = sqrtf(sS[pair_index(i, i, K)]) * nk;
        const float sik = sS[i <= k ? pair_index(i, k, K) : pair_index(k, i, K)];
        const float s = den > 0.f ? sik / den : 0.f;
        if (sim) sim[(long long)i * K + k] = s;
        if (i != k) sum += 1.f - s;
    }
    const float a0 = alpha_in[k];
    alpha_out[k] = K > 1 ? a0 + sum / (float)(K - 1) : a0;
}

__global__ void alpha_kernel(const float* __restrict__ P, int K, int nchunk, const float* alpha_in,
                             float* alpha_out, float* __restrict__ sim) {
    pdl_wait();
    pdl_trigger();
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= K) return;
    const float nk = sqrtf(pair_sum(P, k, k, K, nchunk));
    float sum = 0.f;
    for (int i = 0; i < K; ++i) {
        const float den = sqrtf(pair_sum(P, i, i, K, nchunk)) * nk;
        const float s = den > 0.f ? pair_sum(P, i, k, K, nchunk) / den : 0.f;
        if (sim) sim[(long long)i * K + k] = s;
        if (i != k) sum += 1.f - s;
    }
    const float a0 = alpha_in[k];
    alpha_out[k] = K > 1 ? a0 + sum / (float)(K - 1) : a0;
}

}  // namespace

hc_status launch_mask_score(const DeviceCtx* ctx, const void* O, hc_dtype dt, int K, long long N,
                            int D, const float* alpha_in, float* alpha_out, float* sim,
                            cudaStream_t s) {
    const bool tc = dt == HC_BF16;
    // 256-wide tensor-core tiles halve the operand bytes per flop; they pay
    // when K*D padded to a multiple of 256 keeps at least 80% of the Gram's
    // entries useful (measured: K*D = 960 in 61 us instead of 103 us with
    // 128 tiles; K*D = 640, padded to 768, in 48 us instead of 39 us), and
    // small K*D keeps 128 tiles (fewer row splits, less split-K traffic).
    const long long kd_256 = ((long long)K * D + 255) / 256 * 256;
    const bool big = tc && (long long)K * D >= 512 &&
                     (double)K * D * (double)K * D >= 0.8 * (double)kd_256 * (double)kd_256;
    const int tile = big ? 256 : 128;
    const int tile_shift = big ? 8 : 7;
    const int KD = K * D;
    const int nt = (KD + tile - 1) / tile;
    const int Mp = nt * tile;
    const int T = nt * (nt + 1) / 2;
    // Row splits: one CTA per SM (the kernel's shared memory), so pick the
    // smallest split count whose waves of splits * T items are >= 95% full
    // (else the fullest), with at least one 64-row block per split.
    long long max_splits = (N + kBK - 1) / kBK;
    const long long cap_splits = 8ll * ctx->num_sms / T + 1;
    if (max_splits > cap_splits) max_splits = cap_splits;
    if (max_splits < 1) max_splits = 1;
    int splits = 1;
    double best = 0.0;
    for (int sp = 1; sp <= max_splits; ++sp) {
        const long long items_sp = (long long)sp * T;
        const long long waves = (items_sp + ctx->num_sms - 1) / ctx->num_sms;
        const double eff = (double)items_sp / (double)(waves * ctx->num_sms);
        if (eff > best + 1e-9) {
            best = eff;
            splits = sp;
        }
        if (eff >= 0.95) break;
    }
    long long rps = (N + splits - 1) / splits;
    rps = (rps + kBK - 1) / kBK * kBK;
    if (rps < kBK) rps = kBK;
    const long long items = (long long)splits * T;

    const bool wide = D % 8 == 0 && (uintptr_t)O % 16 == 0;
    const bool packed = tc && !wide && (D % 2 != 0 || (uintptr_t)O % 4 != 0);
    const int n_pairs = K * (K + 1) / 2;
    const int nchunk = (D * D + kPairChunk - 1) / kPairChunk;
    const size_t part_bytes = sizeof(float) * (size_t)items * tile * tile;
    const size_t s_bytes = sizeof(float) * (size_t)n_pairs * nchunk;
    const size_t pack_off = (part_bytes + s_bytes + 255) / 256 * 256;
    const size_t pack_bytes = packed ? sizeof(__nv_bfloat16) * (size_t)N * Mp : 0;
    uint8_t* ws = (uint8_t*)stream_workspace(s, pack_off + pack_bytes);
    if (!ws) return HC_ERR_CUDA;
    float* part = (float*)ws;
    float* S = (float*)(ws + part_bytes);

    if (N == 0) {
        hc_status st = check_cuda(cudaMemsetAsync(S, 0, s_bytes, s), "cudaMemsetAsync(S)");
        if (st != HC_OK) return st;
    } else {
        GramArgs g{};
        g.src = O;
        g.N = N;
        g.Dsrc = D;
        g.Mvalid = KD;
        g.tile = tile;
        g.nt = nt;
        g.T = T;
        g.splits = splits;
        g.rows_per_split = rps;
        g.part = part;
        g.status = ctx->status;
        hc_status st;
        if (tc) {
            if (packed) {
                __nv_bfloat16* opack = (__nv_bfloat16*)(ws + pack_off);
                long long blocks = (N * Mp + 255) / 256;
                if (blocks > (long long)ctx->num_sms * 16) blocks = (long long)ctx->num_sms * 16;
                st = launch_pdl(pack_kernel, dim3((unsigned)blocks), dim3(256), 0, s, "pack_kernel",
                                (const __nv_bfloat16*)O, N, D, KD, Mp, opack);
                if (st != HC_OK) return st;
                g.src = opack;
                g.Dsrc = Mp;
                g.Mvalid = Mp;
            }
            static bool attr_set[64] = {};
            if (!attr_set[ctx->device]) {
                const void* fns[4] = {(const void*)gram_tc_kernel<128, true>,
                                      (const void*)gram_tc_kernel<128, false>,
                                      (const void*)gram_tc_kernel<256, true>,
                                      (const void*)gram_tc_kernel<256, false>};
                for (const void* f : fns) {
                    st = check_cuda(cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                         (int)kSmemTc),
                                    "cudaFuncSetAttribute(gram_tc_kernel)");
                    if (st != HC_OK) return st;
                }
                attr_set[ctx->device] = true;
            }
            const bool w16 = wide || packed;
            const dim3 grid((unsigned)items), block(kThreadsTc);
            if (big)
                st = w16 ? launch_pdl(gram_tc_kernel<256, true>, grid, block, kSmemTc, s,
                                      "gram_tc_kernel", g)
                         : launch_pdl(gram_tc_kernel<256, false>, grid, block, kSmemTc, s,
                                      "gram_tc_kernel", g);
            else
                st = w16 ? launch_pdl(gram_tc_kernel<128, true>, grid, block, kSmemTc, s,
                                      "gram_tc_kernel", g)
                         : launch_pdl(gram_tc_kernel<128, false>, grid, block, kSmemTc, s,
                                      "gram_tc_kernel", g);
        } else {
            st = launch_pdl(gram_simt_kernel, dim3((unsigned)items), dim3(kSimtThreads), 0, s,
                            "gram_simt_kernel", g);
        }
        if (st != HC_OK) return st;
        st = launch_pdl(pair_kernel, dim3((unsigned)(n_pairs * nchunk)), dim3(kPairThreads), 0, s,
                        "pair_kernel", (const float*)part, K, D, tile_shift, nt, T, splits, nchunk,
                        S);
        if (st != HC_OK) return st;
    }
    if (K <= kAlphaSmallK)
        return launch_pdl(alpha_small_kernel, dim3(1), dim3(kAlphaThreads), 0, s,
                          "alpha_small_kernel", (const float*)S, K, nchunk, alpha_in, alpha_out,
                          sim);
    return launch_pdl(alpha_kernel, dim3((unsigned)((K + 127) / 128)), dim3(128), 0, s,
                      "alpha_kernel", (const float*)S, K, nchunk, alpha_in, alpha_out, sim);
}

}  // namespace hc
