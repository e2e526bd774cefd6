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
// upper-triangle 128 x 128 tiles are computed), and a squared block norm
// needs the complete sum over N before squaring. So:
//   1. gram: split-K partial tiles of G, one work item per (row split,
//      upper tile), written to a workspace [item][128][128] fp32.
//      bf16: tcgen05 (both operands MN-major from shared memory, fp32
//      accumulators in TMEM); fp32: CUDA-core FFMA tiles.
//   2. pairs: one block per pair i <= k sums the splits of every element of
//      its D x D block (in a fixed order), squares and reduces: S[i][k].
//   3. alpha: one block turns S into sim and the update.
// Deterministic: no atomics, every sum in a fixed order.
//
// bf16 operands are read straight from [K, N, D] with 16-byte cp.async when
// D is a multiple of 8 (a 16-byte chunk never straddles two masks); other D
// are first packed into a zero-padded [N, Mp] copy (Mp = K*D rounded up to
// 128) in the workspace.
#include <cuda_bf16.h>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kTile = 128;  // G tile edge (both operands: 128 feature columns)
constexpr int kBK = 64;     // rows of O per pipeline stage (the contraction dim)
constexpr int kStages = 6;
constexpr int kOpBytes = kBK * kTile * 2;  // one operand tile of a stage (two 64-column atoms)
constexpr int kProducerWarps = 4, kEpilogueWarps = 4;
constexpr int kMmaWarp = kProducerWarps + kEpilogueWarps;
constexpr int kThreadsTc = (kMmaWarp + 1) * 32;
constexpr int kPartElems = kTile * kTile;
constexpr size_t kSmemTc = 1024 + (size_t)kStages * 2 * kOpBytes + 256;
// kind::f16 instruction descriptor: D fp32 (bit 4), A and B bf16 (bits 7,
// 10), A and B MN-major (bits 15, 16), N >> 3 at 17, M >> 4 at 24.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) |
                            ((uint32_t)(kTile >> 3) << 17) | ((uint32_t)(kTile >> 4) << 24);

struct GramArgs {
    const void* src;   // [Ksrc, N, Dsrc] (Ksrc = K, or 1 for the packed copy)
    long long N;       // rows
    int Dsrc;          // columns per source block
    int Mvalid;        // columns of O_all that exist (K*D); beyond: zeros
    int nt;            // tiles per edge of G
    int T;             // upper-triangle tiles
    int splits;
    long long rows_per_split;  // multiple of kBK
    float* part;       // [splits * T][128][128]
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
// column cc = t % 16 of the 128 feature columns (atom cc / 8, chunk cc % 8 in
// the 128-byte row) and rows t / 16 + 8 i. In shared memory each operand is
// two 64-column atoms of kBK rows x 128 bytes, chunks XOR-swizzled by row
// (the layout a 128-byte-swizzled MN-major descriptor reads). Warp 8 issues
// the MMAs; warps 4-7 move the finished accumulator to the workspace.
__global__ void __launch_bounds__(kThreadsTc, 1) gram_tc_kernel(const GramArgs a) {
    constexpr uint32_t kArrivals = kProducerWarps * 32;
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
        const int t = threadIdx.x;
        const int cc = t & 15, atom = cc >> 3, q = cc & 7;
        // this thread's columns of each operand: source offset and validity
        long long col_off[2];
        bool col_ok[2];
#pragma unroll
        for (int op = 0; op < 2; ++op) {
            const int m = (op == 0 ? tm : tn) * kTile + cc * 8;
            col_ok[op] = m < a.Mvalid;
            const int blk = col_ok[op] ? m / a.Dsrc : 0;
            col_off[op] = col_ok[op] ? (long long)blk * a.N * a.Dsrc + (m - blk * a.Dsrc) : 0;
        }
        const int nops = diag ? 1 : 2;
        bool ok = true;
        for (int kb = 0; kb < num_kb; ++kb) {
            const int s = kb % kStages;
            const uint32_t ph = (uint32_t)((kb / kStages) & 1);
            if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, a.status)) {
                ok = false;
                break;
            }
            const long long n0 = r_begin + (long long)kb * kBK;
            for (int op = 0; op < nops; ++op) {
                const uint32_t st = (op == 0 ? sA : sB) + s * kOpBytes + atom * (kBK * 128);
#pragma unroll
                for (int i = 0; i < kBK / 8; ++i) {
                    const int r = (t >> 4) + 8 * i;
                    const long long n = n0 + r;
                    const bool valid = col_ok[op] && n < r_end;
                    const __nv_bfloat16* gp = src + (valid ? col_off[op] + n * a.Dsrc : 0);
                    cp_async_16(st + r * 128 + ((q ^ (r & 7)) << 4), gp, valid);
                }
            }
            cp_async_arrive_noinc(full_bar(s));
        }
        cp_async_wait_all();
        (void)ok;
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
                    const uint64_t ad = desc_sw128(a_st + k * 16 * 128, kBK * 128, 1024);
                    const uint64_t bd = desc_sw128(b_st + k * 16 * 128, kBK * 128, 1024);
                    tc_mma_bf16(tmem_base, ad, bd, kIdesc, (kb | k) != 0 ? 1u : 0u);
                }
                tc_commit(empty_bar(s));
            }
            if (ok && num_kb > 0) tc_commit(tfull_bar);
            // every MMA issued by this thread has completed once fin_bar fires
            tc_commit(fin_bar);
            int no_abort = 0;
            mbar_wait(fin_bar, 0, &no_abort, a.status);
            if (ok && num_kb == 0) mbar_arrive(tfull_bar);  // empty split: zeros
        }
        __syncwarp();
    } else {
        const int ew = warp - kProducerWarps;  // == warp % 4: TMEM lanes 32*ew..+32
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
                    for (int j = 0; j < 32; ++j) r[j] = 0u;
                }
                float4* d4 = reinterpret_cast<float4*>(dst + cb * 32);
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    d4[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                        __uint_as_float(r[4 * j + 2]),
                                        __uint_as_float(r[4 * j + 3]));
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

// ---------------------------------------------------------------- fp32: CUDA cores
// 256 threads, 8 x 8 outputs each, rows of O staged 16 at a time.
constexpr int kSimtThreads = 256;
constexpr int kSimtBK = 16;

__global__ void __launch_bounds__(kSimtThreads) gram_simt_kernel(const GramArgs a) {
    __shared__ float As[kSimtBK][kTile];
    __shared__ float Bs[kSimtBK][kTile];
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
    const int mm = t & (kTile - 1);
    long long off[2];
    bool okc[2];
#pragma unroll
    for (int op = 0; op < 2; ++op) {
        const int m = (op == 0 ? tm : tn) * kTile + mm;
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
        const float(*Bp)[kTile] = diag ? As : Bs;
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
    float* dst = a.part + (long long)item * kPartElems;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        float4* d4 = reinterpret_cast<float4*>(dst + (ty * 8 + i) * kTile + tx * 8);
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
        const long long n = e / Mp;
        const int m = (int)(e - n * Mp);
        __nv_bfloat16 v = __float2bfloat16_rn(0.f);
        if (m < KD) {
            const int k = m / D;
            v = O[((long long)k * N + n) * D + (m - k * D)];
        }
        opack[e] = v;
    }
}

// ---------------------------------------------------------------- pairs
// Block p <-> pair (i, k), i <= k (row-major over the upper triangle of the
// K x K matrix). S[i][k] = sum over the D x D block of (sum over splits)^2.
constexpr int kPairThreads = 256;

__global__ void __launch_bounds__(kPairThreads)
    pair_kernel(const float* __restrict__ part, int K, int D, int nt, int T, int splits,
                float* __restrict__ S) {
    __shared__ double red[kPairThreads / 32];
    pdl_wait();
    pdl_trigger();
    int i = 0, rem = blockIdx.x;
    while (rem >= K - i) {
        rem -= K - i;
        ++i;
    }
    const int k = i + rem;
    float acc = 0.f;
    const int DD = D * D;
    for (int idx = threadIdx.x; idx < DD; idx += kPairThreads) {
        const int d = idx / D, e = idx - d * D;
        int m = i * D + d, m2 = k * D + e;
        if (m > m2) {  // below the diagonal: the symmetric entry of an upper tile
            const int tmp = m;
            m = m2;
            m2 = tmp;
        }
        const int t = tile_index(m >> 7, m2 >> 7, nt);
        const long long off = ((long long)(m & 127) << 7) + (m2 & 127);
        float g = 0.f;
        for (int s = 0; s < splits; ++s) g += __ldg(part + ((long long)s * T + t) * kPartElems + off);
        acc = fmaf(g, g, acc);
    }
    double v = acc;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
        double tot = 0.0;
        for (int w = 0; w < kPairThreads / 32; ++w) tot += red[w];
        S[i * K + k] = (float)tot;
        S[k * K + i] = (float)tot;
    }
}

// ---------------------------------------------------------------- alpha
__global__ void alpha_kernel(const float* __restrict__ S, int K, const float* alpha_in,
                             float* alpha_out, float* __restrict__ sim) {
    pdl_wait();
    pdl_trigger();
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
        const double nk = sqrt((double)S[k * K + k]);
        double sum = 0.0;
        for (int i = 0; i < K; ++i) {
            const double den = sqrt((double)S[i * K + i]) * nk;
            const double s = den > 0.0 ? (double)S[i * K + k] / den : 0.0;
            if (sim) sim[i * K + k] = (float)s;
            if (i != k) sum += 1.0 - s;
        }
        const float a0 = alpha_in[k];
        alpha_out[k] = K > 1 ? (float)((double)a0 + sum / (double)(K - 1)) : a0;
    }
}

}  // namespace

hc_status launch_mask_score(const DeviceCtx* ctx, const void* O, hc_dtype dt, int K, long long N,
                            int D, const float* alpha_in, float* alpha_out, float* sim,
                            cudaStream_t s) {
    const int KD = K * D;
    const int Mp = (KD + kTile - 1) / kTile * kTile;
    const int nt = Mp / kTile;
    const int T = nt * (nt + 1) / 2;
    int splits = ctx->num_sms / T;
    if (splits < 1) splits = 1;
    const long long max_splits = (N + kBK - 1) / kBK;
    if (splits > max_splits) splits = (int)(max_splits > 0 ? max_splits : 1);
    long long rps = (N + splits - 1) / splits;
    rps = (rps + kBK - 1) / kBK * kBK;
    if (rps < kBK) rps = kBK;
    const long long items = (long long)splits * T;

    const bool tc = dt == HC_BF16;
    const bool packed = tc && (D % 8 != 0 || (uintptr_t)O % 16 != 0);
    const size_t part_bytes = sizeof(float) * (size_t)items * kPartElems;
    const size_t s_bytes = sizeof(float) * (size_t)K * K;
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
                st = check_cuda(cudaFuncSetAttribute(gram_tc_kernel,
                                                     cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                     (int)kSmemTc),
                                "cudaFuncSetAttribute(gram_tc_kernel)");
                if (st != HC_OK) return st;
                attr_set[ctx->device] = true;
            }
            st = launch_pdl(gram_tc_kernel, dim3((unsigned)items), dim3(kThreadsTc), kSmemTc, s,
                            "gram_tc_kernel", g);
        } else {
            st = launch_pdl(gram_simt_kernel, dim3((unsigned)items), dim3(kSimtThreads), 0, s,
                            "gram_simt_kernel", g);
        }
        if (st != HC_OK) return st;
        st = launch_pdl(pair_kernel, dim3((unsigned)(K * (K + 1) / 2)), dim3(kPairThreads), 0, s,
                        "pair_kernel", (const float*)part, K, D, nt, T, splits, S);
        if (st != HC_OK) return st;
    }
    return launch_pdl(alpha_kernel, dim3(1), dim3(256), 0, s, "alpha_kernel", (const float*)S, K,
                      alpha_in, alpha_out, sim);
}

}  // namespace hc
