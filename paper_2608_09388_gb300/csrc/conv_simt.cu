// Spiral convolution / linear layer on CUDA cores (FFMA, fp32 accumulate).
//
// Used for fp32 (genuine IEEE fp32 multiply-adds: no TF32) and for bf16
// shapes the tensor-core kernel does not take (channel counts that are not a
// multiple of 8, e.g. a 45-channel input or a 42- or 1-wide output head).
//
// Each CTA owns a 64-row x 64-column output tile and walks K = L*C_in in
// chunks of KC (128 when K <= 256, else 64): the A chunk is gathered through the per-tile table of source
// rows (idx() of Eq. 4: -1 when the tap is absent) and the W chunk read
// directly, every load of a chunk issued before any is used (one dependent
// round trip per KC of K rather than per 16: the small layers this kernel
// serves are latency-bound; deeper layers take the smaller chunk, whose
// registers and shared memory let more CTAs share an SM); each thread then
// accumulates a 4x4 block. The
// grid is persistent over row tiles because the row count N' is only known on
// the device.
#include <cuda_bf16.h>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kBM = 64;
constexpr int kBN = 64;
constexpr int kThreads = 256;
constexpr int kAPitch = kBM + 4;  // floats per As row (16-byte aligned rows)

// Shared memory of a chunk depth: As [KC][kAPitch] and Bs [KC][kBN] floats.
template <int KC>
constexpr size_t chunk_smem_bytes() {
    return sizeof(float) * (size_t)(KC * kAPitch + KC * kBN);
}

template <typename T>
__device__ __forceinline__ float to_float(T v);
template <>
__device__ __forceinline__ float to_float<float>(float v) {
    return v;
}
template <>
__device__ __forceinline__ float to_float<__nv_bfloat16>(__nv_bfloat16 v) {
    return __bfloat162float(v);
}
template <typename T>
__device__ __forceinline__ T from_float(float v);
template <>
__device__ __forceinline__ float from_float<float>(float v) {
    return v;
}
template <>
__device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

template <typename T, int kKC>
__global__ void __launch_bounds__(kThreads) conv_simt_kernel(const ConvArgs a) {
    constexpr int kAsFloats = kKC * kAPitch;
    constexpr int kBsFloats = kKC * kBN;
    // per thread per chunk: A rows tid/kKC + (256/kKC) i, B k-rows tid/64 + 4i
    constexpr int kAPer = kBM * kKC / kThreads;
    constexpr int kBPer = kKC * kBN / kThreads;
    constexpr int kAStep = kThreads / kKC;
    // dynamic: As [kKC][kAPitch] float, Bs [kKC][kBN] float, src_tab [kBM][L] int
    extern __shared__ __align__(16) float smem_f[];
    float* const As = smem_f;
    float* const Bs = smem_f + kAsFloats;
    int* const src_tab = reinterpret_cast<int*>(smem_f + kAsFloats + kBsFloats);

    const T* __restrict__ x = static_cast<const T*>(a.x);
    const T* __restrict__ W = static_cast<const T*>(a.W);
    T* __restrict__ y = static_cast<T*>(a.y);
    pdl_wait();
    pdl_trigger();
    const long long rows = active_rows(a);
    const long long m_tiles = (rows + kBM - 1) / kBM;
    const int n0 = blockIdx.y * kBN;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int L = a.L, C_in = a.C_in, C_out = a.C_out, K = a.K;

    for (long long mt = blockIdx.x; mt < m_tiles; mt += gridDim.x) {
        const long long m0 = mt * kBM;
        __syncthreads();  // the previous tile is done with src_tab
        {
            // Four threads per row, slots l = part + 4*j: the coordinate, the
            // spiral entries and the row_of lookups are each issued together
            // (three dependent round trips per tile).
            const int r = tid >> 2, part = tid & 3;
            const long long n = m0 + r;
            const bool in = n < rows;
            const long long nn = in ? n : 0;
            unsigned err = 0;
            int b = 0, v = 0;
            if (a.mode == kSparseDenseX || a.mode == kSparseCompactX) {
                b = __ldg(a.coords + 2 * nn);
                v = __ldg(a.coords + 2 * nn + 1);
            } else if (a.mode == kDense) {
                b = (int)(nn / a.V);
                v = (int)(nn - (long long)b * a.V);
            }
            const bool in_range = b >= 0 && b < a.B && v >= 0 && v < a.V;
            if (in && !in_range) err |= kErrIndex;
            const bool ok = in && in_range;
            if (!ok) b = v = 0;
            const bool linear = a.mode == kLinear;
            const bool rb = a.mode == kRulebook;
            // Loads from clamped, always-valid addresses first; checks after.
            int u[HC_MAX_SPIRAL / 4];
#pragma unroll
            for (int j = 0; j < HC_MAX_SPIRAL / 4; ++j) {
                const int l = part + 4 * j < L ? part + 4 * j : L - 1;
                u[j] = linear ? 0
                       : rb   ? __ldg(a.rulebook + (long long)l * a.capacity + nn)
                              : __ldg(a.spiral + (long long)v * L + l);
            }
#pragma unroll
            for (int j = 0; j < HC_MAX_SPIRAL / 4; ++j) {
                const int l = part + 4 * j;
                if (l >= L) continue;
                int src = -1;
                if (ok && linear) {
                    src = (int)n;
                } else if (ok && rb) {
                    if (u[j] < -1 || u[j] >= a.x_rows) err |= kErrIndex;
                    else src = u[j];
                } else if (ok) {
                    const int uu = u[j];
                    if (uu < -1 || uu >= a.V) err |= kErrIndex;
                    if (uu >= 0 && uu < a.V) {
                        const long long dr = (long long)b * a.V + uu;
                        if (a.mode == kDense) {
                            src = (int)dr;
                        } else {
                            const int jj = __ldg(a.row_of + dr);
                            if (jj < -1 || jj >= rows) err |= kErrIndex;
                            if (jj >= 0 && jj < rows) src = a.mode == kSparseDenseX ? (int)dr : jj;
                        }
                    }
                }
                src_tab[r * L + l] = src;
            }
            if (err) report(a.status, err);
        }
        __syncthreads();

        float acc[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

        // this thread's A column of every chunk (k = k0 + ka) and B column o
        const int ka = tid & (kKC - 1), ra = tid / kKC;
        const int ob = tid & (kBN - 1), kbr = tid >> 6;
        for (int k0 = 0; k0 < K; k0 += kKC) {
            const int k = k0 + ka;
            const bool kin = k < K;
            const int l = kin ? k / C_in : 0, c = kin ? k - l * C_in : 0;
            float av_[kAPer], bv_[kBPer];
            // every load of the chunk first ...
#pragma unroll
            for (int i = 0; i < kAPer; ++i) {
                const int r = ra + kAStep * i;
                const int s = kin ? src_tab[r * L + l] : -1;
                av_[i] = s >= 0 ? to_float(x[(long long)s * C_in + c]) : 0.f;
            }
#pragma unroll
            for (int i = 0; i < kBPer; ++i) {
                const int kk = kbr + 4 * i, col = n0 + ob;
                bv_[i] = (k0 + kk < K && col < C_out)
                             ? to_float(W[(long long)(k0 + kk) * C_out + col])
                             : 0.f;
            }
            // ... then the stores to shared memory
#pragma unroll
            for (int i = 0; i < kAPer; ++i) As[ka * kAPitch + ra + kAStep * i] = av_[i];
#pragma unroll
            for (int i = 0; i < kBPer; ++i) Bs[(kbr + 4 * i) * kBN + ob] = bv_[i];
            __syncthreads();
            const int kn = K - k0 < kKC ? K - k0 : kKC;
#pragma unroll 16
            for (int kk = 0; kk < kn; ++kk) {
                const float4 av = *reinterpret_cast<const float4*>(&As[kk * kAPitch + ty * 4]);
                const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk * kBN + tx * 4]);
                const float ar[4] = {av.x, av.y, av.z, av.w};
                const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(ar[i], br[j], acc[i][j]);
            }
            __syncthreads();
        }

#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const long long n = m0 + ty * 4 + i;
            if (n >= rows) continue;
            T* dp = nullptr;  // fused scatter destination row, if any
            if (a.out_dense) {
                const int b = __ldg(a.out_coords + 2 * n), v = __ldg(a.out_coords + 2 * n + 1);
                if (b >= 0 && b < a.out_B && v >= 0 && v < a.out_V)
                    dp = static_cast<T*>(a.out_dense) + ((long long)b * a.out_V + v) * C_out;
                else
                    report(a.status, kErrIndex);
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int col = n0 + tx * 4 + j;
                if (col >= C_out) continue;
                const float z = acc[i][j] + (a.bias ? __ldg(a.bias + col) : 0.f);
                const T val = from_float<T>(act_apply(z, a.act));
                if (y) y[n * C_out + col] = val;
                if (dp) dp[col] = val;
            }
        }
    }
}

}  // namespace

hc_status launch_conv_simt(const DeviceCtx* ctx, const ConvArgs& a, hc_dtype dt, cudaStream_t s) {
    long long cap_tiles = (a.capacity + kBM - 1) / kBM;
    long long gx = cap_tiles < (long long)ctx->num_sms * 8 ? cap_tiles : (long long)ctx->num_sms * 8;
    if (gx < 1) gx = 1;
    dim3 grid((unsigned)gx, (unsigned)((a.C_out + kBN - 1) / kBN));
    const size_t tab = sizeof(int) * (size_t)kBM * a.L;
    static bool attr_set[64] = {};
    if (!attr_set[ctx->device]) {
        hc_status st = HC_OK;
        auto allow = [&](auto kernel, size_t bytes) {
            if (st == HC_OK)
                st = check_cuda(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                     (int)bytes),
                                "cudaFuncSetAttribute(conv_simt_kernel)");
        };
        const size_t tab_max = sizeof(int) * (size_t)kBM * HC_MAX_SPIRAL;
        allow(conv_simt_kernel<float, 128>, chunk_smem_bytes<128>() + tab_max);
        allow(conv_simt_kernel<__nv_bfloat16, 128>, chunk_smem_bytes<128>() + tab_max);
        allow(conv_simt_kernel<float, 64>, chunk_smem_bytes<64>() + tab_max);
        allow(conv_simt_kernel<__nv_bfloat16, 64>, chunk_smem_bytes<64>() + tab_max);
        if (st != HC_OK) return st;
        attr_set[ctx->device] = true;
    }
    if (a.K <= 256) {
        const size_t smem = chunk_smem_bytes<128>() + tab;
        if (dt == HC_F32)
            return launch_pdl(conv_simt_kernel<float, 128>, grid, dim3(kThreads), smem, s,
                              "conv_simt_kernel", a);
        return launch_pdl(conv_simt_kernel<__nv_bfloat16, 128>, grid, dim3(kThreads), smem, s,
                          "conv_simt_kernel", a);
    }
    const size_t smem = chunk_smem_bytes<64>() + tab;
    if (dt == HC_F32)
        return launch_pdl(conv_simt_kernel<float, 64>, grid, dim3(kThreads), smem, s,
                          "conv_simt_kernel", a);
    return launch_pdl(conv_simt_kernel<__nv_bfloat16, 64>, grid, dim3(kThreads), smem, s,
                      "conv_simt_kernel", a);
}

}  // namespace hc
