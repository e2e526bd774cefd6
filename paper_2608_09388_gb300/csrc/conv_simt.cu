// Spiral convolution / linear layer on CUDA cores (FFMA, fp32 accumulate).
//
// Used for fp32 (genuine IEEE fp32 multiply-adds: no TF32) and for bf16
// shapes the tensor-core kernel does not take (channel counts that are not a
// multiple of 8, e.g. a 45-channel input or a 42- or 1-wide output head).
//
// Each CTA owns a 64-row x 64-column output tile and walks K = L*C_in in
// steps of 16: the A tile is gathered through the per-tile table of source
// rows (idx() of Eq. 4: -1 when the tap is absent), the W tile is read
// directly, and each thread accumulates a 4x4 block. The grid is persistent
// over row tiles because the row count N' is only known on the device.
#include <cuda_bf16.h>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kBM = 64;
constexpr int kBN = 64;
constexpr int kBK = 16;
constexpr int kThreads = 256;

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

template <typename T>
__global__ void __launch_bounds__(kThreads) conv_simt_kernel(const ConvArgs a) {
    __shared__ __align__(16) float As[kBK][kBM + 4];
    __shared__ __align__(16) float Bs[kBK][kBN];
    extern __shared__ int src_tab[];  // [kBM][L]

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

        for (int k0 = 0; k0 < K; k0 += kBK) {
            for (int e = tid; e < kBM * kBK; e += kThreads) {
                const int r = e / kBK, kk = e - r * kBK;
                const int k = k0 + kk;
                float val = 0.f;
                if (k < K) {
                    const int l = k / C_in, c = k - l * C_in;
                    const int s = src_tab[r * L + l];
                    if (s >= 0) val = to_float(x[(long long)s * C_in + c]);
                }
                As[kk][r] = val;
            }
            for (int e = tid; e < kBK * kBN; e += kThreads) {
                const int kk = e / kBN, o = e - kk * kBN;
                const int k = k0 + kk, col = n0 + o;
                Bs[kk][o] = (k < K && col < C_out) ? to_float(W[(long long)k * C_out + col]) : 0.f;
            }
            __syncthreads();
#pragma unroll
            for (int kk = 0; kk < kBK; ++kk) {
                const float4 av = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
                const float4 bv = *reinterpret_cast<const float4*>(&Bs[kk][tx * 4]);
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
    size_t smem = sizeof(int) * (size_t)kBM * a.L;
    if (dt == HC_F32)
        return launch_pdl(conv_simt_kernel<float>, grid, dim3(kThreads), smem, s,
                          "conv_simt_kernel", a);
    return launch_pdl(conv_simt_kernel<__nv_bfloat16>, grid, dim3(kThreads), smem, s,
                      "conv_simt_kernel", a);
}

}  // namespace hc
