// Sparse / dense spiral convolution and linear layer on the sm_103a tensor
// cores: gather -> tcgen05.mma (bf16 x bf16 -> fp32 in TMEM) -> fused
// bias + activation epilogue -> bf16 compact rows.
//
// The gathered operand A is the implicit [rows, L*C_in] matrix whose row n
// is the concatenation over spiral slots l of the input row idx(b, spiral[v][l])
// (zeros for absent taps, Eq. 4); the layer computes A * W + bias (Eq. 5 with
// the bias of Eq. 6) and the activation of Eq. 10.
//
// One persistent CTA per SM, 352 threads in five roles (384 with two-half
// items). A work item is tm 128-row halves of output rows times BN output
// channels; both halves are multiplied by the same W slice of every stage,
// which halves the weight traffic and the per-stage overhead per MMA of
// large layers. tm = 2 for the dense layer when it gives every SM at least
// two items, and for a rulebook call whose host-side row estimate gives
// every SM one; a rulebook call without an estimate but with the capacity
// for that many goes to conv_tc_auto_kernel, which reads the row count on
// the device and runs whichever role set it calls for; else tm = 1.
//   warp 9     index warp: for each item, resolves the L x (tm*128) tap table
//              (from the rulebook, or coords -> spiral -> row_of, i.e. idx()
//              of Eq. 4) with every load of a phase in flight at once, into
//              one of two tables, so the next item's table is built while the
//              current one is used (two-half items: warp 11 builds half 1);
//   warps 0-3  producers: fill a stage with the tm x 128 rows x 64 bf16 of A
//              for one k-block. The 128 threads gather A with 16-byte cp.async
//              through the tap table (zero-fill for absent taps and for k
//              past L*C_in) and signal completion on the stage's "full"
//              mbarrier without blocking;
//   warp 10    weight loader (one thread): the 64 x BN slice of W of each
//              stage by TMA (one 3-D box when C_out is a multiple of 64) onto
//              the same barrier (transaction count). Gather and weight loads
//              thus use different engines, and the gather warps never wait on
//              a TMA issue (which held the whole ring back when a gather
//              thread issued it);
//   warp 8     MMA issuer (one thread): per stage 4 x tm tcgen05.mma
//              (M = 128, N = BN, K = 16) into the item's TMEM accumulators,
//              tcgen05.commit frees the stage;
//   warps 4-7  epilogue: tcgen05.ld each half's 128 x BN fp32 accumulator
//              (warp w reads TMEM lanes 32*(w%4)..+32), activation, round to
//              bf16 and store; then tcgen05.st the bias of the item after
//              next into every row of the freed accumulators, onto which its
//              MMAs accumulate. Two accumulator sets (2*tm*BN TMEM columns)
//              let the epilogue of one item overlap the main loop of the next.
// The dense layer with 128 output channels and two-half items (TR) swaps the
// operands: D^T = W^T A^T, one tcgen05.mma of M = 128 channels (the W slice,
// MN-major, as staged) x N = 256 rows (the two halves of A, K-major, as
// staged) per K16 step instead of two of 128 x 128, i.e. half the MMAs and
// a quarter less shared-memory operand traffic per k-block (dense layer
// 200.7 -> 181.6 us at 64 x 10475 rows, L = 9, 128 -> 128). Its accumulator
// holds a channel per TMEM lane and a row per column, so the epilogue stages
// each 32 x 32 block transposed through shared memory, and the bias is one
// value per lane.
// The roles are one function template (conv_roles) instantiated per half
// count and layout: each role runs its whole loop in a copy compiled for its
// half count (a run-time half loop between the MMAs and copies cost ~1 us
// per launch at the small layers), and conv_tc_auto_kernel holds the
// one-half and the transposed two-half copies, one branch taken per launch.
// The stage ring holds a.stages two-half stages; one-half items cut the same
// bytes into more (up to kRing) stages of 16 KB of A plus the W slice.
// Shared-memory operand layouts (canonical tcgen05 forms, 128-byte swizzle):
//   A: K-major, per half row r at r*128 bytes, 16-byte chunk q
//      stored at chunk q ^ (r % 8); 8-row groups 1024 bytes apart (SBO).
//   B: MN-major (W is [K, C_out] row-major, C_out contiguous), per 64-column
//      block a [64 K-rows x 128 bytes] slab, K-row kr at kr*128 with chunk
//      q stored at q ^ (kr % 8); 8-row groups 1024 bytes apart (SBO), the
//      64-column blocks BK*128 bytes apart (LBO).
// The TMA 128-byte swizzle writes exactly the B layout (stage buffers are
// 1024-byte aligned); the cp.async gather computes the A swizzle itself.
// Every mbarrier wait is bounded (hc::kWaitLimitNs); on timeout the CTA
// records HC_ERR_TIMEOUT, unwinds, waits for its own copies and MMAs and
// frees its TMEM.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "hc_internal.cuh"

namespace hc {
namespace {

constexpr int kBM = 128;  // rows per tile half = TMEM lanes
constexpr int kBK = 64;   // bf16 per 128-byte smem row
constexpr int kAHalfBytes = kBM * kBK * 2;  // A of one 128-row half for one k-block
constexpr int kProducerWarps = 4;
constexpr int kEpilogueWarps = 4;
constexpr int kMmaWarp = kProducerWarps + kEpilogueWarps;
constexpr int kIndexWarp = kMmaWarp + 1;
constexpr int kWeightWarp = kIndexWarp + 1;
// Two-half items have a second index warp (half 1 of every tap table): one
// warp resolving 2 x 128 rows x L slots per item fell behind the producers
// (dense layer at L = 12: the table took ~12.7 us per item against 6.3 us of
// gathers). One-half items launch without it.
constexpr int kIndexWarp2 = kWeightWarp + 1;
template <int TM>
constexpr int kThreadsFor = (TM == 2 ? kIndexWarp2 + 1 : kWeightWarp + 1) * 32;
constexpr int kTabChunk = 6;  // spiral slots resolved per pass of the index warp
constexpr size_t kSmemLimit = 227 * 1024;  // opt-in dynamic shared memory per CTA

// BN output channels per tile; TM 128-row halves per work item, all sharing
// every W stage.
template <int BN, int TM>
struct Cfg {
    static_assert(BN == 64 || BN == 128, "tile widths");
    static_assert(TM == 1 || TM == 2, "halves per item");
    static constexpr int kTabRows = TM * kBM;  // rows of a tap table
    static constexpr int kAStageBytes = TM * kAHalfBytes;
    static constexpr int kBStageBytes = kBK * BN * 2;
    // Pipeline depth: as many stages as fit next to the tap tables (which
    // grow with L), between kMinStages and kMaxStages.
    static constexpr int kMaxStages = TM == 2 ? (BN == 64 ? 5 : 4) : (BN == 64 ? 8 : 6);
    static constexpr int kMinStages = 2;
    // two accumulator sets, each one BN-column accumulator per half
    static constexpr int kTmemCols = 2 * TM * BN;
    // Instruction descriptor, kind::f16: D fp32 (bit 4), A bf16 (bits 7-9 = 1),
    // B bf16 (bits 10-12 = 1), A K-major (bit 15 = 0), B MN-major (bit 16 = 1),
    // N >> 3 at bits 17-22, M >> 4 at bits 24-28.
    static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 16) |
                                       ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
    static constexpr int kBarBytes = 8 * (2 * kMaxStages + 9);
    // barriers, then 16 bytes (TMEM address, abort flag), then the two tap
    // tables ([L][kTabRows] int32 each) at a 128-byte boundary.
    static constexpr int kTabOffset = (kBarBytes + 16 + 127) / 128 * 128;
    // After the tables: one 2 KB staging buffer per epilogue warp (32 rows x
    // 64 bytes of bf16 output).
    static constexpr int kEpiBytes = kEpilogueWarps * 32 * 64;
    static size_t smem_bytes(int L, int stages) {
        return 1024 + (size_t)stages * (kAStageBytes + kBStageBytes) + kTabOffset +
               2 * sizeof(int) * (size_t)kTabRows * L + kEpiBytes;
    }
    static int stages_for(int L) {
        int st = kMaxStages;
        while (st > kMinStages && smem_bytes(L, st) > kSmemLimit) --st;
        return st;
    }
};

// Shared-memory matrix descriptor: start address, leading and stride byte
// offsets (>> 4), fixed version bits 46-48 = 0b001, 128-byte swizzle (2 at
// bits 61-63), base offset 0 (stage buffers are 1024-byte aligned).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(lbo >> 4) << 16) |
           ((uint64_t)(sbo >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// Epilogue of one 32-column chunk of a warp's 32 output rows: activation,
// bf16 rounding (RNE), then the stores. Lane i holds row i's 32 fp32 sums
// (bias included) in r. The rows go through a 2 KB shared buffer (16-byte
// pieces XOR-swizzled by row so that neither the writes nor the reads have
// bank conflicts) and leave it so that each store instruction writes eight
// rows x 64 contiguous bytes, instead of 32 scattered 16-byte pieces. Each
// row goes to its compact position and to its dense position of the fused
// scatter: lane i stores rows 8k + i/4 (k = 0..3), whose addresses it holds
// in yk[k] and dk[k] (0 = not written).
// Activation and bf16 rounding of a chunk: p[h] holds columns 2h (low
// half) and 2h + 1 (high half).

// Transposed epilogue chunk: lane = output channel, r[j] = row j of the
// chunk; activation, bf16, written transposed into the warp's staging
// buffer ([32 rows][32 channels] bf16). Rows j and j + 1 of the lane's
// channel are rounded as one bf16 pair; neighbouring lanes swap pairs and
// each builds one 32-bit word of two channels with a byte permute, the even
// lane for row j, the odd lane for row j + 1. Each store then writes two
// whole 64-byte rows (16-bit stores of two lanes into one word took two
// shared-memory wavefronts each).
template <int ACT>
__device__ __forceinline__ void tr_stage(const uint32_t (&r)[32], uint32_t stage, int lane) {
    const uint32_t odd = (uint32_t)lane & 1u;
    // even lane: its row-j half, then the neighbour's; odd lane: the
    // neighbour's row-(j+1) half, then its own
    const uint32_t sel = odd ? 0x3276u : 0x5410u;
    const uint32_t col = stage + (uint32_t)(lane & ~1) * 2u + odd * 64u;
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
        const __nv_bfloat162 b = __floats2bfloat162_rn(act_fixed<ACT>(__uint_as_float(r[j])),
                                                       act_fixed<ACT>(__uint_as_float(r[j + 1])));
        const uint32_t own = *reinterpret_cast<const uint32_t*>(&b);
        const uint32_t nb = __shfl_xor_sync(0xffffffffu, own, 1);
        uint32_t w;
        asm("prmt.b32 %0, %1, %2, %3;\n" : "=r"(w) : "r"(own), "r"(nb), "r"(sel));
        asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(col + (uint32_t)(j * 64)), "r"(w)
                     : "memory");
    }
}

template <int ACT>
__device__ __forceinline__ void epilogue_pack(const uint32_t (&r)[32], uint32_t (&p)[16]) {
#pragma unroll
    for (int h = 0; h < 16; ++h) {
        const __nv_bfloat162 b = __floats2bfloat162_rn(act_fixed<ACT>(__uint_as_float(r[2 * h])),
                                                       act_fixed<ACT>(__uint_as_float(r[2 * h + 1])));
        p[h] = *reinterpret_cast<const uint32_t*>(&b);
    }
}

__device__ __forceinline__ void epilogue_store(const uint32_t (&p)[16], uint32_t stage, int lane,
                                               const long long (&yk)[4], const long long (&dk)[4],
                                               int col0, int C_out) {
#pragma unroll
    for (int j8 = 0; j8 < 4; ++j8)
        sts_v4(stage + (uint32_t)(lane * 64 + ((j8 ^ ((lane >> 1) & 3)) << 4)),
               make_uint4(p[4 * j8], p[4 * j8 + 1], p[4 * j8 + 2], p[4 * j8 + 3]));
    __syncwarp();
    // all four shared-memory reads first, then the stores (the reads do not
    // wait behind the previous row group's stores)
    uint4 v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int R = 8 * k + (lane >> 2), piece = lane & 3;
        v[k] = lds_u4(stage + (uint32_t)(R * 64 + ((piece ^ ((R >> 1) & 3)) << 4)));
    }
    const int col = col0 + (lane & 3) * 8;
    if (col < C_out) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (yk[k]) *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(yk[k]) + col) = v[k];
            if (dk[k]) *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(dk[k]) + col) = v[k];
        }
    }
    __syncwarp();  // the buffer is reused by the next chunk
}

template <int ACT>
__device__ __forceinline__ void epilogue_chunk(const uint32_t (&r)[32], uint32_t stage, int lane,
                                               const long long (&yk)[4], const long long (&dk)[4],
                                               int col0, int C_out) {
    uint32_t p[16];
    epilogue_pack<ACT>(r, p);
    epilogue_store(p, stage, lane, yk, dk, col0, C_out);
}

// Group-norm statistics of one warp's 32 rows (lane = row). Every lane
// holds, per channel group, the mean and M2 of its CPG values of the group;
// the warp writes one (count, mean, M2) per frame present to slot (frame +
// block) of the partials, for NG groups g0 .. g0 + ng - 1 at once.

// Column j of a packed chunk (bf16 pairs, column 2h in the low half of
// p[h]) as fp32.
__device__ __forceinline__ float bf_col(const uint32_t (&p)[16], int j) {
    return __uint_as_float((j & 1) ? (p[j >> 1] & 0xffff0000u) : (p[j >> 1] << 16));
}

// Sum of N consecutive columns j0 .. (squared deviations from m when Sq) by
// a pairwise tree: log2 N levels of independent additions. j0 is known at
// compile time after unrolling (the values stay in registers).
template <int N, bool Sq>
__device__ __forceinline__ float tree_sum(const uint32_t (&p)[16], int j0, float m = 0.f) {
    float t[N];
#pragma unroll
    for (int i = 0; i < N; ++i) {
        const float x = bf_col(p, j0 + i);
        t[i] = Sq ? (x - m) * (x - m) : x;
    }
#pragma unroll
    for (int w = N / 2; w >= 1; w /= 2)
#pragma unroll
        for (int i = 0; i < w; ++i) t[i] += t[i + w];
    return t[0];
}

// All 32 rows active and in frame fb (most blocks): the lanes hold equal
// counts, so every butterfly level merges two halves of equal size n by the
// pairwise update of Chan, Golub and LeVeque: mean = (mean_a + mean_b) / 2,
// M2 = M2_a + M2_b + d^2 n / 2. Both partners of a level compute the same
// values (the operations are symmetric in a and b).
template <int NG>
__device__ __forceinline__ void gn_flush_whole(const ConvArgs& a, long long block, int fb, int g0,
                                               int ng, float n, float (&mean)[NG],
                                               float (&m2)[NG], int lane) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
#pragma unroll
        for (int q = 0; q < NG; ++q) {
            const float mb = __shfl_xor_sync(0xffffffffu, mean[q], o);
            const float qb = __shfl_xor_sync(0xffffffffu, m2[q], o);
            const float d = mb - mean[q];
            m2[q] = (m2[q] + qb) + d * d * (0.5f * n);
            mean[q] = (mean[q] + mb) * 0.5f;
        }
        n *= 2.f;
    }
    if (lane == 0) {
#pragma unroll
        for (int q = 0; q < NG; ++q)
            if (q < ng)
                *reinterpret_cast<float4*>(a.gn_part + 4 * ((fb + block) * a.gn_G + g0 + q)) =
                    make_float4(n, mean[q], m2[q], 0.f);
    }
}

// Rows of a block that straddles a frame boundary or the last active row
// (gn_b = the lane's frame, -1 past the active rows): no merge across lanes;
// every active row stores its own (mean, M2) of group g to the per-row
// partials (row * G + g), and the normalising pass merges them with the
// frame's whole blocks.
__device__ __forceinline__ void gn_store_row(const ConvArgs& a, long long row, int gn_b, int g,
                                             float mean, float m2) {
    if (gn_b >= 0)
        *reinterpret_cast<float2*>(a.gn_rows + 2 * (row * a.gn_G + g)) = make_float2(mean, m2);
}

// Statistics of one 32-column chunk (columns col0 .. col0 + 31) as stored
// (v: the packed bf16 values) for groups of CPG <= 32 channels, which lie
// inside the chunk and are flushed at once. whole: all 32 rows active and
// in one frame.
template <int CPG>
__device__ __forceinline__ void gn_chunk(const ConvArgs& a, const uint32_t (&v)[16], int col0,
                                         long long block, int gn_b, bool whole, int lane) {
    // the chunk's 32 / CPG groups, two at a time (register pressure)
    constexpr int NG = 32 / CPG, NB = NG < 2 ? NG : 2;
    // C_out is a multiple of CPG: the groups in range are whole
    const int ng = (a.C_out - col0) / CPG < NG ? (a.C_out - col0) / CPG : NG;
#pragma unroll
    for (int q0 = 0; q0 < NG; q0 += NB) {
        if (q0 >= ng) break;
        float mean[NB], m2[NB];
#pragma unroll
        for (int q = 0; q < NB; ++q) {
            mean[q] = tree_sum<CPG, false>(v, (q0 + q) * CPG) * (1.f / CPG);
            m2[q] = tree_sum<CPG, true>(v, (q0 + q) * CPG, mean[q]);
        }
        const int g0 = col0 / CPG + q0, nb = ng - q0 < NB ? ng - q0 : NB;
        if (whole)
            gn_flush_whole<NB>(a, block, gn_b, g0, nb, (float)CPG, mean, m2, lane);
        else
#pragma unroll
            for (int q = 0; q < NB; ++q)
                if (q < nb) gn_store_row(a, block * 32 + lane, gn_b, g0 + q, mean[q], m2[q]);
    }
}

// The same for groups of cpg = 64 or 128 channels: merged over their chunks
// in (run_mean, run_m2) and flushed by their last chunk.
__device__ __forceinline__ void gn_chunk_wide(const ConvArgs& a, const uint32_t (&v)[16], int col0,
                                              int cpg, long long block, int gn_b, bool whole,
                                              int lane, float& run_mean, float& run_m2) {
    const float mean = tree_sum<32, false>(v, 0) * (1.f / 32.f);
    const float m2 = tree_sum<32, true>(v, 0, mean);
    // chunk k (from 0) of the group joins 32 values to the 32 k before it:
    // the pairwise update with n_a = 32 k, n_b = 32
    const int k = (col0 & (cpg - 1)) >> 5;
    if (k == 0) {
        run_mean = mean, run_m2 = m2;
    } else {
        const float na = 32.f * k, rr = 1.f / (float)(k + 1), d = mean - run_mean;
        run_mean = fmaf(d, rr, run_mean);
        run_m2 += m2 + d * d * na * rr;
    }
    if (((col0 + 32) & (cpg - 1)) == 0) {
        float m1[1] = {run_mean}, q1[1] = {run_m2};
        const int g = col0 / cpg;
        if (whole)
            gn_flush_whole<1>(a, block, gn_b, g, 1, (float)cpg, m1, q1, lane);
        else
            gn_store_row(a, block * 32 + lane, gn_b, g, run_mean, run_m2);
    }
}

// The statistics of a chunk for the group width of the call (a power of two
// from 8 to 128, checked by the launcher), from the values as stored (v:
// packed bf16).
__device__ __forceinline__ void gn_stats_chunk(const ConvArgs& a, const uint32_t (&v)[16],
                                               int col0, long long block, int gn_b, bool whole,
                                               int lane, float& run_mean, float& run_m2) {
    switch (a.gn_cpg) {
        case 8: gn_chunk<8>(a, v, col0, block, gn_b, whole, lane); break;
        case 16: gn_chunk<16>(a, v, col0, block, gn_b, whole, lane); break;
        case 32: gn_chunk<32>(a, v, col0, block, gn_b, whole, lane); break;
        default:
            gn_chunk_wide(a, v, col0, a.gn_cpg, block, gn_b, whole, lane, run_mean, run_m2);
            break;
    }
}

// Where a kernel's barriers sit, as indices of 8-byte slots from the start of
// its barrier block, where its tap tables start (bytes from that block) and
// how many rows each table has room for. Compile-time, so that every
// barrier and table address is the block's address plus an immediate.
template <int kFull_, int kEmpty_, int kTfull_, int kTempty_, int kFin_, int kTabfull_,
          int kTabempty_, int kTabOffset_, int kTabRoom_>
struct BarSlots {
    static constexpr int kFull = kFull_, kEmpty = kEmpty_, kTfull = kTfull_, kTempty = kTempty_,
                         kFin = kFin_, kTabfull = kTabfull_, kTabempty = kTabempty_,
                         kTabOffset = kTabOffset_, kTabRoom = kTabRoom_;
};
// conv_tc_kernel's block: full and empty per stage (kMaxStages each), the two
// accumulator pairs, fin, the table pairs.
template <class C>
using RingSlots = BarSlots<0, C::kMaxStages, 2 * C::kMaxStages, 2 * C::kMaxStages + 2,
                           2 * C::kMaxStages + 4, 2 * C::kMaxStages + 5, 2 * C::kMaxStages + 7,
                           C::kTabOffset, C::kTabRows>;

// Run-time part of a launch's shared memory and TMEM.
struct ConvSmem {
    uint32_t ring;             // stage s at ring + s * (A bytes + W bytes)
    int nst;                   // stages in the ring
    uint32_t bars;             // the barrier block
    volatile int* abort_flag;  // set by the first role that gives up
    uint32_t tmem_base;
};

// The five roles of a launch on TM-half items of BN channels (after the
// prologue: barriers initialised, TMEM allocated, launch dependency
// passed). The arguments come by value: read through a reference to the
// kernel parameter, the layers ran up to 14% slower. `prefetched`: this thread (the index warp) has already copied
// the first item's rulebook entries into tap table 0, completing
// tabfull(0) through the copies.
template <int BN, int TM, bool TR, class S>
__device__ __forceinline__ void conv_roles(const ConvArgs a, const CUtensorMap& tmap_w,
                                           const ConvSmem& sm, const long long rows,
                                           const bool prefetched) {
    using C = Cfg<BN, TM>;
    static_assert(!TR || (TM == 2 && BN == 128), "the transposed MMA takes 2 x 128 rows, 128 channels");
    // transposed MMA: D fp32, A (W) bf16 MN-major (bit 15), B (rows) bf16
    // K-major, N = 256 at bits 17-22, M = 128 at bits 24-28
    constexpr uint32_t kIdescTR = (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) |
                                  ((uint32_t)(256 >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
    constexpr int kTabRows = C::kTabRows;
    constexpr uint32_t kStageBytes = C::kAStageBytes + C::kBStageBytes;
    const int nst = sm.nst;
    // stage st: TM halves of A (16 KB each), then the W slice (1024-byte aligned)
    auto a_stage = [&](int st) { return sm.ring + (uint32_t)st * kStageBytes; };
    auto b_stage = [&](int st) {
        return sm.ring + (uint32_t)st * kStageBytes + (uint32_t)C::kAStageBytes;
    };
    const uint32_t sBar = sm.bars;
    auto full_bar = [&](int s) { return sBar + 8u * (S::kFull + s); };
    auto empty_bar = [&](int s) { return sBar + 8u * (S::kEmpty + s); };
    auto tfull_bar = [&](int i) { return sBar + 8u * (S::kTfull + i); };
    auto tempty_bar = [&](int i) { return sBar + 8u * (S::kTempty + i); };
    const uint32_t fin_bar = sBar + 8u * S::kFin;
    auto tabfull_bar = [&](int i) { return sBar + 8u * (S::kTabfull + i); };
    auto tabempty_bar = [&](int i) { return sBar + 8u * (S::kTabempty + i); };
    volatile int* const abort_flag = sm.abort_flag;
    const uint32_t tmem_base = sm.tmem_base;
    // Tap tables, [2][L][TM * 128] int32 (room for [2][L][kTabRoom]): entry
    // (l, r) is the input row feeding slot l of row r of the work item, or
    // -1; then the epilogue staging.
    static_assert(S::kTabRoom >= kTabRows, "tap table room");
    const uint32_t tab0 = sBar + S::kTabOffset;
    const uint32_t epi0 = tab0 + 2u * (uint32_t)(S::kTabRoom * a.L) * 4u;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int n_tiles = (a.C_out + BN - 1) / BN;
    constexpr int item_rows = TM * kBM;
    const long long m_items = (rows + item_rows - 1) / item_rows;
    const long long work_total = m_items * n_tiles;
    const int num_kb = (a.K + kBK - 1) / kBK;
    const int L = a.L, C_in = a.C_in, C_out = a.C_out, K = a.K;
    const uint32_t tab_bytes = (uint32_t)(kTabRows * L) * 4u;

    if (warp < kProducerWarps) {
        // ------------------------------------------------------------ producers
        // A is gathered by all 128 producer threads with 16-byte cp.async
        // (row r of the stage at r*128 bytes, chunk q at q ^ (r % 8)), whose
        // completion each thread signals on the stage's "full" barrier
        // without blocking (cp.async.mbarrier.arrive.noinc).
        const __nv_bfloat16* __restrict__ x = static_cast<const __nv_bfloat16*>(a.x);
        const int t = threadIdx.x;  // 0..127
        const int q = t & 7;        // 16-byte chunk of the 128-byte row
        const unsigned xr = (unsigned)a.x_rows;
        int st_s = 0;        // stage of the current iteration (it % stages)
        uint32_t st_ph = 0;  // its phase parity ((it / stages) & 1)
        int lt = 0;
        bool ok = true;
        for (long long w = blockIdx.x; w < work_total && ok; w += gridDim.x, ++lt) {
            const int buf = lt & 1;
            if (!mbar_wait(tabfull_bar(buf), (uint32_t)((lt >> 1) & 1), abort_flag, a.status)) {
                ok = false;
                break;
            }
            const uint32_t tab_s = tab0 + (uint32_t)buf * tab_bytes;
            int l = (q * 8) / C_in;  // slot and channel of this thread's chunk at k-block 0
            int c = q * 8 - l * C_in;
            for (int kb = 0; kb < num_kb; ++kb) {
                const int s = st_s;
                const uint32_t ph = st_ph;
                if (!mbar_wait(empty_bar(s), ph ^ 1u, abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                const bool kval = kb * kBK + q * 8 < K;
                {
                    // All table entries first, then the copies: half h's 128
                    // rows at a_stage + h * 16 KB, its entries at table rows
                    // h * 128 ..
                    int src[TM][8];
#pragma unroll
                    for (int h = 0; h < TM; ++h)
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int r = h * kBM + (t >> 3) + 16 * i;
                            src[h][i] = kval ? lds_s32(tab_s + (uint32_t)(l * kTabRows + r) * 4u)
                                             : -1;
                        }
#pragma unroll
                    for (int h = 0; h < TM; ++h)
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int r = (t >> 3) + 16 * i;
                            const bool in_x = (unsigned)src[h][i] < xr;  // -1: absent tap
                            const __nv_bfloat16* gp =
                                x + (in_x ? (long long)src[h][i] * C_in + c : 0);
                            cp_async_16(a_stage(s) + h * kAHalfBytes + r * 128 +
                                            ((q ^ (r & 7)) << 4),
                                        gp, in_x);
                        }
                }
                cp_async_arrive_noinc(full_bar(s));
                if (++st_s == nst) {
                    st_s = 0;
                    st_ph ^= 1u;
                }
                c += kBK;
                while (c >= C_in) {
                    c -= C_in;
                    ++l;
                }
            }
            // Addresses of this tile's copies are issued: the table is free.
            if (ok) mbar_arrive(tabempty_bar(buf));
        }
        cp_async_wait_all();
    } else if (warp == kWeightWarp) {
        // ------------------------------------------------------------ weight loader
        if (lane == 0) {
            constexpr uint32_t kWBytes = (uint32_t)(BN / 64) * (kBK * 128u);
            long long it = 0;
            int st_s = 0;
            uint32_t st_ph = 0;
            bool ok = true;
            for (long long w = blockIdx.x; w < work_total && ok; w += gridDim.x) {
                const int n0 = ((int)w % n_tiles) * BN;  // w < 2^31
                for (int kb = 0; kb < num_kb; ++kb) {
                    const int s = st_s;
                    if (!mbar_wait(empty_bar(s), st_ph ^ 1u, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(full_bar(s), kWBytes);
                    if (a.w3d) {
                        // both 64-column blocks of the slice in one copy
                        tma_load_3d(b_stage(s), &tmap_w, 0, kb * kBK, n0 / 64,
                                    full_bar(s));
                    } else {
#pragma unroll
                        for (int nb = 0; nb < BN / 64; ++nb)
                            tma_load_2d(b_stage(s) + nb * (kBK * 128), &tmap_w,
                                        n0 + nb * 64, kb * kBK, full_bar(s));
                    }
                    ++it;
                    if (++st_s == nst) {
                        st_s = 0;
                        st_ph ^= 1u;
                    }
                }
            }
            if (!ok) {
                // Let the weight copies already issued land before the CTA
                // exits (bounded: the full barriers also count the gather
                // threads' arrivals, which an unwinding producer may not make).
                for (long long j = it > nst ? it - nst : 0; j < it; ++j)
                    mbar_wait_drain(full_bar((int)(j % nst)), (uint32_t)((j / nst) & 1), a.status);
            }
        }
        __syncwarp();
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            long long it = 0;
            int st_s = 0;        // stage of iteration it (it % stages)
            uint32_t st_ph = 0;  // its phase parity ((it / stages) & 1)
            int lt = 0;
            bool ok = true;
            const bool has_bias = a.bias != nullptr;  // accumulators start at the bias
            for (long long w = blockIdx.x; w < work_total && ok; w += gridDim.x, ++lt) {
                const int acc = lt & 1;
                const uint32_t acc_ph = (uint32_t)((lt >> 1) & 1);
                // released by the epilogue once it holds the bias (or is free)
                if (!mbar_wait(tempty_bar(acc), acc_ph, abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // accumulator of half h: columns (acc * TM + h) * BN
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * TM * BN);
                for (int kb = 0; kb < num_kb; ++kb) {
                    const int s = st_s;
                    const uint32_t ph = st_ph;
                    if (!mbar_wait(full_bar(s), ph, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // The A operand was written by cp.async (generic proxy):
                    // order it before the tensor core's async-proxy reads.
                    fence_proxy_async_smem();
                    const uint32_t a_st = a_stage(s);
                    const uint32_t b_st = b_stage(s);
                    if constexpr (TR) {
                        // A operand: the W slice (MN-major, M = 128 output
                        // channels); B operand: the item's 256 gathered rows
                        // (K-major, N = 256, both halves contiguous)
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t wd =
                                smem_desc_sw128(b_st + k * 16 * 128, kBK * 128, 1024);
                            const uint64_t rd = smem_desc_sw128(a_st + k * 32, 16, 1024);
                            const uint32_t acc_in = (has_bias || (kb | k) != 0) ? 1u : 0u;
                            tc_mma_bf16(d_tmem, wd, rd, kIdescTR, acc_in);
                        }
                    } else {
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t bd =
                                smem_desc_sw128(b_st + k * 16 * 128, kBK * 128, 1024);
                            const uint32_t acc_in = (has_bias || (kb | k) != 0) ? 1u : 0u;
#pragma unroll
                            for (int h = 0; h < TM; ++h) {
                                const uint64_t ad =
                                    smem_desc_sw128(a_st + h * kAHalfBytes + k * 32, 16, 1024);
                                tc_mma_bf16(d_tmem + (uint32_t)(h * BN), ad, bd, C::kIdesc,
                                            acc_in);
                            }
                        }
                    }
                    tc_commit(empty_bar(s));
                    ++it;
                    if (++st_s == nst) {
                        st_s = 0;
                        st_ph ^= 1u;
                    }
                }
                if (!ok) break;
                tc_commit(tfull_bar(acc));
            }
            // Every MMA issued by this thread has completed once fin_bar fires.
            tc_commit(fin_bar);
            mbar_wait_drain(fin_bar, 0, a.status);
        }
        __syncwarp();
    } else if (warp == kIndexWarp || (TM == 2 && warp == kIndexWarp2)) {
        // two-half items: kIndexWarp builds half 0 of every table, kIndexWarp2 half 1
        const int h_lo = warp == kIndexWarp ? 0 : 1;
        const int h_hi = TM == 2 ? h_lo + 1 : 1;
        // ------------------------------------------------------------ index warp
        // Lane handles rows lane + 32*i (i < 4) of the tile. Phase 1 loads the
        // coordinates, phase 2 all spiral entries of a chunk of slots, phase 3
        // all row_of lookups of that chunk. Loads are issued from clamped,
        // always-valid addresses and checked afterwards, so that every load
        // of a phase is in flight at once.
        int lt = 0;
        for (long long w = blockIdx.x; w < work_total; w += gridDim.x, ++lt) {
            const int buf = lt & 1;
            if (!mbar_wait(tabempty_bar(buf), (uint32_t)(((lt >> 1) & 1) ^ 1), abort_flag,
                           a.status))
                break;
            const long long m_item = (long long)((int)w / n_tiles) * item_rows;
            unsigned err = 0;
            for (int h = h_lo; h < h_hi; ++h) {
            // half h: rows m0 .. m0 + 127, table entries (l, r) at tab_s + (l * kTabRows + r) * 4
            const long long m0 = m_item + h * kBM;
            const uint32_t tab_s = tab0 + (uint32_t)buf * tab_bytes + (uint32_t)(h * kBM) * 4u;
            if (a.mode == kRulebook) {
                // Precomputed mapping: one coalesced pass over the tile's
                // rulebook columns, entries checked against the input's rows
                // (the first tile's table may have been filled before the loop).
                long long col[4];
                bool live[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const long long p = m0 + lane + 32 * i;
                    live[i] = p < rows;
                    col[i] = live[i] ? p : 0;
                }
                constexpr int kRbChunk = 12;
                if (lt == 0 && prefetched) {
                    // the prefetched table, already with the producers:
                    // report its bad entries (the producers skip them)
                    cp_async_wait_all();
                    for (int d = 0; d < L; ++d)
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const int ev = lds_s32(tab_s + (uint32_t)(d * kTabRows + lane + 32 * i) * 4u);
                            if (live[i] && (ev < -1 || ev >= a.x_rows)) err |= kErrIndex;
                        }
                }
                for (int l0 = 0; l0 < L && !(lt == 0 && prefetched); l0 += kRbChunk) {
                    int e[4][kRbChunk];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int d = 0; d < kRbChunk; ++d) {
                            const int lc = l0 + d < L ? l0 + d : L - 1;
                            e[i][d] = __ldg(a.rulebook + (long long)lc * a.capacity + col[i]);
                        }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int d = 0; d < kRbChunk; ++d) {
                            if (l0 + d >= L) continue;
                            const int ev = e[i][d];
                            int src = -1;
                            if (live[i]) {
                                if (ev < -1 || ev >= a.x_rows) err |= kErrIndex;
                                else src = ev;
                            }
                            sts_s32(tab_s + (uint32_t)((l0 + d) * kTabRows + lane + 32 * i) * 4u, src);
                        }
                }
                continue;
            }
            int bb[4], vv[4];
            bool ok[4];
            const bool sparse = a.mode == kSparseDenseX || a.mode == kSparseCompactX;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const long long n = m0 + lane + 32 * i;
                const long long nn = n < rows ? n : 0;
                if (sparse) {
                    bb[i] = __ldg(a.coords + 2 * nn);
                    vv[i] = __ldg(a.coords + 2 * nn + 1);
                } else if (a.mode == kDense) {
                    bb[i] = (int)(nn / a.V);
                    vv[i] = (int)(nn - (long long)bb[i] * a.V);
                } else {
                    bb[i] = 0;
                    vv[i] = 0;
                }
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const long long n = m0 + lane + 32 * i;
                const bool in_range = bb[i] >= 0 && bb[i] < a.B && vv[i] >= 0 && vv[i] < a.V;
                ok[i] = n < rows && in_range;
                if (n < rows && !in_range) err |= kErrIndex;
                if (!ok[i]) {
                    bb[i] = 0;
                    vv[i] = 0;
                }
            }
            if (a.mode == kLinear) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    sts_s32(tab_s + (uint32_t)(lane + 32 * i) * 4u,
                            ok[i] ? (int)(m0 + lane + 32 * i) : -1);
            } else {
                for (int l0 = 0; l0 < L; l0 += kTabChunk) {
                    int u[4][kTabChunk];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int d = 0; d < kTabChunk; ++d) {
                            const int lc = l0 + d < L ? l0 + d : L - 1;
                            u[i][d] = __ldg(a.spiral + (long long)vv[i] * L + lc);
                        }
                    int dr[4][kTabChunk];  // dense row b*V + u (< 2^31), or -1
                    int j[4][kTabChunk];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int d = 0; d < kTabChunk; ++d) {
                            const int uu = u[i][d];
                            const bool live = ok[i] && l0 + d < L;
                            if (live && (uu < -1 || uu >= a.V)) err |= kErrIndex;
                            const bool tap = live && uu >= 0 && uu < a.V;
                            dr[i][d] = tap ? bb[i] * a.V + uu : -1;
                        }
                    if (sparse) {
#pragma unroll
                        for (int i = 0; i < 4; ++i)
#pragma unroll
                            for (int d = 0; d < kTabChunk; ++d)
                                j[i][d] = __ldg(a.row_of + (dr[i][d] >= 0 ? dr[i][d] : 0));
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
#pragma unroll
                        for (int d = 0; d < kTabChunk; ++d) {
                            if (l0 + d >= L) continue;
                            int src = -1;
                            if (dr[i][d] >= 0) {
                                if (!sparse) {
                                    src = dr[i][d];
                                } else {
                                    const int jj = j[i][d];
                                    if (jj < -1 || jj >= rows) err |= kErrIndex;
                                    if (jj >= 0 && jj < rows)
                                        src = a.mode == kSparseDenseX ? dr[i][d] : jj;
                                }
                            }
                            sts_s32(tab_s + (uint32_t)((l0 + d) * kTabRows + lane + 32 * i) * 4u, src);
                        }
                }
            }
            }  // halves
            if (err) report(a.status, err);
            if (!(lt == 0 && prefetched)) mbar_arrive(tabfull_bar(buf));  // else the copies did
        }
        if (prefetched) cp_async_wait_all();  // a CTA without items
    } else if (warp < kMmaWarp) {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - kProducerWarps;  // == warp % 4: TMEM lanes 32*ew..+32
        __nv_bfloat16* __restrict__ y = static_cast<__nv_bfloat16*>(a.y);
        if constexpr (TR) {
        // TMEM lane = output channel 32*ew + lane, column = row of the item
        const uint32_t t_lane = tmem_base + ((uint32_t)(ew * 32) << 16);
        auto release_tr = [&](int acc, long long w) {
            if (a.bias && w < work_total) {
                const uint32_t bv = __float_as_uint(__ldg(a.bias + 32 * ew + lane));
                uint32_t r[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) r[j] = bv;
#pragma unroll 1
                for (int cb = 0; cb < 8; ++cb)
                    tmem_st_32x32b_x32(t_lane + (uint32_t)(acc * 256 + cb * 32), r);
                tmem_st_wait();
            }
            tc_fence_before();
            mbar_arrive(tempty_bar(acc));
        };
        release_tr(0, blockIdx.x);
        release_tr(1, blockIdx.x + (long long)gridDim.x);
        const uint32_t stage = epi0 + (uint32_t)ew * 2048u;
        int lt = 0;
        for (long long w = blockIdx.x; w < work_total; w += gridDim.x, ++lt) {
            const long long m_item = (long long)((int)w / n_tiles) * item_rows;
            const int acc = lt & 1;
            if (!mbar_wait(tfull_bar(acc), (uint32_t)((lt >> 1) & 1), abort_flag, a.status)) break;
            tc_fence_after();
#pragma unroll 1
            for (int cb = 0; cb < 8; ++cb) {
                uint32_t r[32];
                tmem_ld_32x32b_x32(t_lane + (uint32_t)(acc * 256 + cb * 32), r);
                tmem_ld_wait();
                if (a.act == HC_ACT_ELU) tr_stage<HC_ACT_ELU>(r, stage, lane);
                else if (a.act == HC_ACT_RELU) tr_stage<HC_ACT_RELU>(r, stage, lane);
                else tr_stage<HC_ACT_NONE>(r, stage, lane);
                __syncwarp();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int j = (lane >> 2) + 8 * q, p = lane & 3;
                    const uint4 v = lds_u4(stage + (uint32_t)(j * 64 + p * 16));
                    const long long row = m_item + cb * 32 + j;
                    if (y && row < rows)
                        *reinterpret_cast<uint4*>(y + row * C_out + 32 * ew + 8 * p) = v;
                }
                __syncwarp();
            }
            release_tr(acc, w + 2 * (long long)gridDim.x);
        }
        } else {
        // Accumulator buffer acc is handed to the MMA warp holding the bias of
        // tile w in every row (the MMAs then accumulate onto it), so the bias
        // costs the epilogue nothing once the sums are ready.
        auto release = [&](int acc, long long w) {
            if (a.bias && w < work_total) {
                const int n0 = ((int)w % n_tiles) * BN;
#pragma unroll 1
                for (int cb = 0; cb < BN / 32; ++cb) {
                    uint32_t r[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col = n0 + cb * 32 + j;
                        r[j] = col < C_out ? __float_as_uint(__ldg(a.bias + col)) : 0u;
                    }
                    for (int h = 0; h < TM; ++h)
                        tmem_st_32x32b_x32(tmem_base + ((uint32_t)(ew * 32) << 16) +
                                               (uint32_t)((acc * TM + h) * BN + cb * 32),
                                           r);
                }
                tmem_st_wait();
            }
            tc_fence_before();
            mbar_arrive(tempty_bar(acc));
        };
        release(0, blockIdx.x);
        release(1, blockIdx.x + (long long)gridDim.x);
        int lt = 0;
        bool live = true;
        for (long long w = blockIdx.x; w < work_total && live; w += gridDim.x, ++lt) {
            const long long m_item = (long long)((int)w / n_tiles) * item_rows;
            const int n0 = ((int)w % n_tiles) * BN;  // w < 2^31
            const int acc = lt & 1;
            const uint32_t ph = (uint32_t)((lt >> 1) & 1);
            for (int h = 0; h < TM; ++h) {
            const long long m0 = m_item + h * kBM;
            // Everything that does not need the accumulator is loaded while
            // the main loop runs: this lane's row addresses (0 = not
            // written; the fused scatter's needs the row's coordinate).
            const long long row = m0 + ew * 32 + lane;
            const bool rvalid = row < rows;
            const long long row_y = (rvalid && y) ? (long long)(y + row * C_out) : 0;
            long long row_d = 0;
            if (rvalid && a.out_dense) {
                const int b = __ldg(a.out_coords + 2 * row), v = __ldg(a.out_coords + 2 * row + 1);
                if (b >= 0 && b < a.out_B && v >= 0 && v < a.out_V)
                    row_d = (long long)(static_cast<__nv_bfloat16*>(a.out_dense) +
                                        ((long long)b * a.out_V + v) * C_out);
                else
                    report(a.status, kErrIndex);
            }
            int gn_b = -1;  // frame of this lane's row, for the group-norm statistics
            if (a.gn_part && rvalid) {
                gn_b = __ldg(a.gn_coords + 2 * row);
                if (gn_b < 0 || gn_b >= a.gn_B) {
                    report(a.status, kErrIndex);
                    gn_b = -1;
                }
            }
            // all 32 rows of this warp active and in one frame
            const int gn_b0 = __shfl_sync(0xffffffffu, gn_b, 0);
            const bool gn_whole = __all_sync(0xffffffffu, gn_b >= 0 && gn_b == gn_b0);
            float run_mean = 0.f, run_m2 = 0.f;
            // the addresses of the rows this lane stores in every chunk
            long long yk[4], dk[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                yk[k] = __shfl_sync(0xffffffffu, row_y, 8 * k + (lane >> 2));
                dk[k] = __shfl_sync(0xffffffffu, row_d, 8 * k + (lane >> 2));
            }
            if (h == 0) {
                if (!mbar_wait(tfull_bar(acc), ph, abort_flag, a.status)) {
                    live = false;
                    break;
                }
                tc_fence_after();
            }
            const uint32_t stage = epi0 + (uint32_t)ew * 2048u;
            const uint32_t acc_col = (uint32_t)((acc * TM + h) * BN);
#pragma unroll 1
            for (int cb = 0; cb < BN / 32; ++cb) {
                uint32_t r[32];
                tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(ew * 32) << 16) + acc_col + (uint32_t)(cb * 32),
                                   r);
                tmem_ld_wait();
                const int col0 = n0 + cb * 32;
                if (a.gn_part) {
                    // with statistics the activation is the identity (it
                    // follows the normalisation)
                    uint32_t p[16];
                    epilogue_pack<HC_ACT_NONE>(r, p);
                    if (col0 < C_out)
                        gn_stats_chunk(a, p, col0, (m0 + ew * 32) / 32, gn_b, gn_whole, lane,
                                       run_mean, run_m2);
                    epilogue_store(p, stage, lane, yk, dk, col0, C_out);
                } else if (a.act == HC_ACT_ELU)
                    epilogue_chunk<HC_ACT_ELU>(r, stage, lane, yk, dk, col0, C_out);
                else if (a.act == HC_ACT_RELU)
                    epilogue_chunk<HC_ACT_RELU>(r, stage, lane, yk, dk, col0, C_out);
                else
                    epilogue_chunk<HC_ACT_NONE>(r, stage, lane, yk, dk, col0, C_out);
            }
            }  // halves
            if (!live) break;
            release(acc, w + 2 * (long long)gridDim.x);  // the item after next
        }
        }
    }
}

template <int BN, int TM, bool TR>
__global__ void __launch_bounds__(kThreadsFor<TM>, 1)
    conv_tc_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_w) {
    using C = Cfg<BN, TM>;
    constexpr int kTabRows = C::kTabRows;
    // "full": one cp.async completion arrival per producer thread, plus the
    // expect-tx arrival of the weight loader.
    constexpr int kStageArrivals = kProducerWarps * 32 + 1;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const base_ptr = smem_raw + (base - raw);
    const uint32_t sA = base;  // the stage ring (a.stages two-half stages)
    const int nst = a.stages;
    constexpr uint32_t kStageBytes = C::kAStageBytes + C::kBStageBytes;
    const uint32_t sBar = sA + (uint32_t)nst * kStageBytes;
    uint8_t* const misc = base_ptr + (sBar - base) + C::kBarBytes;
    volatile uint32_t* const tmem_holder = reinterpret_cast<volatile uint32_t*>(misc);
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(misc + 4);
    const uint32_t tab0 = sBar + C::kTabOffset;  // tap table 0

    auto full_bar = [&](int s) { return sBar + 8u * s; };
    auto empty_bar = [&](int s) { return sBar + 8u * (C::kMaxStages + s); };
    auto tfull_bar = [&](int i) { return sBar + 8u * (2 * C::kMaxStages + i); };
    auto tempty_bar = [&](int i) { return sBar + 8u * (2 * C::kMaxStages + 2 + i); };
    const uint32_t fin_bar = sBar + 8u * (2 * C::kMaxStages + 4);
    auto tabfull_bar = [&](int i) { return sBar + 8u * (2 * C::kMaxStages + 5 + i); };
    auto tabempty_bar = [&](int i) { return sBar + 8u * (2 * C::kMaxStages + 7 + i); };

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kMaxStages; ++s) {
            mbar_init(full_bar(s), kStageArrivals);
            mbar_init(empty_bar(s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(tfull_bar(i), 1);
            mbar_init(tempty_bar(i), kEpilogueWarps * 32);
        }
        mbar_init(fin_bar, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(tabfull_bar(i), 32 * TM);  // the index warps' lanes
            mbar_init(tabempty_bar(i), kProducerWarps * 32);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == kWeightWarp && lane == 0) prefetch_tensormap(&tmap_w);
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32((const void*)tmem_holder), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;
    // The prologue above touched only on-chip state; global memory written
    // by the previous grid is read from here on.
    pdl_wait();
    pdl_trigger();

    // Rulebook mode (one-half items): the index warp copies its first tile's
    // entries into tap table 0 (cp.async, rows clamped to the capacity,
    // always valid memory) before the row count arrives, so the two L2 round
    // trips overlap, and the copies themselves complete the table's "full"
    // barrier: the producers start on the entries as copied. They are not
    // checked first (a pass over them before the hand-over cost ~0.7 us of
    // the launch); the producers read zeros for any entry outside
    // [0, x_rows) (entries of rows past the count are never checked, and
    // those rows are never stored), and the index warp reports bad entries
    // of active rows once the table is handed over.
    const bool prefetch = TM == 1 && warp == kIndexWarp && a.mode == kRulebook;
    if (prefetch) {
        const long long m0p = (blockIdx.x / ((a.C_out + BN - 1) / BN)) * (long long)kBM;
        for (int d = 0; d < a.L; ++d)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const long long n = m0p + lane + 32 * i;
                cp_async_4(tab0 + (uint32_t)(d * kTabRows + lane + 32 * i) * 4u,
                           a.rulebook + (long long)d * a.capacity + (n < a.capacity ? n : 0), true);
            }
        cp_async_arrive_noinc(tabfull_bar(0));
    }

    const ConvSmem sm{sA, nst, sBar, abort_flag, tmem_base};
    conv_roles<BN, TM, TR, RingSlots<C>>(a, tmap_w, sm, active_rows(a), prefetch);
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::kTmemCols);
    }
}

// Shared memory of the row-count-dispatched kernel below: a ring as long as
// the larger of the one-half (32 KB) and two-half (48 KB) rings, one barrier
// block (full / empty for up to six stages, the accumulator, fin and
// table-empty barriers, and a table-full pair per half count), the tap
// tables sized for two-half items, and the epilogue staging.
struct AutoLayout {
    static constexpr int kRing1 = 6, kRing2 = 4;  // most stages per half count
    static constexpr int kFull = 0, kEmpty = 6, kTfull = 12, kTempty = 14, kFin = 16,
                         kTabfull1 = 17, kTabempty = 19, kTabfull2 = 21, kBars = 23;
    static constexpr int kTabOffset = (8 * kBars + 16 + 127) / 128 * 128;
    static constexpr int kStage1 = Cfg<128, 1>::kAStageBytes + Cfg<128, 1>::kBStageBytes;
    static constexpr int kStage2 = Cfg<128, 2>::kAStageBytes + Cfg<128, 2>::kBStageBytes;
    __host__ __device__ static size_t ring_bytes(int st1, int st2) {
        const size_t r1 = (size_t)st1 * kStage1, r2 = (size_t)st2 * kStage2;
        return r1 > r2 ? r1 : r2;
    }
    static size_t fixed_bytes(int L) {
        return 1024 + kTabOffset + 2 * sizeof(int) * (size_t)(2 * kBM) * L +
               Cfg<128, 2>::kEpiBytes;
    }
    static size_t smem_bytes(int L, int st1, int st2) { return fixed_bytes(L) + ring_bytes(st1, st2); }
    static void stages_for(int L, int& st1, int& st2) {
        const size_t avail = kSmemLimit - fixed_bytes(L);
        st1 = (int)(avail / kStage1 < (size_t)kRing1 ? avail / kStage1 : kRing1);
        st2 = (int)(avail / kStage2 < (size_t)kRing2 ? avail / kStage2 : kRing2);
    }
};

// 128-channel sparse calls (rulebook, or taps resolved from coords, spiral
// and row_of) whose row count is on the device: every CTA reads the count
// after the launch dependency and runs two-half transposed items when each
// CTA gets at least one (rows >= 256 per CTA), one-half items otherwise.
// Both role sets are compiled in and each branch is taken whole, so neither
// pays for the other in its loops. The one-half roles' rulebook-mode
// first-table prefetch (issued before the count is known) completes its own
// table-full pair; when the two-half roles run instead, the prefetching
// warp waits for those copies before the tables are rebuilt, and their
// arrival lands on barriers nothing waits on.
__global__ void __launch_bounds__(kThreadsFor<2>, 1)
    conv_tc_auto_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_w) {
    using L_ = AutoLayout;
    constexpr int kStageArrivals = kProducerWarps * 32 + 1;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const base_ptr = smem_raw + (base - raw);
    const uint32_t ring = (uint32_t)L_::ring_bytes(a.stages, a.stages_tr);
    const uint32_t sBar = base + ring;
    uint8_t* const misc = base_ptr + ring + 8 * L_::kBars;
    volatile uint32_t* const tmem_holder = reinterpret_cast<volatile uint32_t*>(misc);
    volatile int* const abort_flag = reinterpret_cast<volatile int*>(misc + 4);
    const uint32_t tab0 = sBar + L_::kTabOffset;  // the one-half roles' table 0
    auto bar = [&](int i) { return sBar + 8u * i; };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < L_::kRing1; ++s) {
            mbar_init(bar(L_::kFull + s), kStageArrivals);
            mbar_init(bar(L_::kEmpty + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(L_::kTfull + i), 1);
            mbar_init(bar(L_::kTempty + i), kEpilogueWarps * 32);
            mbar_init(bar(L_::kTabfull1 + i), 32);  // one index warp
            mbar_init(bar(L_::kTabempty + i), kProducerWarps * 32);
            mbar_init(bar(L_::kTabfull2 + i), 64);  // two index warps
        }
        mbar_init(bar(L_::kFin), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == kWeightWarp && lane == 0) prefetch_tensormap(&tmap_w);
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32((const void*)tmem_holder), Cfg<128, 2>::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;
    pdl_wait();
    pdl_trigger();

    // rulebook mode: the one-half roles' first table, copied while the row
    // count is read (as in conv_tc_kernel)
    const bool prefetch = warp == kIndexWarp && a.mode == kRulebook;
    if (prefetch) {
        const long long m0p = (long long)blockIdx.x * kBM;
        for (int d = 0; d < a.L; ++d)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const long long n = m0p + lane + 32 * i;
                cp_async_4(tab0 + (uint32_t)(d * kBM + lane + 32 * i) * 4u,
                           a.rulebook + (long long)d * a.capacity + (n < a.capacity ? n : 0), true);
            }
        cp_async_arrive_noinc(bar(L_::kTabfull1));
    }
    const long long rows = active_rows(a);
    using S1 = BarSlots<L_::kFull, L_::kEmpty, L_::kTfull, L_::kTempty, L_::kFin, L_::kTabfull1,
                        L_::kTabempty, L_::kTabOffset, 2 * kBM>;
    using S2 = BarSlots<L_::kFull, L_::kEmpty, L_::kTfull, L_::kTempty, L_::kFin, L_::kTabfull2,
                        L_::kTabempty, L_::kTabOffset, 2 * kBM>;
    if ((rows + 2 * kBM - 1) / (2 * kBM) >= (long long)gridDim.x) {
        if (prefetch) cp_async_wait_all();
        conv_roles<128, 2, true, S2>(a, tmap_w, ConvSmem{base, a.stages_tr, sBar, abort_flag, tmem_base},
                                     rows, false);
    } else {
        conv_roles<128, 1, false, S1>(a, tmap_w, ConvSmem{base, a.stages, sBar, abort_flag, tmem_base},
                                      rows, prefetch);
    }
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, Cfg<128, 2>::kTmemCols);
    }
}

// C_in not a multiple of 8: x [rows, C_in] and W [L*C_in, C_out] copied with
// zero channels appended up to C_pad (a multiple of 8), so that every tap's
// slice of a gathered row starts on a 16-byte boundary. 16-byte pieces of
// the outputs, one per thread (grid-stride): first x's (rows past *count
// skipped when count is given: compact inputs hold N' rows), then W's.
__global__ void __launch_bounds__(256) channel_pad_kernel(
    const uint16_t* __restrict__ x, long long x_rows, const int32_t* __restrict__ count, int C_in,
    int C_pad, uint4* __restrict__ xp, const uint4* __restrict__ W, int L, int C_out,
    uint4* __restrict__ Wp) {
    pdl_wait();
    pdl_trigger();
    long long rows = x_rows;
    if (count) {
        const long long n = *count;
        rows = n < 0 ? 0 : (n < x_rows ? n : x_rows);
    }
    const int xq = C_pad / 8;   // 16-byte pieces per padded row of x
    const int wq = C_out / 8;   // 16-byte pieces per row of W
    const long long nx = rows * xq;
    const long long nw = (long long)L * C_pad * wq;
    for (long long i = blockIdx.x * 256ll + threadIdx.x; i < nx + nw; i += gridDim.x * 256ll) {
        if (i < nx) {
            const long long r = i / xq;
            const int c0 = (int)(i - r * xq) * 8;
            const uint16_t* src = x + r * C_in + c0;
            uint32_t v[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t lo = c0 + 2 * e < C_in ? src[2 * e] : 0u;
                const uint32_t hi = c0 + 2 * e + 1 < C_in ? src[2 * e + 1] : 0u;
                v[e] = lo | (hi << 16);
            }
            xp[i] = make_uint4(v[0], v[1], v[2], v[3]);
        } else {
            const long long j = i - nx;
            const long long rp = j / wq;  // padded row l * C_pad + c
            const int l = (int)(rp / C_pad), c = (int)(rp - (long long)l * C_pad);
            Wp[j] = c < C_in ? W[((long long)l * C_in + c) * wq + (j - rp * wq)]
                             : make_uint4(0u, 0u, 0u, 0u);
        }
    }
}

// ---------------------------------------------------------------- host side

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix with a 128-byte
// swizzled box of box_cols x box_rows.
hc_status encode_2d(CUtensorMap* m, const void* base, long long rows, long long cols, int box_cols,
                    int box_rows) {
    auto enc = tensor_map_encoder();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled is unavailable");
        return HC_ERR_CUDA;
    }
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled failed (%d)", (int)r);
        return HC_ERR_CUDA;
    }
    return HC_OK;
}

// The weight matrix [K, C_out] (C_out a multiple of 64) as the 3-D tensor
// [C_out / 64][K][64] with 128-byte swizzled boxes of 64 x box_k x box_blocks.
hc_status encode_w3d(CUtensorMap* m, const void* base, long long K, long long C_out, int box_k,
                     int box_blocks) {
    auto enc = tensor_map_encoder();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled is unavailable");
        return HC_ERR_CUDA;
    }
    cuuint64_t dims[3] = {64, (cuuint64_t)K, (cuuint64_t)(C_out / 64)};
    cuuint64_t strides[2] = {(cuuint64_t)C_out * 2, 128};
    cuuint32_t box[3] = {64, (cuuint32_t)box_k, (cuuint32_t)box_blocks};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("cuTensorMapEncodeTiled (3-D weight view) failed (%d)", (int)r);
        return HC_ERR_CUDA;
    }
    return HC_OK;
}

// W: [K rows, C_out]. With C_out a multiple of 64, the 3-D view
// [C_out / 64][K][64] (the 64-column blocks 128 bytes apart) takes a tile's
// BN columns of a k-block in one box of 64 x 64 x BN/64; otherwise 2-D boxes
// of 64 K-rows x 64 output channels, one per block.
hc_status encode_weights(CUtensorMap* tw, ConvArgs& ka, int BN) {
    memset(tw, 0, sizeof *tw);
    ka.w3d = ka.C_out % 64 == 0;
    if (ka.w3d) return encode_w3d(tw, ka.W, ka.K, ka.C_out, kBK, BN / 64);
    return encode_2d(tw, ka.W, ka.K, ka.C_out, 64, kBK);
}

template <typename Kernel>
hc_status set_smem_limit(const DeviceCtx* ctx, Kernel k, bool (&done)[64], const char* what) {
    if (!done[ctx->device]) {
        hc_status st = check_cuda(
            cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemLimit),
            what);
        if (st != HC_OK) return st;
        done[ctx->device] = true;
    }
    return HC_OK;
}

template <int BN, int TM, bool TR = false>
hc_status launch_bn(const DeviceCtx* ctx, const ConvArgs& a, cudaStream_t s) {
    using C = Cfg<BN, TM>;
    static bool attr_set[64] = {};
    hc_status st = set_smem_limit(ctx, conv_tc_kernel<BN, TM, TR>, attr_set,
                                  "cudaFuncSetAttribute(conv_tc_kernel)");
    if (st != HC_OK) return st;
    CUtensorMap tw;
    ConvArgs ka = a;
    st = encode_weights(&tw, ka, BN);
    if (st != HC_OK) return st;
    const long long n_tiles = (a.C_out + BN - 1) / BN;
    const long long cap_work = (a.capacity + TM * kBM - 1) / (TM * kBM) * n_tiles;
    long long grid = cap_work < ctx->num_sms ? cap_work : ctx->num_sms;
    if (grid < 1) grid = 1;
    ka.stages = C::stages_for(a.L);
    return launch_pdl(conv_tc_kernel<BN, TM, TR>, dim3((unsigned)grid), dim3(kThreadsFor<TM>),
                      C::smem_bytes(a.L, ka.stages), s, "conv_tc_kernel", ka, tw);
}

// conv_tc_auto_kernel: one CTA per SM, or one per 128-row item of the
// capacity when there are fewer.
hc_status launch_auto(const DeviceCtx* ctx, const ConvArgs& a, cudaStream_t s) {
    static bool attr_set[64] = {};
    hc_status st = set_smem_limit(ctx, conv_tc_auto_kernel, attr_set,
                                  "cudaFuncSetAttribute(conv_tc_auto_kernel)");
    if (st != HC_OK) return st;
    CUtensorMap tw;
    ConvArgs ka = a;
    st = encode_weights(&tw, ka, 128);
    if (st != HC_OK) return st;
    const long long items = (a.capacity + kBM - 1) / kBM;
    long long grid = items < ctx->num_sms ? items : ctx->num_sms;
    if (grid < 1) grid = 1;
    AutoLayout::stages_for(a.L, ka.stages, ka.stages_tr);
    return launch_pdl(conv_tc_auto_kernel, dim3((unsigned)grid), dim3(kThreadsFor<2>),
                      AutoLayout::smem_bytes(a.L, ka.stages, ka.stages_tr), s,
                      "conv_tc_auto_kernel", ka, tw);
}

}  // namespace

bool conv_tc_supported(const ConvArgs& a, hc_dtype dt) {
    // C_in not a multiple of 8 runs on channel-padded copies of x and W (x
    // itself is read by 2-byte loads then)
    const bool pad = a.C_in % 8 != 0;
    const uintptr_t al = (pad ? 0 : (uintptr_t)a.x) | (uintptr_t)a.W | (uintptr_t)a.y |
                         (uintptr_t)a.out_dense;
    // tile indices are 32-bit in the kernel
    const long long tiles = (a.capacity + kBM - 1) / kBM * ((a.C_out + 63) / 64);
    return dt == HC_BF16 && a.C_out % 8 == 0 && al % 16 == 0 && (uintptr_t)a.x % 2 == 0 &&
           a.L <= HC_MAX_SPIRAL && tiles < (1ll << 31);
}

size_t conv_tc_pad_bytes(const ConvArgs& a) {
    if (a.C_in % 8 == 0) return 0;
    const size_t C_pad = (size_t)(a.C_in + 7) / 8 * 8;
    const size_t xb = ((size_t)a.x_rows * C_pad * 2 + 255) / 256 * 256;
    return xb + (size_t)a.L * C_pad * (size_t)a.C_out * 2;
}

int conv_tc_tile_n(const ConvArgs& a) {
    return a.C_out <= 64 ? 64 : 128;
}

hc_status launch_conv_tc(const DeviceCtx* ctx, const ConvArgs& a, cudaStream_t s) {
    if (a.C_in % 8 != 0) {
        // pad the channels (into the caller's workspace), then the same
        // kernel on C_pad channels: the appended channels are zeros in x and
        // rows of zeros in W, so every sum is unchanged
        if (!a.pad_ws) {
            set_error("conv_tc: C_in=%d needs the channel-padding workspace", a.C_in);
            return HC_ERR_INVALID_ARG;
        }
        const int C_pad = (a.C_in + 7) / 8 * 8;
        char* ws = static_cast<char*>(a.pad_ws);
        const size_t xb = ((size_t)a.x_rows * C_pad * 2 + 255) / 256 * 256;
        ConvArgs b = a;
        b.x = ws;
        b.W = ws + xb;
        b.C_in = C_pad;
        b.K = a.L * C_pad;
        b.pad_ws = nullptr;
        // compact inputs: only the first N' rows are read
        const int32_t* rows_from = a.mode == kSparseCompactX ? a.count : nullptr;
        const long long work = a.x_rows * (C_pad / 8) + (long long)a.L * C_pad * (a.C_out / 8);
        long long grid = (work + 255) / 256;
        const long long cap = 8ll * ctx->num_sms;
        if (grid > cap) grid = cap;
        if (grid < 1) grid = 1;
        hc_status st = launch_pdl(channel_pad_kernel, dim3((unsigned)grid), dim3(256), 0, s,
                                  "channel_pad_kernel", static_cast<const uint16_t*>(a.x),
                                  a.x_rows, rows_from, a.C_in, C_pad, reinterpret_cast<uint4*>(ws),
                                  static_cast<const uint4*>(a.W), a.L, a.C_out,
                                  reinterpret_cast<uint4*>(ws + xb));
        if (st != HC_OK) return st;
        return launch_conv_tc(ctx, b, s);
    }
    // Two-half items when the row count is known on the host (the dense
    // layer) and fills every SM with at least two of them: they halve the
    // weight traffic and per-stage overhead per MMA. A sparse call's row
    // count lives on the device, and two-half code paths compiled into the
    // loops of the one-half kernel cost the small layers ~1 us (instruction
    // fetch); such calls take two-half items through a row estimate or
    // conv_tc_auto_kernel (below), one-half items otherwise.
    const long long n_tiles = (a.C_out + 127) / 128;
    const bool two = a.mode == kDense && (a.capacity + 2 * kBM - 1) / (2 * kBM) * n_tiles >=
                                             2ll * ctx->num_sms;
    // A sparse call whose caller expects at least one two-half item per SM
    // (rows_hint) runs them too, with the transposed product (128 output
    // channels, no fused scatter or statistics): 250 -> 179 us at 670k rows,
    // 32 -> 28 us at 67k rows (1.7 items per SM), the same at 33k (0.9 per
    // SM), 11 -> 18 us at 6.8k (0.2 per SM). The results are the same either
    // way.
    // Without an estimate (rows_hint 0), a sparse call (rulebook or
    // resolved taps) whose capacity could fill every SM with two-half items
    // leaves the choice to the CTAs, which read the row count
    // (conv_tc_auto_kernel).
    const bool sparse = a.mode == kRulebook || a.mode == kSparseDenseX ||
                        a.mode == kSparseCompactX;
    if (sparse && a.C_out == 128 && !a.out_dense && !a.gn_part && a.C_in % 8 == 0) {
        if (a.mode == kRulebook && (a.rows_hint + 2 * kBM - 1) / (2 * kBM) >= ctx->num_sms)
            return launch_bn<128, 2, true>(ctx, a, s);
        if (a.rows_hint == 0 && (a.capacity + 2 * kBM - 1) / (2 * kBM) >= ctx->num_sms)
            return launch_auto(ctx, a, s);
    }
    if (conv_tc_tile_n(a) == 64) return launch_bn<64, 1>(ctx, a, s);
    return two ? (a.C_out == 128 && !a.out_dense && !a.gn_part ? launch_bn<128, 2, true>(ctx, a, s)
                                                                : launch_bn<128, 2, false>(ctx, a, s))
               : launch_bn<128, 1, false>(ctx, a, s);
}

}  // namespace hc
