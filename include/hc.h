/*
 * hc.h -- C ABI of libhc, the GB300 (sm_103a) sparse contact operators of
 * "ECO: Efficient Human-Contact Representation for Human-Scene Interaction".
 *
 * A sparse contact mask over body-mesh vertices selects the rows of a dense
 * human-scene tensor (Eq. 1); the selected rows are decomposed into a
 * coordinate list C' and compact features S' (Eq. 2); sparse layers then run
 * on the compact rows only (Sec. 3.2): convolution over each vertex's spiral
 * neighbourhood (Eqs. 4-5), linear (Eq. 6) and activation (Eq. 10).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every pointer argument is a DEVICE pointer on the current CUDA device,
 *    except where a comment says otherwise. The caller owns every buffer;
 *    nothing is retained after the call returns.
 *  - Work is enqueued on `stream` (NULL = the legacy default stream) and is
 *    asynchronous: the return status reports argument checks and launch
 *    errors only. Problems found on the device (an out-of-range index, a
 *    count above capacity, a bounded wait that ran out) set a sticky device
 *    status word, read and cleared by hc_get_device_status().
 *  - The active-row count N' stays on the device (`count`, one int32), so a
 *    chain of calls needs no host synchronisation and can be captured into a
 *    CUDA graph once the library has set itself up on the device (see
 *    hc_mask_compact).
 *  - Layouts are row-major. dtype HC_F32 means IEEE binary32; HC_BF16 means
 *    bfloat16 storage with fp32 accumulation (tensor cores) and a
 *    round-to-nearest-even store. Bias is always fp32. The input, weight and
 *    output of one call share one dtype.
 *  - Neighbours outside the active set contribute nothing (Eq. 4 keeps only
 *    kernel taps whose coordinate is present in C), which equals the dense
 *    layer on the masked input (Eq. 1) restricted to active rows.
 *  - Sizes are int; B*V and every row count must stay below 2^31.
 */
#ifndef HC_H
#define HC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* hc_stream_t; /* same type as cudaStream_t */

typedef enum {
    HC_OK = 0,
    HC_ERR_INVALID_ARG = 1,   /* null pointer, bad size, bad enum, misaligned pointer */
    HC_ERR_UNSUPPORTED = 2,   /* valid but not supported (e.g. L > HC_MAX_SPIRAL) */
    HC_ERR_CAPACITY = 3,      /* device: count exceeded the stated capacity */
    HC_ERR_INVALID_INDEX = 4, /* device: spiral/row_of/coords entry out of range */
    HC_ERR_TIMEOUT = 5,       /* device: a bounded wait inside a kernel ran out */
    HC_ERR_CUDA = 6           /* CUDA runtime error; see hc_last_error_string() */
} hc_status;

typedef enum { HC_F32 = 0, HC_BF16 = 1 } hc_dtype;
typedef enum { HC_ACT_NONE = 0, HC_ACT_ELU = 1, HC_ACT_RELU = 2 } hc_act;
typedef enum {
    HC_LAYOUT_DENSE = 0,  /* [B, V, C]: row (b, v) at (b*V + v)*C */
    HC_LAYOUT_COMPACT = 1 /* [N', C]: row n is the n-th entry of coords */
} hc_layout;

#define HC_MAX_SPIRAL 32 /* largest spiral length L */

/*
 * hc_mask_compact -- decomposition of a masked tensor into coordinates (Eq. 2)
 * and the inverse index map idx() used by the sparse convolution (Eq. 4).
 *
 *   mask     [B, V] uint8. Row (b, v) is active iff mask[b*V + v] != 0
 *            (the paper's mask holds 0/1, Eq. 1; any nonzero byte counts).
 *   coords   [B*V, 2] int32 capacity. Receives the active rows as (b, v)
 *            pairs in ascending (b, v) order: the coordinate matrix C'.
 *   row_of   [B, V] int32, or NULL. Receives the position of (b, v) in
 *            coords, or -1 if inactive.
 *   batch_offsets [B+1] int32, or NULL. Receives the number of active rows
 *            in frames before b; batch_offsets[B] = N'. Rows of frame b are
 *            [batch_offsets[b], batch_offsets[b+1]).
 *   count    one int32: receives N'.
 * B >= 0, V >= 0; B*V == 0 gives N' = 0. Results are bit-exact and unique.
 *
 * Scratch: a small per-(device, stream) workspace (one int32 per 4096 mask
 * bytes) is allocated by the library on the first call that needs it and
 * kept until process exit. Make the first call on each device and stream
 * outside stream capture; later calls allocate nothing unless a larger mask
 * is seen. Calls on one stream are ordered; calls on different streams use
 * different workspaces.
 */
hc_status hc_mask_compact(const uint8_t* mask, int B, int V, int32_t* coords,
                          int32_t* row_of, int32_t* batch_offsets, int32_t* count,
                          hc_stream_t stream);

/*
 * hc_mask_compact_static -- hc_mask_compact that allocates nothing. The paper
 * has no counterpart; this entry point exists for callers of this library
 * that cannot allocate device memory at the moment they compact a mask:
 * processes that hand all device memory to their own pool up front and must
 * not allocate behind its back, and code on a path where a cudaMalloc or
 * cudaFree (which can synchronise the whole device) is not allowed.
 *
 * Same arguments, results and errors as hc_mask_compact (bit-identical
 * outputs). Differences:
 *  - Scratch: a fixed array of HC_STATIC_MAX_MASK_BYTES / 4096 int32 (16 KiB)
 *    inside the library's device image, present on every GPU that loads the
 *    library until the process exits. No cudaMalloc, cudaFree or allocating
 *    library routine is called.
 *  - Limit: B*V may not exceed HC_STATIC_MAX_MASK_BYTES; larger masks are
 *    rejected with HC_ERR_UNSUPPORTED before anything is launched.
 *  - Set-up: the first call on each device looks up the array's device
 *    address (with that device current); make that first call before any
 *    stream capture.
 *  - Sharing: every call on a device uses the same array, which keeps the
 *    previous call's contents (each call rewrites what it reads, so no
 *    clearing is needed). Calls whose kernels overlap on the GPU (e.g. on
 *    two streams without ordering between them) race on it.
 */
#define HC_STATIC_MAX_MASK_BYTES (4096 * 4096)
hc_status hc_mask_compact_static(const uint8_t* mask, int B, int V, int32_t* coords,
                                 int32_t* row_of, int32_t* batch_offsets, int32_t* count,
                                 hc_stream_t stream);

/*
 * hc_sparse_spiral_conv_fwd -- sparse convolution on the spiral
 * neighbourhood (Eqs. 4-5) with fused bias (Eq. 6) and activation (Eq. 10).
 *
 * For each active row n < N' with coordinate (b, v) = coords[n]:
 *   y[n, o] = act( bias[o] + sum_{l<L} sum_{c<C_in}
 *                  S(b, spiral[v*L + l])[c] * W[(l*C_in + c)*C_out + o] )
 * where S(b, u) is the input row of (b, u) when u >= 0 and row_of[b*V+u] >= 0,
 * and the term is absent otherwise. Slot 0 of the spiral is the vertex
 * itself (the centre tap); -1 entries mean "no neighbour".
 *
 *   x        x_layout DENSE: [B, V, C_in]; COMPACT: [N', C_in] in coords order
 *   coords, row_of, count   as written by hc_mask_compact (row_of required)
 *   spiral   [V, L] int32, entries in [-1, V)
 *   W        [L*C_in, C_out] of dtype dt, row index l*C_in + c
 *   bias     [C_out] fp32, or NULL for zero
 *   y        [B*V, C_out] capacity of dtype dt; rows 0..N'-1 are written,
 *            in coords order (the conv outputs the centre coordinates, Eq. 5).
 * 1 <= L <= HC_MAX_SPIRAL, C_in >= 1, C_out >= 1.
 * Out-of-range spiral/row_of/coords entries contribute nothing and set
 * HC_ERR_INVALID_INDEX; a count above B*V is clamped and sets HC_ERR_CAPACITY.
 * bf16 with C_out % 8 == 0 and 16-byte aligned W, y runs on the tensor cores
 * (tcgen05); other shapes run on CUDA cores. With C_in % 8 != 0 (x then
 * needs only 2-byte alignment) x and W are first copied, with zero channels
 * appended up to C_pad = the next multiple of 8, into the per-stream
 * workspace (x_rows * C_pad * 2 + L * C_pad * C_out * 2 bytes; compact inputs
 * copy their first N' rows only); the sums are unchanged. With C_out = 128
 * and B*V of at least 256 rows per SM, the kernel reads N' on the device and
 * multiplies 256-row items (two 128-row halves sharing each weight stage) when
 * every SM gets one, 128-row items otherwise; the results are the same bits
 * either way.
 */
hc_status hc_sparse_spiral_conv_fwd(const void* x, hc_layout x_layout, hc_dtype dt,
                                    const int32_t* coords, const int32_t* row_of,
                                    const int32_t* count, const int32_t* spiral, int B, int V,
                                    int L, int C_in, int C_out, const void* W, const float* bias,
                                    hc_act act, void* y, hc_stream_t stream);

/*
 * hc_conv_rulebook -- the indexing matrix of the sparse convolution (Eq. 4),
 * materialised: for every active row n < N' and spiral slot l < L,
 *   rulebook[l*(B*V) + n] = the input row feeding that tap, or -1 when the
 *   tap is absent (spiral[v*L+l] == -1, or the neighbour (b, u) is inactive).
 * The input row is b*V + u for x_layout DENSE and row_of[b*V + u] for
 * COMPACT. The coordinates do not change from layer to layer (Eq. 5), so one
 * rulebook serves every conv layer run on the same mask.
 *   coords, row_of, count   as written by hc_mask_compact
 *   spiral    [V, L] int32, entries in [-1, V)
 *   rulebook  [L, B*V] int32, slot-major, caller-owned; columns n >= N'
 *             are not written.
 * Out-of-range entries are reported (HC_ERR_INVALID_INDEX) and stored as -1.
 */
hc_status hc_conv_rulebook(const int32_t* coords, const int32_t* row_of, const int32_t* count,
                           const int32_t* spiral, int B, int V, int L, hc_layout x_layout,
                           int32_t* rulebook, hc_stream_t stream);

/*
 * hc_mask_compact_rulebook -- hc_mask_compact followed by hc_conv_rulebook on
 * its output (Eq. 2 and the Eq. 4 indexing matrix), in two kernels when
 * V <= 65535: a count pass, then one pass per (frame, block of 1024
 * vertices) that ranks the frame's mask bytes in shared memory and writes
 * coords, row_of, batch_offsets, count and the rulebook columns of its
 * active vertices, every tap lookup answered from shared memory. Larger
 * frames run the two operations' own kernels. The results are identical to
 * the two calls (bit-exact).
 *   mask, B, V, coords, row_of, batch_offsets, count   as hc_mask_compact
 *                                                      (row_of required)
 *   spiral, L, x_layout, rulebook                      as hc_conv_rulebook
 * Out-of-range spiral entries are reported (HC_ERR_INVALID_INDEX) and their
 * taps stored as -1. Uses the library's per-stream workspace (one int32 per
 * 4096 mask bytes).
 */
hc_status hc_mask_compact_rulebook(const uint8_t* mask, int B, int V, const int32_t* spiral, int L,
                                   hc_layout x_layout, int32_t* coords, int32_t* row_of,
                                   int32_t* batch_offsets, int32_t* count, int32_t* rulebook,
                                   hc_stream_t stream);

/*
 * hc_sparse_conv_rulebook_fwd -- the sparse convolution (Eq. 5) with fused
 * bias (Eq. 6) and activation (Eq. 10), through a precomputed rulebook:
 *   y[n, o] = act( bias[o] + sum_{l<L, r = rulebook[l*capacity+n] >= 0}
 *                  sum_{c<C_in} x[r, c] * W[(l*C_in + c)*C_out + o] ),  n < N'
 *   x         [x_rows, C_in] of dtype dt; rulebook entries must lie in
 *             [-1, x_rows) (others are reported and skipped)
 *   rulebook  [L, capacity] int32 as written by hc_conv_rulebook
 *             (capacity = B*V there)
 *   count     N' on the device, at most capacity (clamped, HC_ERR_CAPACITY)
 *   W, bias, act as for hc_sparse_spiral_conv_fwd.
 *   y         [capacity, C_out] compact output of dtype dt, or NULL.
 *   out       [B, V, C_out] dense output of dtype dt, or NULL: when given, row
 *             n is also written at coords[n] = (b, v), the scatter of
 *             hc_scatter_dense fused into the epilogue (inactive rows of out
 *             are not touched). Needs coords (as written by hc_mask_compact),
 *             B >= 1 and V >= 1. At least one of y and out must be given.
 * Results equal hc_sparse_spiral_conv_fwd (and hc_scatter_dense without
 * zero fill) on the same inputs.
 */
hc_status hc_sparse_conv_rulebook_fwd(const void* x, hc_dtype dt, int x_rows,
                                      const int32_t* rulebook, const int32_t* count, int capacity,
                                      int L, int C_in, int C_out, const void* W, const float* bias,
                                      hc_act act, void* y, const int32_t* coords, int B, int V,
                                      void* out, hc_stream_t stream);

/*
 * hc_sparse_conv_rulebook_fwd_hint -- hc_sparse_conv_rulebook_fwd with the
 * caller's host-side estimate of N' (rows_hint >= 0; 0 = unknown), which
 * the call uses only to choose how the tensor cores tile the rows. The
 * tiling that is fastest for many rows (two 128-row halves per item sharing
 * every weight stage, multiplied as one M = 128 channels x N = 256 rows
 * product) is slower when there are too few items to fill the GPU; it
 * applies to bf16, C_out = 128, and neither out nor group-norm statistics.
 * With rows_hint giving at least one such item per SM (about 39k rows on
 * 152 SMs) the launch uses it directly; with a smaller nonzero estimate it
 * uses one-half items; with none (0, and in hc_sparse_conv_rulebook_fwd)
 * a call whose capacity could fill the SMs with such items launches a
 * kernel that reads N' on the device and chooses (a little slower than a
 * direct launch at small N': ~0.2 us). The results are bit-identical in
 * every case, so any estimate (the previous batch's count, the mask's
 * expected density) is safe: a wrong one only costs time. rows_hint < 0 is
 * HC_ERR_INVALID_ARG.
 */
hc_status hc_sparse_conv_rulebook_fwd_hint(const void* x, hc_dtype dt, int x_rows,
                                           const int32_t* rulebook, const int32_t* count,
                                           int capacity, int L, int C_in, int C_out,
                                           const void* W, const float* bias, hc_act act, void* y,
                                           const int32_t* coords, int B, int V, void* out,
                                           long long rows_hint, hc_stream_t stream);

/*
 * hc_sparse_linear_fwd -- linear layer on compact rows (Eq. 6), row-wise
 *   y[n, o] = act( bias[o] + sum_{c<C_in} x[n, c] * W[c*C_out + o] ),  n < N'
 * The coordinates are unchanged (C' = C).
 *   x [capacity, C_in], y [capacity, C_out], W [C_in, C_out] of dtype dt;
 *   count: one int32 on the device (N'), must not exceed `capacity`
 *   (clamped, HC_ERR_CAPACITY).
 */
hc_status hc_sparse_linear_fwd(const void* x, hc_dtype dt, const int32_t* count, int capacity,
                               int C_in, int C_out, const void* W, const float* bias, hc_act act,
                               void* y, hc_stream_t stream);

/*
 * hc_sparse_group_norm_fwd -- group normalisation of compact rows (Eqs. 7-9),
 * statistics taken over each frame's active rows only. Frame b owns the rows
 * [batch_offsets[b], batch_offsets[b+1]) (as written by hc_mask_compact); the
 * C channels form G groups of C/G consecutive channels. For every (b, g), over
 * the n = rows(b) * C/G values of the group:
 *   mu = sum / n,  var = sum((v - mu)^2) / n,  out = (v - mu) / sqrt(var + eps)
 * then out * gamma[c] + beta[c] (each optional: NULL = 1 / 0) and the
 * activation act (Eq. 10). G = 1 is layer normalisation.
 *   x, y      [capacity, C] of dtype dt; y may be x (in place). Rows outside
 *             every frame's range are not touched.
 *   batch_offsets [B+1] int32 on the device, non-decreasing, within
 *             [0, capacity]; otherwise HC_ERR_INVALID_INDEX is reported
 *             (hc_get_device_status) and the output is unspecified, but no
 *             access leaves x, y or the library's workspace.
 * Statistics in fp32 by pairwise (count, mean, M2) merging; the variance is
 * taken around the mean, never as E[x^2] - mean^2. Uses the library's
 * per-stream workspace ((B + 2 * SMs) * G * 16 bytes at most).
 */
hc_status hc_sparse_group_norm_fwd(const void* x, hc_dtype dt, const int32_t* batch_offsets, int B,
                                   int capacity, int C, int G, float eps, const float* gamma,
                                   const float* beta, hc_act act, void* y, hc_stream_t stream);

/*
 * hc_sparse_conv_gn_fwd -- a convolution layer followed by group
 * normalisation and the activation, the order of a block of the encoder
 * (Eqs. 5-6, then Eqs. 7-9, then Eq. 10):
 *   z = conv(x) + bias            as hc_sparse_conv_rulebook_fwd with act
 *                                 NONE, stored in y (dtype dt)
 *   y = act(GN(z) * gamma + beta) as hc_sparse_group_norm_fwd on y in place
 * The group statistics are those of z as stored (bf16-rounded for bf16).
 *   x, rulebook, count, capacity, L, C_in, C_out, W, bias as for
 *             hc_sparse_conv_rulebook_fwd; y [capacity, C_out] of dtype dt
 *   coords    [capacity, 2] int32 from hc_mask_compact (frame of row n is
 *             coords[2n]), batch_offsets [B+1] from the same call: the frame
 *             table must start at 0, end at *count and agree with coords
 *             (HC_ERR_INVALID_INDEX otherwise, output unspecified)
 *   G, eps, gamma, beta, act as for hc_sparse_group_norm_fwd (G divides C_out)
 * bf16 with C_out/G a power of two from 8 to the tensor-core tile (64
 * channels when C_out <= 64, else 128), C_out/8 a power of two: the
 * tensor-core epilogue writes one partial (count, mean, M2) per (frame,
 * 32-row block inside the frame, group), and one per (row, group) for blocks
 * shared by two frames, and a single normalising pass merges them (two
 * launches, y written once by each). Otherwise the two operations run one
 * after the other. Uses the library's per-stream workspace
 * ((B + capacity/32 + 1) * G * 16 + capacity * G * 8 bytes, or that of
 * hc_sparse_group_norm_fwd).
 */
hc_status hc_sparse_conv_gn_fwd(const void* x, hc_dtype dt, int x_rows, const int32_t* rulebook,
                                const int32_t* count, int capacity, int L, int C_in, int C_out,
                                const void* W, const float* bias, const int32_t* coords,
                                const int32_t* batch_offsets, int B, int G, float eps,
                                const float* gamma, const float* beta, hc_act act, void* y,
                                hc_stream_t stream);

/*
 * hc_conv_rulebook_transpose -- the Eq. 4 mapping read backwards, for the
 * input gradient: for every input row j, the taps (n, l) with
 * rulebook[l][n] == j, n < *count, as keys n*L + l in ascending order.
 *   rulebook  [L, capacity] from hc_conv_rulebook (capacity = its stride)
 *   row_ptr   [x_rows + 1] int32: row j's keys are taps[row_ptr[j] ..
 *             row_ptr[j+1])
 *   taps      [L * capacity] int32
 * Entries outside [-1, x_rows) are skipped and reported
 * (HC_ERR_INVALID_INDEX). Computed once per mask and reused by every layer.
 * Uses the library's per-stream workspace (2 int32 per input row).
 */
hc_status hc_conv_rulebook_transpose(const int32_t* rulebook, const int32_t* count, int capacity,
                                     int L, int x_rows, int32_t* row_ptr, int32_t* taps,
                                     hc_stream_t stream);

/*
 * hc_sparse_conv_rulebook_bwd -- gradients of the sparse spiral convolution
 * computed by hc_sparse_conv_rulebook_fwd. The paper gives the forward only
 * (Eqs. 4-5, 6, 10); these follow from it by the chain rule:
 *   dz[n][o]  = dy[n][o] * act'(y[n][o])   (ELU: 1 if y > 0 else y + 1;
 *                                           ReLU: 1 if y > 0 else 0)
 *   dbias[o]  = sum_n dz[n][o]
 *   dW[l*C_in + c][o] = sum_n x[j(n,l)][c] * dz[n][o]
 *   dx[j][c]  = sum over taps (n, l) reading row j of sum_o dz[n][o] W[l*C_in + c][o]
 * over output rows n < *count, with j(n,l) = rulebook[l][n] (absent taps -1
 * contribute nothing).
 *   x        [x_rows, C_in] input rows the forward read (dense B*V rows or
 *            compact), dtype dt; needed for dW
 *   y, dy    [capacity, C_out] forward output and upstream gradient, dt
 *   W        [L*C_in, C_out], dt; needed for dx
 *   row_ptr, taps  from hc_conv_rulebook_transpose; needed for dx
 *   dx       [x_rows, C_in], dt, every row written (0 where no tap reads
 *            it), or NULL
 *   dW       [L*C_in, C_out] fp32 or NULL;  dbias [C_out] fp32 or NULL
 * bf16: dW on tensor cores (tcgen05, fp32 accumulation); dz and the
 * per-tap products dz W^T are rounded to bf16 once before the input-gradient
 * sums. fp32: CUDA cores throughout. Every sum runs in a fixed order
 * (deterministic). Uses the library's per-stream workspace.
 */
hc_status hc_sparse_conv_rulebook_bwd(const void* x, hc_dtype dt, int x_rows,
                                      const int32_t* rulebook, const int32_t* count, int capacity,
                                      int L, int C_in, int C_out, const void* W, const void* y,
                                      const void* dy, hc_act act, const int32_t* row_ptr,
                                      const int32_t* taps, void* dx, float* dW, float* dbias,
                                      hc_stream_t stream);

/*
 * hc_mask_score_update -- the mask-score update of Eq. 3 (Sec. 3.1, Sparse
 * Mask Selection). O holds the outputs of K masks, [K, N, D] row-major (mask
 * k's N rows of D features). With S[i][k] = || O_i^T O_k ||_F^2:
 *   sim[i][k]    = S[i][k] / (|| O_k^T O_k ||_F * || O_i^T O_i ||_F)
 *   alpha_out[k] = alpha_in[k] + 1/(K-1) * sum over i != k of (1 - sim[i][k])
 * Readings: a mask whose output is all zero has similarity 0 to every mask;
 * with K = 1 alpha is copied unchanged.
 *   O          [K, N, D] of dtype dt (bf16: tensor cores, fp32 accumulation;
 *              fp32: CUDA cores, fp32 accumulation)
 *   alpha_in, alpha_out  [K] fp32 on the device; may be the same buffer
 *   sim        [K, K] fp32 or NULL
 * K*D at most HC_MASK_SCORE_MAX_FEATURES (else HC_ERR_UNSUPPORTED). Uses the
 * library's per-stream workspace: 64 KiB per work item (upper-triangle
 * 128 x 128 tiles of the [K*D]^2 Gram matrix times row splits, about the
 * SM count), plus N * K*D (rounded to 128) bf16 when D is not a multiple of 8.
 */
#define HC_MASK_SCORE_MAX_FEATURES 8192
hc_status hc_mask_score_update(const void* O, hc_dtype dt, int K, int N, int D,
                               const float* alpha_in, float* alpha_out, float* sim,
                               hc_stream_t stream);

/*
 * hc_mask_select_topk -- the kappa masks kept at inference (Sec. 3.1, Sparse
 * Mask Selection): indices of the kappa highest scores of alpha [K] (fp32,
 * device), highest first; equal scores lowest index first; a NaN score ranks
 * below every number. selected: [kappa] int32 on the device.
 * K at most HC_TOPK_MAX_MASKS.
 */
#define HC_TOPK_MAX_MASKS 32768
hc_status hc_mask_select_topk(const float* alpha, int K, int kappa, int32_t* selected,
                              hc_stream_t stream);

/*
 * hc_kappa_masks -- every kept mask applied to every sample (Eq. 1 per kept
 * mask, Sec. 3.1): out [B*kappa, V] with frame b*kappa + j equal to
 * masks[selected[j]] ([K, V] uint8). The result feeds hc_mask_compact; a
 * selected index outside [0, K) gives an all-zero frame and
 * HC_ERR_INVALID_INDEX.
 */
hc_status hc_kappa_masks(const uint8_t* masks, int K, int V, const int32_t* selected, int kappa,
                         int B, uint8_t* out, hc_stream_t stream);

/*
 * hc_gather_rows -- the feature matrix S' of Eq. 2: y[n] = x[f / fps, v] for
 * the n-th active coordinate (f, v) = coords[n], n < *count, where x is the
 * dense [B_in, V, C] input of dtype dt and fps = frames_per_sample (kappa
 * after hc_kappa_masks, else 1). Rows are copied bit for bit; y is
 * [capacity, C]. A coordinate outside the input is reported
 * (HC_ERR_INVALID_INDEX) and its row left untouched; *count above capacity
 * is clamped (HC_ERR_CAPACITY). x may be pinned host memory (cudaHostAlloc,
 * the same pointer on the device under unified addressing): the kernel then
 * reads only the active rows across the host link (zero-copy), which is how
 * a dense host-side input becomes compact device rows without copying the
 * whole tensor.
 * coords may be NULL: y[n] = row n of x (x viewed as B_in * V rows of C;
 * frames_per_sample unused) for n < *count, rows n >= B_in * V reported
 * (HC_ERR_INVALID_INDEX) and left untouched: a copy of the first N' rows
 * sized on the device. With y in pinned host memory this reads compact
 * results back without the host learning N' first (no host wait between
 * the producing call and the copy).
 */
hc_status hc_gather_rows(const void* x, hc_dtype dt, int B_in, int V, int C, const int32_t* coords,
                         const int32_t* count, int capacity, int frames_per_sample, void* y,
                         hc_stream_t stream);

/*
 * hc_scatter_dense -- inverse of the decomposition (Eq. 2): compact rows back
 * into a dense [B, V, C] tensor.
 *   zero_fill == 0: out[coords[n]] = y[n] for n < N'; other rows untouched.
 *   zero_fill != 0: every row of out is written: y[n] at coords[n], zeros
 *                   elsewhere (the masked tensor of Eq. 1).
 *   y [N', C] of dtype dt (elements are copied bit for bit), coords/count as
 *   written by hc_mask_compact, out [B, V, C].
 *   row_of   [B, V] as written by hc_mask_compact, or NULL. Optional: with
 *            zero_fill it lets one pass write every dense row exactly once
 *            (coords may then be NULL); without it the zero fill is a
 *            separate pass over out before the scatter. Ignored when
 *            zero_fill == 0. (The problem statement's call has no row_of;
 *            passing NULL gives exactly that call.)
 */
hc_status hc_scatter_dense(const void* y, hc_dtype dt, const int32_t* coords,
                           const int32_t* row_of, const int32_t* count, int B, int V, int C,
                           int zero_fill, void* out, hc_stream_t stream);

/*
 * hc_spiral_conv_fwd -- the dense spiral-conv layer the sparse one replaces
 * (Sec. 3.2), used as the speed-up denominator: every (b, v) is an output row,
 *   y[(b*V+v), o] = act( bias[o] + sum_l sum_c x[b, spiral[v*L+l], c] *
 *                                            W[(l*C_in + c)*C_out + o] )
 * with -1 spiral entries skipped. x [B, V, C_in], y [B, V, C_out].
 */
hc_status hc_spiral_conv_fwd(const void* x, hc_dtype dt, const int32_t* spiral, int B, int V,
                             int L, int C_in, int C_out, const void* W, const float* bias,
                             hc_act act, void* y, hc_stream_t stream);

/*
 * hc_get_device_status -- synchronises `stream`, then reads and clears the
 * current device's sticky status word. Returns HC_OK if no kernel reported a
 * problem since the last read, else the lowest-numbered device error seen
 * (HC_ERR_CAPACITY, HC_ERR_INVALID_INDEX or HC_ERR_TIMEOUT), or HC_ERR_CUDA
 * if the synchronisation itself failed.
 */
hc_status hc_get_device_status(hc_stream_t stream);

/*
 * hc_test_set_option -- hooks for this library's own tests; the paper has no
 * counterpart and the operators never need them. They reach code paths that
 * ordinary inputs do not select. Settings stay until changed.
 *   HC_TEST_GROUP_NORM_PATH (process-wide): 0 = the library's own choice
 *       (default); 1 = always the per-(frame, group) kernel; 2 = the
 *       row-range kernels wherever the layout allows them.
 *   HC_TEST_WAIT_LIMIT_NS (current device): how long the pipelined kernels
 *       (tensor-core conv, mask score, weight gradient) wait on any one
 *       pipeline barrier before they give up, report HC_ERR_TIMEOUT and
 *       unwind. value > 0 sets it in nanoseconds; 0 restores the default
 *       (2 s). The unwind's own waits, for copies and MMAs already issued,
 *       always keep the default. A lowered limit makes ordinary calls fail
 *       with HC_ERR_TIMEOUT and unspecified outputs: it exists to test that
 *       path. Synchronous (a small host-to-device copy).
 * Returns HC_ERR_INVALID_ARG for an unknown option or a value out of range.
 */
typedef enum { HC_TEST_GROUP_NORM_PATH = 1, HC_TEST_WAIT_LIMIT_NS = 2 } hc_test_option;
hc_status hc_test_set_option(int option, long long value);

/* Text of the last host-side error on the calling thread ("" if none). */
const char* hc_last_error_string(void);

/* Library version, "major.minor.patch". */
const char* hc_version(void);

#ifdef __cplusplus
}
#endif

#endif /* HC_H */
