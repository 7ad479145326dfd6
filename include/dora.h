/*
 * dora.h -- C ABI of the GB300 (sm_103a) deployment hot path of DORA's pruned
 * Vision Transformer forward ("DORA: Dynamic Online Reinforcement Agent for
 * Token Pruning in Vision Transformers").
 *
 * What the path computes (Eq. 1, Sec. 3.1):
 *     H_attn = H + Attention(LayerNorm(H))
 *     H_keep = H_attn with the selected visual rows deleted (CLS and the order
 *              of survivors kept)
 *     H_next = H_keep + MLP(LayerNorm'(H_keep))
 * for a batch whose images carry different token counts, packed row after row
 * into one [T, D] bf16 buffer with int32 sequence boundaries cu[B+1]
 * (cu[0] = 0, image i owns rows [cu[i], cu[i+1]), its row cu[i] is CLS).
 *
 * Conventions shared by every entry point:
 *  - Every pointer is device memory owned by the caller, unless a comment says
 *    "host".  The library never allocates and keeps no pointer after a call.
 *  - bf16 tensors are passed as raw 16-bit patterns (dora_bf16), row-major and
 *    contiguous.  Pointers handed to the tensor-memory-accelerator paths
 *    (dora_linear, dora_varlen_attn, dora_pruned_block) must be 16-byte aligned.
 *  - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream) and never synchronises the host, except dora_read_status.
 *  - The return value is a host-side status.  Host-side argument checks fail
 *    fast with DORA_ERR_INVALID_ARG / DORA_ERR_UNSUPPORTED and launch nothing.
 *  - Problems only the device can see (a keep count outside [1, n_i], an image
 *    longer than max_seqlen, a bounded wait that ran out) are written to an
 *    optional device int32 `status` word: the first nonzero code wins and the
 *    kernel carries on with clamped values.  Kernels never trap.
 *  - Row counts that depend on earlier device work (T_out after a deletion)
 *    stay on the device: callers pass capacities (`*_cap`, upper bounds used
 *    for grid sizes and buffer bounds) and the kernels read the live count
 *    from cu[batch].
 *  - The current CUDA device must be compute capability 10.3 (GB300);
 *    otherwise every entry point returns DORA_ERR_UNSUPPORTED.
 */
#ifndef DORA_H_
#define DORA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t dora_bf16;            /* raw bfloat16 bits */
typedef struct CUstream_st* dora_stream_t;  /* same type as cudaStream_t */

enum dora_status {
  DORA_OK = 0,
  DORA_ERR_INVALID_ARG = 1,        /* host check: null pointer, bad size, misalignment */
  DORA_ERR_UNSUPPORTED = 2,        /* head_dim != 64, dim % 64 != 0, device is not sm_103 */
  DORA_ERR_CUDA = 3,               /* a CUDA runtime/driver call failed */
  DORA_ERR_TIMEOUT = 4,            /* device: a bounded pipeline wait ran out */
  DORA_ERR_DEVICE_BAD_COUNT = 5,   /* device: keep count outside [1, n_i]; clamped */
  DORA_ERR_DEVICE_SEQLEN = 6,      /* device: an image is longer than max_seqlen,
                                      or a row index/count exceeds a capacity */
  DORA_ERR_SCRATCH_TOO_SMALL = 7,  /* dora_pruned_block_noalloc: the block needs more
                                      than DORA_NOALLOC_SCRATCH_BYTES of scratch */
};

/* Epilogues of dora_linear. */
enum dora_epilogue {
  DORA_EPI_BIAS = 0,          /* y = x W^T + b                 */
  DORA_EPI_BIAS_GELU = 1,     /* y = GELU(x W^T + b), exact erf */
  DORA_EPI_BIAS_RESIDUAL = 2  /* y = r + x W^T + b             */
};

/* Human-readable name of a status code (static string). */
const char* dora_status_string(int code);

/* ABI version, currently 2. */
int dora_version(void);

/*
 * dora_select_keep -- deterministic top-k deletion, one image at a time
 * (Sec. 3.2 "Sampling and deployment"; Appendix A.3: at inference the
 * selector removes the k_l highest-scoring visual tokens; CLS is never
 * selected).
 *
 * scores       fp32 [T_in], row-aligned with the packed input; higher = remove
 *              first.  The entry of each image's CLS row is ignored.
 * cu_in        int32 [batch+1] input boundaries.
 * keep_counts  int32 [batch]: m_i, tokens image i keeps, CLS included
 *              (m_i = n_i - k_i).  Valid range 1 <= m_i <= n_i (an empty image
 *              keeps 0).  Out-of-range values are clamped into the range and
 *              DORA_ERR_DEVICE_BAD_COUNT is written to *status.
 * max_seqlen   upper bound of n_i (<= 8192); sizes shared memory.  An image
 *              longer than this keeps nothing and raises DORA_ERR_DEVICE_SEQLEN.
 * kept_idx     out int32 [capacity >= T_in]: global input row of every kept
 *              token, image after image, ascending within an image.
 * cu_out       out int32 [batch+1]: cu_out[i+1] - cu_out[i] = clamped m_i.
 * status       nullable device int32.
 * Ties: among equal scores the lower index is kept.  Order of scores: -0 ==
 * +0, every NaN ranks above +inf.  Bit-exact and deterministic.
 */
int dora_select_keep(const float* scores, const int32_t* cu_in, const int32_t* keep_counts,
                     int32_t batch, int32_t max_seqlen, int32_t* kept_idx, int32_t* cu_out,
                     int32_t* status, dora_stream_t stream);

/*
 * dora_compact -- hard deletion by stream compaction (Sec. 3.1 pruning
 * operator; Sec. 3.5 "Inference": surviving sequences are compacted into a
 * packed buffer with explicit sequence boundaries, per-image order kept).
 *
 * x          bf16 [t_in_cap, dim] rows to gather from.
 * kept_idx   int32 [T_out] from dora_select_keep; every entry < t_in_cap.
 * cu_out     int32 [batch+1] from dora_select_keep; T_out = cu_out[batch].
 * ids_in     nullable int32 [t_in_cap]: original token id of each input row.
 * packed     out bf16 [capacity >= t_in_cap, dim]: packed[r] = x[kept_idx[r]],
 *            bit for bit.
 * ids_out    nullable out int32: ids_out[r] = ids_in[kept_idx[r]].
 * dim % 8 == 0.  An index or T_out beyond t_in_cap is skipped and raises
 * DORA_ERR_DEVICE_SEQLEN.
 */
int dora_compact(const dora_bf16* x, int32_t dim, const int32_t* kept_idx, const int32_t* cu_out,
                 int32_t batch, int32_t t_in_cap, const int32_t* ids_in, dora_bf16* packed,
                 int32_t* ids_out, int32_t* status, dora_stream_t stream);

/*
 * dora_select_compact -- dora_select_keep and the compaction of the kept
 * rows in one launch (Sec. 3.2 "Sampling and deployment" and Appendix A.3
 * for the kept set; Sec. 3.1 pruning operator and Sec. 3.5 "Inference" for
 * the packed buffer).
 *
 * Arguments as dora_select_keep, plus:
 * x          bf16 [t_in_cap, dim] rows to gather from (16-byte aligned;
 *            dim % 8 == 0, dim <= 2048).
 * ids_in     nullable int32 [t_in_cap]; ids_out nullable out int32 (given
 *            together): ids_out[r] = ids_in[kept_idx[r]].
 * mv_in      nullable fp32 [t_in_cap, 2]; mv_out nullable out (given
 *            together, 8-byte aligned): mv_out[r] = mv_in[kept_idx[r]].
 * packed     out bf16 [capacity >= t_in_cap, dim]: packed[r] =
 *            x[kept_idx[r]], bit for bit.
 * kept_idx, cu_out and status are written exactly as dora_select_keep
 * writes them, except that an image whose rows do not lie inside
 * [0, t_in_cap) keeps nothing and raises DORA_ERR_DEVICE_SEQLEN.
 */
int dora_select_compact(const float* scores, const int32_t* cu_in, const int32_t* keep_counts,
                        int32_t batch, int32_t max_seqlen, const dora_bf16* x, int32_t dim,
                        int32_t t_in_cap, const int32_t* ids_in, const float* mv_in,
                        int32_t* kept_idx, int32_t* cu_out, dora_bf16* packed,
                        int32_t* ids_out, float* mv_out, int32_t* status, dora_stream_t stream);

/*
 * dora_compact_ln -- dora_compact fused with the LayerNorm' that follows the
 * deletion in Eq. 1: also writes ln_out[r] = LayerNorm(packed[r]) with affine
 * ln_w, ln_b (bf16 [dim]) and epsilon eps (biased variance, fp32 statistics).
 * dim % 8 == 0 and dim <= 2048.
 */
int dora_compact_ln(const dora_bf16* x, int32_t dim, const int32_t* kept_idx,
                    const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                    const int32_t* ids_in, const dora_bf16* ln_w, const dora_bf16* ln_b,
                    float eps, dora_bf16* packed, int32_t* ids_out, dora_bf16* ln_out,
                    int32_t* status, dora_stream_t stream);

/*
 * dora_compact_stats -- dora_compact that also carries the row moments of
 * every kept row (see "LayerNorm folded into the linear after it" below):
 * mv_out[r] = mv_in[kept_idx[r]] (fp32 [t_in_cap, 2] each, 8-byte aligned),
 * the input of the LayerNorm' folded into fc1, bit for bit what the rows had
 * before the deletion.
 */
int dora_compact_stats(const dora_bf16* x, int32_t dim, const int32_t* kept_idx,
                       const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                       const int32_t* ids_in, const float* mv_in, dora_bf16* packed,
                       int32_t* ids_out, float* mv_out, int32_t* status, dora_stream_t stream);

/*
 * dora_layernorm -- y = LayerNorm(x) row by row (the LayerNorm of Eq. 1),
 * biased variance, fp32 statistics, affine w, b (bf16 [dim]).
 * rows_cap   rows the buffers hold; rows_dev (nullable) points at the live row
 *            count on the device (e.g. cu + batch); rows beyond it are skipped.
 * dim % 8 == 0 and dim <= 2048.
 */
int dora_layernorm(const dora_bf16* x, int32_t rows_cap, const int32_t* rows_dev, int32_t dim,
                   const dora_bf16* w, const dora_bf16* b, float eps, dora_bf16* y,
                   dora_stream_t stream);

/*
 * dora_linear -- y = epilogue(x W^T + b) on tcgen05 tensor cores, the QKV,
 * projection and MLP linears of Eq. 1 applied to the packed rows.
 * x          bf16 [m_cap, k] (16-byte aligned, k % 64 == 0).
 * m_dev      nullable: live row count on the device; rows >= it are neither
 *            computed nor written.  NULL means m_cap rows.
 * w          bf16 [n, k], nn.Linear layout (16-byte aligned, n % 32 == 0).
 * bias       nullable bf16 [n].
 * residual   bf16 [m_cap, n], required for DORA_EPI_BIAS_RESIDUAL; may not
 *            alias y.
 * y          out bf16 [m_cap, n].
 * Accumulation is fp32; the result is rounded once to bf16.
 */
int dora_linear(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                const dora_bf16* w, int32_t n, const dora_bf16* bias, const dora_bf16* residual,
                int32_t epilogue, dora_bf16* y, int32_t* status, dora_stream_t stream);

/*
 * LayerNorm folded into the linear after it.  The LayerNorm of Eq. 1 before
 * the QKV linear, and LayerNorm' before fc1, need only each row's mean and
 * rstd = 1/sqrt(var + eps) once the affine is moved into the weights:
 *     LayerNorm(x) W^T + b = rstd (x W'^T - mean c) + d,
 *     W' = W diag(gamma) rounded to bf16,  c = W' 1,  d = W beta + b,
 * exact algebra; the GEMM then reads the raw rows.  Two formats carry the row
 * statistics (fp32, from the bf16 values):
 *  - row moments mv [rows_cap, 2]: mv[2 r] = mean and mv[2 r + 1] = biased
 *    variance of row r (what dora_linear_ln reads);
 *  - slice moments sm [dim / 64, rows_cap, 2], slice-major: for row r and
 *    64-column slice s, sm[2 (s rows_cap + r)] = the slice's mean and
 *    sm[2 (s rows_cap + r) + 1] = the sum of squared deviations from it
 *    (what a residual GEMM epilogue can write, a row being split over
 *    several tiles).  dora_merge_moments turns them into row moments with the
 *    pairwise update of Chan, Golub & LeVeque.
 * rows_cap is the row capacity of the call that writes them (rows_cap, m_cap
 * or t_in_cap).
 */

/*
 * dora_row_stats -- row moments of bf16 rows x [rows_cap, dim] into mv
 * (fp32 [rows_cap, 2], 8-byte aligned).  rows_dev (nullable) is the live row
 * count on the device; rows beyond it are skipped.  dim % 8 == 0, dim <= 2048.
 */
int dora_row_stats(const dora_bf16* x, int32_t rows_cap, const int32_t* rows_dev, int32_t dim,
                   float* mv, dora_stream_t stream);

/*
 * dora_merge_moments -- row moments mv (fp32 [rows_cap, 2]) of rows whose
 * slice moments are sm (fp32 [slices, rows_cap, 2]): mean = (1/S) sum mean_s,
 * var = (sum M2_s + 64 sum (mean_s - mean)^2) / (64 S).  rows_dev as in
 * dora_row_stats.
 */
int dora_merge_moments(const float* sm, int32_t rows_cap, const int32_t* rows_dev,
                       int32_t slices, float* mv, dora_stream_t stream);

/*
 * dora_fold_ln_linear -- moves a LayerNorm affine (gamma, beta: bf16 [k])
 * into the linear W [n, k] (bias nullable bf16 [n]) that follows it:
 * w_out [n, k] = bf16(W diag(gamma)) (one rounding: the product of two bf16
 * values is exact in fp32), colsum fp32 [n] = row sums of w_out, colbias fp32
 * [n] = W beta + bias.  Done once per set of weights.  k % 8 == 0; all
 * pointers 16-byte aligned.
 */
int dora_fold_ln_linear(const dora_bf16* w, int32_t n, int32_t k, const dora_bf16* gamma,
                        const dora_bf16* beta, const dora_bf16* bias, dora_bf16* w_out,
                        float* colsum, float* colbias, dora_stream_t stream);

/*
 * dora_linear_ln -- y = LayerNorm(x) W^T + b, or its GELU when gelu != 0,
 * computed as rstd (x W'^T - mean c) + d with W', c (colsum), d (colbias)
 * from dora_fold_ln_linear and each row's mean and var from the row moments
 * mv of x (fp32 [m_cap, 2]; dora_row_stats, dora_merge_moments or
 * dora_compact_stats), rstd = 1/sqrt(var + eps).  eps is the LayerNorm
 * epsilon.  x [m_cap, k] with
 * k % 64 == 0, k <= 2048; n % 32 == 0; m_dev as in dora_linear.  fp32
 * accumulation and epilogue, one rounding to bf16.
 */
int dora_linear_ln(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                   const float* mv, float eps, const dora_bf16* w_folded, int32_t n,
                   const float* colsum, const float* colbias, int32_t gelu, dora_bf16* y,
                   int32_t* status, dora_stream_t stream);

/*
 * dora_linear_residual_stats -- dora_linear with DORA_EPI_BIAS_RESIDUAL that
 * also writes the slice moments of the rounded output rows to stats_out (fp32
 * [n / 64, m_cap, 2]; dora_merge_moments makes row moments of them), for the
 * folded LayerNorm that reads them next.  n % 64 == 0; live rows only.
 */
int dora_linear_residual_stats(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                               const dora_bf16* w, int32_t n, const dora_bf16* bias,
                               const dora_bf16* residual, dora_bf16* y, float* stats_out,
                               int32_t* status, dora_stream_t stream);

/*
 * dora_varlen_attn -- packed variable-length multi-head self-attention
 * (Sec. 3.5 "Inference": attention is confined to each image by the explicit
 * boundaries, no probability matrix is materialised, no token-size terms).
 * For image i and head h:  O = softmax(Q K^T * softmax_scale) V  over the
 * n_i rows of image i only.
 * qkv        bf16 [t_cap, 3, heads, head_dim] (row layout q | k | v).
 * cu_seqlens int32 [batch+1]; cu_seqlens[batch] <= t_cap.
 * max_seqlen upper bound of n_i; sizes the grid (an image longer than it is
 *            only partly computed and raises DORA_ERR_DEVICE_SEQLEN).
 * head_dim   must be 64.  softmax_scale 0 means 1/sqrt(head_dim).
 * out        out bf16 [t_cap, heads*head_dim]; rows >= cu_seqlens[batch] are
 *            not written.
 * fp32 scores and softmax statistics; P is rounded to bf16 for the PV product.
 */
int dora_varlen_attn(const dora_bf16* qkv, const int32_t* cu_seqlens, int32_t batch,
                     int32_t max_seqlen, int32_t t_cap, int32_t heads, int32_t head_dim,
                     float softmax_scale, dora_bf16* out, int32_t* status, dora_stream_t stream);

/*
 * dora_gather_scores -- row-aligned deletion scores from per-image tables
 * indexed by original token id: scores[r] = table[i * table_stride + ids[r]]
 * for every row r of image i.  This stands in for the actor's selector output
 * (Eq. 2) in synthetic workloads; it is not part of Eq. 1.
 * An id outside [0, table_stride) yields NaN and DORA_ERR_DEVICE_SEQLEN.
 */
int dora_gather_scores(const float* table, int32_t table_stride, const int32_t* ids,
                       const int32_t* cu, int32_t batch, float* scores, int32_t* status,
                       dora_stream_t stream);

/* Weights of one block, all bf16 device pointers, linears in nn.Linear layout
 * W[out, in]: w_qkv [3*dim, dim], w_proj [dim, dim], w_fc1 [mlp_dim, dim],
 * w_fc2 [dim, mlp_dim].  Biases may be NULL (zero). */
typedef struct dora_block_weights {
  const dora_bf16* ln1_w;
  const dora_bf16* ln1_b;
  const dora_bf16* w_qkv;
  const dora_bf16* b_qkv;
  const dora_bf16* w_proj;
  const dora_bf16* b_proj;
  const dora_bf16* ln2_w;
  const dora_bf16* ln2_b;
  const dora_bf16* w_fc1;
  const dora_bf16* b_fc1;
  const dora_bf16* w_fc2;
  const dora_bf16* b_fc2;
  int32_t dim;       /* D = heads * 64 */
  int32_t heads;
  int32_t mlp_dim;   /* multiple of 64 */
  float ln_eps;      /* LayerNorm epsilon, e.g. 1e-6 */
  /* Nullable: these weights with both LayerNorms folded in, written by
   * dora_fold_block_weights (256-byte aligned).  NULL = the block folds them
   * into its workspace on every call (same result, more work per call). */
  const void* folded;
} dora_block_weights;

/* Bytes of device workspace dora_pruned_block needs for t_cap rows (it
 * includes room for the folded weights when w->folded is NULL). */
size_t dora_workspace_size(int32_t t_cap, int32_t batch, const dora_block_weights* w);

/* Bytes dora_fold_block_weights writes for these weights. */
size_t dora_folded_weights_size(const dora_block_weights* w);

/*
 * dora_fold_block_weights -- folds LayerNorm (ln1_w, ln1_b) into the QKV
 * linear and LayerNorm' (ln2_w, ln2_b) into fc1 (dora_fold_ln_linear on
 * both), into `folded` (device, 256-byte aligned, folded_bytes >=
 * dora_folded_weights_size(w)).  Call once after loading the weights and put
 * the pointer in w->folded; refold whenever those weights change.
 */
int dora_fold_block_weights(const dora_block_weights* w, void* folded, size_t folded_bytes,
                            dora_stream_t stream);

/*
 * dora_pruned_block -- one block of Eq. 1 on the packed batch:
 *   row moments -> QKV linear with LN1 folded in -> varlen attention
 *     -> projection + residual (+ slice moments) -> merged moments  (H_attn)
 *   [select_keep -> compaction carrying the row moments]            (H_keep)
 *   fc1 with LN2 folded in + GELU -> fc2 + residual                 (H_next)
 * x_in      bf16 [t_cap, dim], rows [0, cu_in[batch]) live.
 * cu_in     int32 [batch+1]; ids_in int32 [t_cap] original token ids
 *           (nullable when scores is NULL).
 * scores    nullable fp32 [t_cap] deletion scores aligned with x_in rows.
 *           NULL = no deletion in this block (gate off for every image): then
 *           keep_counts, cu_out, ids_out and kept_idx are ignored and the
 *           output boundaries are cu_in.
 * keep_counts int32 [batch] tokens kept per image (CLS included).
 * x_out     out bf16 [t_cap, dim]; must not alias x_in.
 * cu_out    out int32 [batch+1]; ids_out out int32 [t_cap];
 * kept_idx  nullable out int32 [t_cap] (workspace is used when NULL).
 * x_in_moments   nullable fp32 [t_cap, 2]: row moments (mean, var) of x_in's
 *                live rows, e.g. the previous block's x_out_moments; NULL =
 *                computed here (one more pass over x_in).
 * x_out_moments  nullable out fp32 [t_cap, 2]: row moments of x_out's live
 *                rows, from fc2's residual epilogue, for the next block's
 *                x_in_moments.  May alias x_in_moments.
 * workspace device buffer of dora_workspace_size() bytes, 256-byte aligned;
 *           it also holds the status word read by dora_read_status.  It must
 *           be zero-filled once after allocation (rows past the live count
 *           are then always finite).
 * All counts after the deletion stay on the device; the call never
 * synchronises, so a sequence of blocks can be captured in a CUDA graph.
 */
int dora_pruned_block(const dora_bf16* x_in, const int32_t* cu_in, const int32_t* ids_in,
                      int32_t batch, int32_t max_seqlen, int32_t t_cap,
                      const dora_block_weights* w, const float* scores,
                      const int32_t* keep_counts, dora_bf16* x_out, int32_t* cu_out,
                      int32_t* ids_out, int32_t* kept_idx, const float* x_in_moments,
                      float* x_out_moments, void* workspace, size_t workspace_bytes,
                      dora_stream_t stream);

/* Device address of the status word inside a dora_pruned_block workspace. */
int32_t* dora_workspace_status(void* workspace);

/*
 * dora_pruned_block_noalloc -- dora_pruned_block for callers that cannot
 * allocate device memory.  The paper has no counterpart: this is a deployment
 * convenience of this library.
 *
 * Who needs it: code that must not call cudaMalloc at the point where it runs
 * the block -- paths that may never synchronise the device (cudaMalloc and
 * cudaFree can), plugins whose host framework owns all device memory and
 * forbids side allocations, processes that reserved the whole device up
 * front.  Such callers pass only inputs and outputs; the block's intermediates
 * live in a scratch array that the library itself holds in device memory.
 *
 * Arguments are those of dora_pruned_block minus the workspace, plus
 * `status` (nullable device int32) which receives the block's status word.
 *
 * Limits and behaviour:
 *  - The scratch array holds DORA_NOALLOC_SCRATCH_BYTES (32 MiB) on every GPU
 *    that loads the library, for the life of the process.  A block whose
 *    dora_workspace_size(t_cap, batch, w) exceeds it is rejected with
 *    DORA_ERR_SCRATCH_TOO_SMALL before anything is launched (32 MiB fits e.g.
 *    a DeiT-Tiny-shape batch of 8 x 197 tokens, or about 2,100 token rows of
 *    a DeiT-Base-shape block with pre-folded weights, 1,600 without).
 *  - The first call on a device looks up the device address of the scratch
 *    array (cudaGetSymbolAddress) with that device current; make that first
 *    call before any stream capture on the device.  The address is kept for
 *    the life of the process, so a cudaDeviceReset after that first call is
 *    not supported: the kept address may no longer be the array's.
 *  - No cudaMalloc, cudaFree or other allocating routine is called.
 *  - Every call on a device shares the same scratch, which keeps the previous
 *    call's contents: the status word in it is cleared at the start of each
 *    call and everything else is written before it is read.  Calls whose work
 *    overlaps on the GPU (different streams, or different host threads,
 *    without ordering between them) race on the scratch and give wrong
 *    results: order them on one stream.
 */
#define DORA_NOALLOC_SCRATCH_BYTES (32u << 20)
int dora_pruned_block_noalloc(const dora_bf16* x_in, const int32_t* cu_in,
                              const int32_t* ids_in, int32_t batch, int32_t max_seqlen,
                              int32_t t_cap, const dora_block_weights* w, const float* scores,
                              const int32_t* keep_counts, dora_bf16* x_out, int32_t* cu_out,
                              int32_t* ids_out, int32_t* kept_idx, const float* x_in_moments,
                              float* x_out_moments, int32_t* status, dora_stream_t stream);

/*
 * The deterministic actor (Sec. 3.2 "The actor"; Appendix A.1-A.3): at a
 * block it reads the block's keys and produces, for every image, the gate
 * decision, the removal count k_l and the deletion scores that
 * dora_select_keep consumes.
 *
 * dora_actor_weights -- bf16 device tensors of the actor, nn.Linear layout
 * [out, in], the shapes of Appendix A.1 (d = backbone width, L = depth,
 * M = (n0 - 4) / 2 budget-head outputs):
 *   gate: gate_w1 [64, d + 19], gate_b1 [64], gate_w2 [1, 64], gate_b2 [1],
 *         gate_emb [L, 16]  -- input order [K_CLS, e^G_l, h_l];
 *   encoder: enc_w_in [128, d], enc_b_in [128], enc_emb [L, 128],
 *         enc_w_h [128, 3], enc_ln1_w/b [128], enc_w_qkv [384, 128] (rows
 *         q, k, v, each four heads of 32), enc_b_qkv [384], enc_w_o [128, 128],
 *         enc_b_o [128], enc_ln2_w/b [128], enc_w_fc1 [256, 128],
 *         enc_b_fc1 [256], enc_w_fc2 [128, 256], enc_b_fc2 [128];
 *   budget head: bud_ln_w/b [128], bud_w1 [128, 128], bud_b1 [128],
 *         bud_w2 [M, 128], bud_b2 [M];
 *   selector: sel_w_k [128], sel_w1 [64, 128], sel_b1 [64], sel_w2 [1, 64],
 *         sel_b2 [1].
 * dim % 64 == 0, dim <= 2048; 6 <= n0 <= 1028; eps = the actor's LayerNorm
 * epsilon; prepared = NULL or the buffer dora_actor_prepare filled (the
 * encoder's folded and padded weights; without it every call rebuilds them
 * in its workspace).  Every pointer 16-byte aligned.
 */
typedef struct {
  const dora_bf16 *gate_w1, *gate_b1, *gate_w2, *gate_b2, *gate_emb;
  const dora_bf16 *enc_w_in, *enc_b_in, *enc_emb, *enc_w_h;
  const dora_bf16 *enc_ln1_w, *enc_ln1_b, *enc_w_qkv, *enc_b_qkv, *enc_w_o, *enc_b_o;
  const dora_bf16 *enc_ln2_w, *enc_ln2_b, *enc_w_fc1, *enc_b_fc1, *enc_w_fc2, *enc_b_fc2;
  const dora_bf16 *bud_ln_w, *bud_ln_b, *bud_w1, *bud_b1, *bud_w2, *bud_b2;
  const dora_bf16 *sel_w_k, *sel_w1, *sel_b1, *sel_w2, *sel_b2;
  int32_t dim, depth, n0;
  float eps;
  const void* prepared;
} dora_actor_weights;

/* Bytes dora_actor_prepare writes; bytes of workspace dora_actor needs for
 * t_cap rows and `batch` images (it includes the prepared weights when
 * w->prepared is NULL). */
size_t dora_actor_prepared_size(const dora_actor_weights* w);
size_t dora_actor_workspace_size(int32_t t_cap, int32_t batch, const dora_actor_weights* w);

/* Builds the encoder's device-side weights once: the per-block input bias
 * b_in + e^C_l (bf16), the QKV and feed-forward weights with their
 * LayerNorms folded in (as dora_fold_ln_linear), and the QKV rows and W_o
 * columns zero-padded from heads of 32 to heads of 64. */
int dora_actor_prepare(const dora_actor_weights* w, void* prepared, size_t prepared_bytes,
                       dora_stream_t stream);

/*
 * dora_actor -- the actor at block `block` (0 <= block < L) for the packed
 * batch.  qkv bf16 [t_cap, 3 dim] is the block's QKV output (its keys are
 * columns [dim, 2 dim), heads concatenated); cu int32 [batch + 1] the image
 * boundaries (row cu[i] is image i's CLS).  rho fp32 [batch] and
 * interventions int32 [batch] are each image's rho_l and E_<l (zeros at
 * block 0); n_l = cu[i+1] - cu[i] - 1 visual tokens.
 * Outputs per image: p_gate fp32 (nullable; the gate probability), gate
 * int32 (1 when p >= 0.5 and a budget is feasible), budget int32 (the
 * highest-logit budget with k <= n_l - 4, ties to the smaller, 0 if none),
 * k int32 (budget when the gate is open, else 0), keep_counts int32
 * (n_l + 1 - k, CLS included), rho_next fp32 and interventions_next int32
 * (nullable; the next block's history: k / n_l and E_<l + gate; may alias
 * rho and interventions).  scores fp32 [t_cap]: the selector's deletion
 * score of every visual row, computed with the image's budget (CLS rows 0).
 * z_out nullable bf16 [t_cap, 128]: the encoder output Z_l.
 * The encoder runs on bf16 GEMMs with fp32 accumulation (heads of 32
 * padded to the attention kernel's 64); gate, budget head and selector in
 * fp32.  The gate decision is the sign of the gate logit (p >= 0.5).
 * workspace: dora_actor_workspace_size bytes, 256-byte aligned; its first
 * word is the status word (dora_workspace_status).
 */
int dora_actor(const dora_bf16* qkv, const int32_t* cu, int32_t batch, int32_t max_seqlen,
               int32_t t_cap, int32_t block, const dora_actor_weights* w, const float* rho,
               const int32_t* interventions, float* p_gate, int32_t* gate, int32_t* budget,
               int32_t* k, int32_t* keep_counts, float* scores, float* rho_next,
               int32_t* interventions_next, dora_bf16* z_out, void* workspace,
               size_t workspace_bytes, dora_stream_t stream);

/*
 * dora_pruned_block_actor -- dora_pruned_block at block `block` with the
 * actor deciding the deletion (Sec. 3.2; Eq. 1): after the attention
 * residual, dora_actor runs on this block's own keys (the QKV linear's
 * output inside the workspace) and its deletion scores feed select_keep.
 * keep_counts NULL: the actor's keep counts are used (gate and budget
 * decide); otherwise these counts, with the actor's scores choosing which
 * tokens go.  The arguments after workspace_bytes are dora_actor's
 * (aw->dim == w->dim; gate, budget, k, actor_keep [batch], scores [t_cap]
 * required; rho_next, interventions_next nullable); the actor's status word
 * is the first word of actor_workspace.  cu_out, ids_in, ids_out required.
 */
int dora_pruned_block_actor(const dora_bf16* x_in, const int32_t* cu_in, const int32_t* ids_in,
                            int32_t batch, int32_t max_seqlen, int32_t t_cap,
                            const dora_block_weights* w, dora_bf16* x_out, int32_t* cu_out,
                            int32_t* ids_out, int32_t* kept_idx, const float* x_in_moments,
                            float* x_out_moments, void* workspace, size_t workspace_bytes,
                            const dora_actor_weights* aw, int32_t block, const float* rho,
                            const int32_t* interventions, const int32_t* keep_counts,
                            int32_t* gate, int32_t* budget, int32_t* k, int32_t* actor_keep,
                            float* scores, float* rho_next, int32_t* interventions_next,
                            void* actor_workspace, size_t actor_workspace_bytes,
                            dora_stream_t stream);

/*
 * The two ends of the forward, which the paper's GFLOPs and throughput count
 * (App. E.4): patch embedding and the classifier head.
 *
 * dora_patch_embed -- images bf16 [batch, channels, height, width] (NCHW) to
 * the packed tokens x0 bf16 [batch * (g + 1), dim], g = (height / patch) *
 * (width / patch): row 0 of each image is cls + pos[0], row 1 + p the patch
 * p (row-major over the patch grid) embedded by the patch x patch, stride
 * patch convolution (w_pe bf16 [dim, channels * patch * patch], the
 * [dim, C, p, p] kernel flattened; b_pe bf16 [dim], nullable) plus pos[1 + p]
 * (pos bf16 [g + 1, dim]; cls bf16 [dim]).  1 <= patch <= 64, 1 <= channels
 * <= 64, height and width multiples of patch, dim % 64 == 0.  The
 * convolution is a relayout (patchify) and one tcgen05 GEMM with fp32
 * accumulation (its output rounded to bf16), then the position add.  When
 * K = channels * patch^2 is not a multiple of 64 (DINOv2's 14-pixel patches:
 * K = 588) the patch matrix is K-padded with zero columns to the next
 * multiple of 64 and a zero-padded copy of w_pe is written to the workspace
 * on each call.  workspace: dora_embed_workspace_size bytes, 256-byte
 * aligned; its first word is a status word.
 */
size_t dora_embed_workspace_size(int32_t batch, int32_t channels, int32_t height, int32_t width,
                                 int32_t patch, int32_t dim);
int dora_patch_embed(const dora_bf16* images, int32_t batch, int32_t channels, int32_t height,
                     int32_t width, int32_t patch, int32_t dim, const dora_bf16* w_pe,
                     const dora_bf16* b_pe, const dora_bf16* cls, const dora_bf16* pos,
                     dora_bf16* x0, void* workspace, size_t workspace_bytes, dora_stream_t stream);

/*
 * dora_classifier_head -- logits bf16 [batch, classes] = LayerNorm(x[cu[i]])
 * W_head^T + b_head for each image i: the final LayerNorm (norm_w, norm_b
 * bf16 [dim], epsilon eps, biased variance, fp32) on the CLS row, then a
 * tcgen05 GEMM (w_head bf16 [classes, dim]; b_head bf16 [classes], nullable).
 * classes % 32 == 0 (pad the head with zero rows), dim % 64 == 0; x bf16
 * [t_cap, dim] packed, cu int32 [batch + 1].  An empty image gives the
 * logits of a zero row.  workspace: dora_head_workspace_size bytes,
 * 256-byte aligned, status word first.
 */
size_t dora_head_workspace_size(int32_t batch, int32_t dim);
int dora_classifier_head(const dora_bf16* x, const int32_t* cu, int32_t batch, int32_t t_cap,
                         int32_t dim, const dora_bf16* norm_w, const dora_bf16* norm_b,
                         float eps, const dora_bf16* w_head, const dora_bf16* b_head,
                         int32_t classes, dora_bf16* logits, void* workspace,
                         size_t workspace_bytes, dora_stream_t stream);

/*
 * DINOv2 backbones (App. E.3: register-free DINOv2-B/14 with its LC1 readout
 * and LayerScale kept).
 *
 * dora_classifier_head_lc1 -- logits bf16 [batch, classes] = u_i W_head^T +
 * b_head with u_i = [LN(x[cu[i]]), mean over j in (cu[i], cu[i+1]) of
 * LN(x[j])] (2 * dim features): the final LayerNorm (norm_w, norm_b bf16
 * [dim], epsilon eps, biased variance, fp32) applied to every surviving row,
 * CLS first, then the mean of the normalised visual rows (zero for an image
 * with only its CLS row; an empty image gives u = 0).  w_head bf16
 * [classes, 2 * dim], b_head bf16 [classes] (nullable), classes % 32 == 0,
 * dim % 64 == 0 and dim <= 2048; x bf16 [t_cap, dim] packed, cu int32
 * [batch + 1].  u is rounded to bf16 before the tcgen05 GEMM.  workspace:
 * dora_head_lc1_workspace_size bytes, 256-byte aligned, status word first
 * (DORA_ERR_DEVICE_SEQLEN for cu outside [0, t_cap]).
 */
size_t dora_head_lc1_workspace_size(int32_t batch, int32_t dim);
int dora_classifier_head_lc1(const dora_bf16* x, const int32_t* cu, int32_t batch, int32_t t_cap,
                             int32_t dim, const dora_bf16* norm_w, const dora_bf16* norm_b,
                             float eps, const dora_bf16* w_head, const dora_bf16* b_head,
                             int32_t classes, dora_bf16* logits, void* workspace,
                             size_t workspace_bytes, dora_stream_t stream);

/*
 * dora_fold_layerscale -- LayerScale (per-channel scale gamma on a residual
 * branch, x + gamma * (W h + b)) folded into the branch's last linear:
 * w_out[i, :] = bf16(gamma_i * w[i, :]), b_out[i] = bf16(gamma_i * b_i).
 * w, w_out bf16 [n, k] (nn.Linear layout, k % 8 == 0, 16-byte aligned;
 * w_out == w is allowed), gamma bf16 [n]; b and b_out bf16 [n], both null or
 * both set (b_out == b allowed).  Each output is the round-to-nearest-even of
 * the exact product.  Called once per block for the attention output and
 * fc2 linears; the folded weights then run through dora_pruned_block.
 */
int dora_fold_layerscale(const dora_bf16* w, const dora_bf16* b, const dora_bf16* gamma,
                         int32_t n, int32_t k, dora_bf16* w_out, dora_bf16* b_out,
                         dora_stream_t stream);

/*
 * Training side (App. A.3 "Training-time sampling and deterministic
 * inference"; App. B.2 "Shadow evaluation procedure").  Scores are fp32,
 * row-aligned with the packed tokens (cu int32 [batch + 1]); each image's CLS
 * row cu[i] takes no part, visual token j of image i is row cu[i] + 1 + j, and
 * an image holds at most 2048 visual tokens (longer: DORA_ERR_DEVICE_SEQLEN,
 * treated as empty).  Device errors go to *status (nullable device int32).
 *
 * dora_pl_sample -- the ordered removal sequence (i_1..i_k) of each image,
 * drawn without replacement from the Plackett-Luce distribution of its scores
 * as the Gumbel-top-k: the k_i largest keys s_j + g_j (fp32 sum; -0 == +0,
 * NaN above +inf, equal keys by higher j first) in decreasing order.  The
 * tie rule is dora_select_keep's, so the sampled set is exactly what the
 * block deletes when it is given the keys as its scores: keys_out fp32
 * [t_cap] (nullable) receives s + g on every visual row (the CLS row: s).
 * gumbel fp32 [t_cap] row-aligned standard Gumbel noise, drawn by the
 * caller; k int32 [batch] (device); order int32 [batch, k_cap] out:
 * order[i, t] = j of the (t+1)-th removal, -1 for t >= k_i.  k_i outside
 * [0, min(n_i, k_cap)] is clamped and raises DORA_ERR_DEVICE_BAD_COUNT.
 */
int dora_pl_sample(const float* scores, const float* gumbel, const int32_t* cu, int32_t batch,
                   int32_t t_cap, const int32_t* k, int32_t k_cap, int32_t* order,
                   float* keys_out, int32_t* status, dora_stream_t stream);

/*
 * dora_pl_logprob -- logp fp32 [batch]: log pi_S(i | k) = sum_t [s_{i_t} -
 * log sum_{j in R_t} exp(s_j)], R_t the visual tokens not removed before step
 * t (App. A.3), for the sequences in order int32 [batch, k_cap] (the first k_i
 * entries used).  grad fp32 [t_cap] (nullable): dlogp_i * d log pi / d s_j for
 * every visual row (CLS rows 0), dlogp fp32 [batch] (nullable: 1).  fp32,
 * log-sum-exp scans without cancellation.  A sequence entry outside
 * [0, n_i) or repeated gives logp NaN, NaN gradients and
 * DORA_ERR_DEVICE_BAD_COUNT.
 */
int dora_pl_logprob(const float* scores, const int32_t* cu, int32_t batch, int32_t t_cap,
                    const int32_t* k, const int32_t* order, int32_t k_cap, float* logp,
                    float* grad, const float* dlogp, int32_t* status, dora_stream_t stream);

/*
 * dora_branch -- complete-prefix shadows as extra sequences of the packed
 * batch (App. B.2): the rows of sequences src int32 [n_branch] (device, each
 * in [0, batch)) are copied, in order, after row cu[batch] of x bf16
 * [t_cap, dim] (in place), with their ids int32 [t_cap] and row moments
 * x_moments fp32 [t_cap, 2] (both nullable).  cu_out int32 [batch + 1 +
 * n_branch]: cu followed by the appended sequences' ends (cu_out == cu is
 * allowed when it has the room); len_out int32 [n_branch] (nullable): their
 * lengths, which are also their keep counts at every later block.  Rows past
 * t_cap are not written: the first appended sequence that does not fit, and
 * every one after it, gets length 0 (DORA_ERR_DEVICE_SEQLEN).
 */
int dora_branch(dora_bf16* x, int32_t* ids, float* x_moments, const int32_t* cu, int32_t batch,
                int32_t t_cap, int32_t dim, const int32_t* src, int32_t n_branch,
                int32_t* cu_out, int32_t* len_out, int32_t* status, dora_stream_t stream);

/*
 * dora_kd_cost -- cost fp32 [shadows]: D = tau^2 sum_c p^N_c log(p^N_c /
 * p_c), p^N = softmax(z_native[img] / tau), p = softmax(z[s] / tau) over the
 * first `classes` columns (App. B.2; tau = 3 there).  z_native bf16
 * [batch, ld], z bf16 [shadows, ld] (row pitch ld >= classes: padded heads);
 * shadow_image int32 [shadows] (device, nullable: shadow s compares with
 * image s); fp32 arithmetic.
 */
int dora_kd_cost(const dora_bf16* z_native, const dora_bf16* z, const int32_t* shadow_image,
                 int32_t shadows, int32_t batch, int32_t classes, int32_t ld, float tau,
                 float* cost, int32_t* status, dora_stream_t stream);

/*
 * dora_step_rewards -- local rewards of each image's actions (App. B.3):
 * r_j = 25 k_j (L - l_j) / (L N0) - a (D_j - D_{j-1}), D_{-1} = 0, for the
 * pruning blocks l_j = blocks[j] (int32 [n_blocks], device, increasing),
 * removals int32 [n_blocks, batch] (device; k = 0 at a gate-off step), L =
 * depth, N0 = n0 visual tokens, a the fidelity coefficient.  cost fp32 is the
 * fidelity-cost array of a batched shadow forward, [(n_blocks + 1) batch] in
 * sequence order: rollout (its D is that of the last pruning block), Native,
 * then the shadows of pruning blocks 0..n_blocks-2.  reward fp32 [n_blocks,
 * batch]; ret fp32 [batch] (nullable): the episode sum, which telescopes to
 * 25 C - a D_final.
 */
int dora_step_rewards(const float* cost, const int32_t* removals, const int32_t* blocks,
                      int32_t n_blocks, int32_t batch, int32_t depth, int32_t n0, float a,
                      float* reward, float* ret, dora_stream_t stream);

/* Synchronises the current device and copies the status word at `status_dev`
 * (a device int32, e.g. dora_workspace_status(ws)) to *code.  Test/debug
 * only: it blocks the host. */
int dora_read_status(const int32_t* status_dev, int32_t* code);

#ifdef __cplusplus
}
#endif

#endif /* DORA_H_ */
