// Launchers of the token kernels (selection, compaction, LayerNorm, gather).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dora {

// The current device if it is an sm_103 part; -1 when the query fails, -2
// for another architecture.
int checked_device();

// Launch with programmatic stream serialization (dependent launch; the kernel
// itself calls pdl_trigger / pdl_wait), unless DORA_NO_PDL is set.
bool pdl_enabled();
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

constexpr int kSelectThreads = 256;
constexpr int kRowThreads = 256;          // 8 rows per CTA, one warp per row
constexpr int kMaxChunksPerLane = 8;      // 16-byte chunks per lane: dim <= 2048
constexpr int kMaxDimRow = 32 * 8 * kMaxChunksPerLane;
// selection: keys and kept list of one image in shared memory (64 KB at the
// limit); the per-thread segment counts are packed into 16-bit halves
constexpr int kMaxSeqlenSelect = 32 * kSelectThreads;
constexpr int kSelectCtas = 512;          // fused compaction: CTAs in all, split over the images
constexpr int kSelectMaxSplits = 8;

cudaError_t launch_select_keep(const float* scores, const int32_t* cu_in,
                               const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                               int32_t* kept_idx, int32_t* cu_out, int32_t* status,
                               cudaStream_t stream);

// Selection fused with the compaction of the kept rows (ids_in/ids_out and
// mv_in/mv_out nullable in pairs): the same kept_idx and cu_out as
// launch_select_keep, then packed[r] = x[kept_idx[r]], ids and row moments.
// mv_slices = 0: mv_in holds row moments [t_in_cap][2], copied; mv_slices =
// S > 0: mv_in holds the rows' slice moments [S][t_in_cap][2], merged per
// kept row (the same bits as launch_merge_moments).
int select_compact_splits(int32_t batch, int32_t max_seqlen);
cudaError_t launch_select_compact(const float* scores, const int32_t* cu_in,
                                  const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                                  const uint16_t* x, int32_t dim, int32_t t_in_cap,
                                  const int32_t* ids_in, const float* mv_in, int32_t* kept_idx,
                                  int32_t* cu_out, uint16_t* packed, int32_t* ids_out,
                                  float* mv_out, int32_t* status, cudaStream_t stream,
                                  int32_t mv_slices = 0);

// ln_out (LayerNorm' of the kept rows) is nullable; so is mv_out, which
// receives mv_in[kept_idx[r]] (row moments, below) for every packed row r.
cudaError_t launch_compact(const uint16_t* x, int32_t dim, const int32_t* kept_idx,
                           const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                           const int32_t* ids_in, const uint16_t* ln_w, const uint16_t* ln_b,
                           float eps, uint16_t* packed, int32_t* ids_out, uint16_t* ln_out,
                           const float* mv_in, float* mv_out, int32_t* status,
                           cudaStream_t stream);

// The input side of a LayerNorm folded into the next linear.
// Row moments: mv[2 r] = mean and mv[2 r + 1] = biased variance of the bf16
// values of row r.
// Slice moments (written by the residual GEMM epilogue, where a row is split
// over several CTAs), slice-major: for row r of a buffer of rows_cap rows and
// 64-column slice s, sm[2 (s rows_cap + r)] is the slice's mean and
// sm[2 (s rows_cap + r) + 1] the sum of squared deviations from it.
constexpr int kSliceCols = 64;
cudaError_t launch_row_stats(const uint16_t* x, int32_t rows_cap, const int32_t* rows_dev,
                             int32_t dim, float* mv, cudaStream_t stream);
// row moments from slice moments (Chan, Golub & LeVeque's pairwise update)
cudaError_t launch_merge_moments(const float* sm, int32_t rows_cap, const int32_t* rows_dev,
                                 int32_t slices, float* mv, cudaStream_t stream);

// LayerNorm affine folded into a linear W [n, k]: w_out = bf16(W diag(gamma)),
// colsum = w_out 1, colbias = W beta + bias (bias nullable).
cudaError_t launch_fold_ln(const uint16_t* w, int32_t n, int32_t k, const uint16_t* gamma,
                           const uint16_t* beta, const uint16_t* bias, uint16_t* w_out,
                           float* colsum, float* colbias, cudaStream_t stream);

cudaError_t launch_layernorm(const uint16_t* x, int32_t rows_cap, const int32_t* rows_dev,
                             int32_t dim, const uint16_t* w, const uint16_t* b, float eps,
                             uint16_t* y, cudaStream_t stream);

cudaError_t launch_gather_scores(const float* table, int32_t stride, const int32_t* ids,
                                 const int32_t* cu, int32_t batch, float* scores, int32_t* status,
                                 cudaStream_t stream);

// tcgen05 GEMM: y = epi(x w^T ...); tensor maps are built inside.  Besides
// the public DORA_EPI_* epilogues, two with a LayerNorm folded in:
//   kEpiLn      y = rstd_r (x w'^T - mean_r colsum) + colbias
//   kEpiLnGelu  the same, then GELU
// with rstd_r = 1/sqrt(var_r + eps) from the row moments (stats_in).
constexpr int kEpiLn = 3;
constexpr int kEpiLnGelu = 4;
struct LinearEpi {
  const uint16_t* bias = nullptr;       // bf16 [n], nullable (plain epilogues)
  const uint16_t* residual = nullptr;   // bf16 [m, n] (residual epilogue)
  const float* stats_in = nullptr;      // row moments of x, [m_cap][2] (LN epilogues)
  const float* colsum = nullptr;        // fp32 [n] (LN epilogues)
  const float* colbias = nullptr;       // fp32 [n] (LN epilogues)
  float* stats_out = nullptr;           // slice moments of y, [n/64][m_cap], nullable
  float eps = 0.f;                      // LayerNorm epsilon (LN epilogues)
  int32_t slices = 0;                   // n / 64 (stats_out)
  int32_t m_reverse = 0;                // 1: walk the row blocks from the last one
};
// lda: row pitch of x in elements (0 = k; a multiple of 8).
cudaError_t launch_linear(const uint16_t* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                          const uint16_t* w, int32_t n, int32_t epilogue, const LinearEpi& ep,
                          uint16_t* y, int32_t* status, cudaStream_t stream, int32_t lda = 0);

// tcgen05 varlen attention.
cudaError_t launch_varlen_attn(const uint16_t* qkv, const int32_t* cu, int32_t batch,
                               int32_t max_seqlen, int32_t t_cap, int32_t heads, float scale,
                               uint16_t* out, int32_t* status, cudaStream_t stream);

// Tensor-map encoding through the driver entry point (no libcuda link).
// swizzle_bytes: 128 (default) or 64 (CU_TENSOR_MAP_SWIZZLE_128B / _64B).
int encode_tmap_2d_bf16(void* map, const void* base, uint64_t inner, uint64_t outer,
                        uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer,
                        int swizzle_bytes = 128);

int num_sms();

}  // namespace dora
