// Launchers of the token kernels (selection, compaction, LayerNorm, gather).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace dora {

constexpr int kSelectThreads = 256;
constexpr int kRowThreads = 256;          // 8 rows per CTA, one warp per row
constexpr int kMaxChunksPerLane = 8;      // 16-byte chunks per lane: dim <= 2048
constexpr int kMaxDimRow = 32 * 8 * kMaxChunksPerLane;
constexpr int kMaxSeqlenSelect = 32 * kSelectThreads;   // one 32-bit mask per thread

cudaError_t launch_select_keep(const float* scores, const int32_t* cu_in,
                               const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                               int32_t* kept_idx, int32_t* cu_out, int32_t* status,
                               cudaStream_t stream);

cudaError_t launch_compact(const uint16_t* x, int32_t dim, const int32_t* kept_idx,
                           const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                           const int32_t* ids_in, const uint16_t* ln_w, const uint16_t* ln_b,
                           float eps, uint16_t* packed, int32_t* ids_out, uint16_t* ln_out,
                           int32_t* status, cudaStream_t stream);

cudaError_t launch_layernorm(const uint16_t* x, int32_t rows_cap, const int32_t* rows_dev,
                             int32_t dim, const uint16_t* w, const uint16_t* b, float eps,
                             uint16_t* y, cudaStream_t stream);

cudaError_t launch_gather_scores(const float* table, int32_t stride, const int32_t* ids,
                                 const int32_t* cu, int32_t batch, float* scores, int32_t* status,
                                 cudaStream_t stream);

// tcgen05 GEMM: y = epi(x w^T + b); tensor maps are built inside.
cudaError_t launch_linear(const uint16_t* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                          const uint16_t* w, int32_t n, const uint16_t* bias,
                          const uint16_t* residual, int32_t epilogue, uint16_t* y,
                          int32_t* status, cudaStream_t stream);

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
