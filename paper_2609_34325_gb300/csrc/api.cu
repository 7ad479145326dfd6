// Host side of the C ABI declared in include/dora.h: argument validation,
// device checks, tensor-map encoding and the kernel sequence of one pruned
// block.  No entry point allocates memory or synchronises (except
// dora_read_status).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include <stdlib.h>

#include <mutex>

#include "dora.h"
#include "token_ops.cuh"

namespace dora {

namespace {

constexpr int kMaxDevices = 64;
int g_arch_ok[kMaxDevices];       // 0 unknown, 1 sm_103, -1 other
int g_num_sms[kMaxDevices];
std::mutex g_mu;

int current_device_checked() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return -1;
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_arch_ok[dev] == 0) {
    int major = 0, minor = 0, sms = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    g_arch_ok[dev] = (major == 10 && minor == 3) ? 1 : -1;
    g_num_sms[dev] = sms > 0 ? sms : 1;
  }
  return g_arch_ok[dev] == 1 ? dev : -2;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned8(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

}  // namespace

int checked_device() { return current_device_checked(); }

bool pdl_enabled() {
  static const bool on = getenv("DORA_NO_PDL") == nullptr;
  return on;
}

int num_sms() {
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= kMaxDevices || g_num_sms[dev] <= 0) return 148;
  return g_num_sms[dev];
}

int encode_tmap_2d_bf16(void* map, const void* base, uint64_t inner, uint64_t outer,
                        uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer,
                        int swizzle_bytes) {
  {
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_encode == nullptr) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                           &q) != cudaSuccess ||
          q != cudaDriverEntryPointSuccess || fn == nullptr)
        return -1;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
  }
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_pitch_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(reinterpret_cast<CUtensorMap*>(map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? 0 : static_cast<int>(r);
}

}  // namespace dora

using namespace dora;

#define DORA_CHECK_ARG(cond) \
  do {                       \
    if (!(cond)) return DORA_ERR_INVALID_ARG; \
  } while (0)

#define DORA_CHECK_DEVICE()                             \
  do {                                                  \
    const int _d = current_device_checked();            \
    if (_d == -1) return DORA_ERR_CUDA;                 \
    if (_d < 0) return DORA_ERR_UNSUPPORTED;            \
  } while (0)

static int cuda_status(cudaError_t e) { return e == cudaSuccess ? DORA_OK : DORA_ERR_CUDA; }

extern "C" {

const char* dora_status_string(int code) {
  switch (code) {
    case DORA_OK: return "ok";
    case DORA_ERR_INVALID_ARG: return "invalid argument";
    case DORA_ERR_UNSUPPORTED: return "unsupported (shape or device)";
    case DORA_ERR_CUDA: return "CUDA error";
    case DORA_ERR_TIMEOUT: return "device wait timed out";
    case DORA_ERR_DEVICE_BAD_COUNT: return "keep count out of range (clamped)";
    case DORA_ERR_DEVICE_SEQLEN: return "sequence longer than max_seqlen or index past capacity";
    case DORA_ERR_SCRATCH_TOO_SMALL: return "block needs more scratch than the no-alloc entry holds";
    default: return "unknown status";
  }
}

int dora_version(void) { return 2; }

int dora_select_keep(const float* scores, const int32_t* cu_in, const int32_t* keep_counts,
                     int32_t batch, int32_t max_seqlen, int32_t* kept_idx, int32_t* cu_out,
                     int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(batch >= 0 && batch <= (1 << 24));
  DORA_CHECK_ARG(max_seqlen >= 0 && max_seqlen <= kMaxSeqlenSelect);
  DORA_CHECK_ARG(cu_in && keep_counts && cu_out);
  DORA_CHECK_ARG(batch == 0 || (scores && kept_idx));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_select_keep(scores, cu_in, keep_counts, batch, max_seqlen, kept_idx,
                                        cu_out, status, reinterpret_cast<cudaStream_t>(stream)));
}

int dora_select_compact(const float* scores, const int32_t* cu_in, const int32_t* keep_counts,
                        int32_t batch, int32_t max_seqlen, const dora_bf16* x, int32_t dim,
                        int32_t t_in_cap, const int32_t* ids_in, const float* mv_in,
                        int32_t* kept_idx, int32_t* cu_out, dora_bf16* packed,
                        int32_t* ids_out, float* mv_out, int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(batch >= 0 && batch <= (1 << 24) && t_in_cap >= 0);
  DORA_CHECK_ARG(max_seqlen >= 0 && max_seqlen <= kMaxSeqlenSelect);
  DORA_CHECK_ARG(cu_in && keep_counts && cu_out);
  DORA_CHECK_ARG(batch == 0 || (scores && kept_idx));
  DORA_CHECK_ARG(dim > 0 && dim % 8 == 0 && dim <= kMaxDimRow);
  DORA_CHECK_ARG(t_in_cap == 0 || (x && packed));
  DORA_CHECK_ARG(aligned16(x) && aligned16(packed));
  DORA_CHECK_ARG((ids_in == nullptr) == (ids_out == nullptr));
  DORA_CHECK_ARG((mv_in == nullptr) == (mv_out == nullptr));
  DORA_CHECK_ARG(aligned8(mv_in) && aligned8(mv_out));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_select_compact(scores, cu_in, keep_counts, batch, max_seqlen,
                                           x, dim, t_in_cap, ids_in, mv_in, kept_idx, cu_out,
                                           packed, ids_out, mv_out, status,
                                           reinterpret_cast<cudaStream_t>(stream)));
}

static int compact_common(const dora_bf16* x, int32_t dim, const int32_t* kept_idx,
                          const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                          const int32_t* ids_in, const dora_bf16* ln_w, const dora_bf16* ln_b,
                          float eps, dora_bf16* packed, int32_t* ids_out, dora_bf16* ln_out,
                          const float* mv_in, float* mv_out, int32_t* status,
                          dora_stream_t stream) {
  DORA_CHECK_ARG(batch >= 0 && t_in_cap >= 0);
  DORA_CHECK_ARG(dim > 0 && dim % 8 == 0 && dim <= kMaxDimRow);
  DORA_CHECK_ARG(cu_out != nullptr);
  DORA_CHECK_ARG(t_in_cap == 0 || (x && kept_idx && packed));
  DORA_CHECK_ARG(aligned16(x) && aligned16(packed) && aligned16(ln_out));
  DORA_CHECK_ARG((ids_out == nullptr) || (ids_in != nullptr));
  if (ln_out) DORA_CHECK_ARG(ln_w && ln_b && aligned16(ln_w) && aligned16(ln_b) && eps >= 0.f);
  if (mv_out) DORA_CHECK_ARG(mv_in && aligned8(mv_in) && aligned8(mv_out));
  DORA_CHECK_DEVICE();
  if (t_in_cap == 0) return DORA_OK;
  return cuda_status(launch_compact(x, dim, kept_idx, cu_out, batch, t_in_cap, ids_in, ln_w, ln_b,
                                    eps, packed, ids_out, ln_out, mv_in, mv_out, status,
                                    reinterpret_cast<cudaStream_t>(stream)));
}

int dora_compact(const dora_bf16* x, int32_t dim, const int32_t* kept_idx, const int32_t* cu_out,
                 int32_t batch, int32_t t_in_cap, const int32_t* ids_in, dora_bf16* packed,
                 int32_t* ids_out, int32_t* status, dora_stream_t stream) {
  return compact_common(x, dim, kept_idx, cu_out, batch, t_in_cap, ids_in, nullptr, nullptr, 0.f,
                        packed, ids_out, nullptr, nullptr, nullptr, status, stream);
}

int dora_compact_stats(const dora_bf16* x, int32_t dim, const int32_t* kept_idx,
                       const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                       const int32_t* ids_in, const float* mv_in, dora_bf16* packed,
                       int32_t* ids_out, float* mv_out, int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(mv_in != nullptr && mv_out != nullptr);
  return compact_common(x, dim, kept_idx, cu_out, batch, t_in_cap, ids_in, nullptr, nullptr, 0.f,
                        packed, ids_out, nullptr, mv_in, mv_out, status, stream);
}

int dora_compact_ln(const dora_bf16* x, int32_t dim, const int32_t* kept_idx,
                    const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                    const int32_t* ids_in, const dora_bf16* ln_w, const dora_bf16* ln_b,
                    float eps, dora_bf16* packed, int32_t* ids_out, dora_bf16* ln_out,
                    int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(ln_out != nullptr);
  return compact_common(x, dim, kept_idx, cu_out, batch, t_in_cap, ids_in, ln_w, ln_b, eps,
                        packed, ids_out, ln_out, nullptr, nullptr, status, stream);
}

int dora_layernorm(const dora_bf16* x, int32_t rows_cap, const int32_t* rows_dev, int32_t dim,
                   const dora_bf16* w, const dora_bf16* b, float eps, dora_bf16* y,
                   dora_stream_t stream) {
  DORA_CHECK_ARG(rows_cap >= 0);
  DORA_CHECK_ARG(dim > 0 && dim % 8 == 0 && dim <= kMaxDimRow);
  DORA_CHECK_ARG(rows_cap == 0 || (x && y));
  DORA_CHECK_ARG(w && b && eps >= 0.f);
  DORA_CHECK_ARG(aligned16(x) && aligned16(y) && aligned16(w) && aligned16(b));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_layernorm(x, rows_cap, rows_dev, dim, w, b, eps, y,
                                      reinterpret_cast<cudaStream_t>(stream)));
}

int dora_linear(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                const dora_bf16* w, int32_t n, const dora_bf16* bias, const dora_bf16* residual,
                int32_t epilogue, dora_bf16* y, int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(m_cap >= 0 && m_cap <= (1 << 30) / 1);
  DORA_CHECK_ARG(k > 0 && k % 64 == 0 && k <= (1 << 16));
  DORA_CHECK_ARG(n > 0 && n % 32 == 0 && n <= (1 << 16));
  DORA_CHECK_ARG(epilogue >= DORA_EPI_BIAS && epilogue <= DORA_EPI_BIAS_RESIDUAL);
  DORA_CHECK_ARG(w && y && (m_cap == 0 || x));
  DORA_CHECK_ARG(aligned16(x) && aligned16(w) && aligned16(y) && aligned16(bias) &&
                 aligned16(residual));
  if (epilogue == DORA_EPI_BIAS_RESIDUAL) DORA_CHECK_ARG(residual && residual != y);
  DORA_CHECK_DEVICE();
  LinearEpi ep;
  ep.bias = bias;
  ep.residual = epilogue == DORA_EPI_BIAS_RESIDUAL ? residual : nullptr;
  return cuda_status(launch_linear(x, m_cap, m_dev, k, w, n, epilogue, ep, y, status,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

int dora_linear_residual_stats(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                               const dora_bf16* w, int32_t n, const dora_bf16* bias,
                               const dora_bf16* residual, dora_bf16* y, float* stats_out,
                               int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(m_cap >= 0 && m_cap <= (1 << 30));
  DORA_CHECK_ARG(k > 0 && k % 64 == 0 && k <= (1 << 16));
  DORA_CHECK_ARG(n > 0 && n % 64 == 0 && n <= (1 << 16));
  DORA_CHECK_ARG(w && y && residual && stats_out && residual != y && (m_cap == 0 || x));
  DORA_CHECK_ARG(aligned16(x) && aligned16(w) && aligned16(y) && aligned16(bias) &&
                 aligned16(residual) && aligned8(stats_out));
  DORA_CHECK_DEVICE();
  LinearEpi ep;
  ep.bias = bias;
  ep.residual = residual;
  ep.stats_out = stats_out;
  ep.slices = n / kSliceCols;
  return cuda_status(launch_linear(x, m_cap, m_dev, k, w, n, DORA_EPI_BIAS_RESIDUAL, ep, y, status,
                                   reinterpret_cast<cudaStream_t>(stream)));
}

int dora_row_stats(const dora_bf16* x, int32_t rows_cap, const int32_t* rows_dev, int32_t dim,
                   float* mv, dora_stream_t stream) {
  DORA_CHECK_ARG(rows_cap >= 0);
  DORA_CHECK_ARG(dim > 0 && dim % 8 == 0 && dim <= kMaxDimRow);
  DORA_CHECK_ARG(rows_cap == 0 || (x && mv));
  DORA_CHECK_ARG(aligned16(x) && aligned8(mv));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_row_stats(x, rows_cap, rows_dev, dim, mv,
                                      reinterpret_cast<cudaStream_t>(stream)));
}

int dora_merge_moments(const float* sm, int32_t rows_cap, const int32_t* rows_dev,
                       int32_t slices, float* mv, dora_stream_t stream) {
  DORA_CHECK_ARG(rows_cap >= 0 && slices > 0 && slices <= (1 << 16) / kSliceCols);
  DORA_CHECK_ARG(rows_cap == 0 || (sm && mv));
  DORA_CHECK_ARG(aligned8(sm) && aligned8(mv));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_merge_moments(sm, rows_cap, rows_dev, slices, mv,
                                          reinterpret_cast<cudaStream_t>(stream)));
}

int dora_fold_ln_linear(const dora_bf16* w, int32_t n, int32_t k, const dora_bf16* gamma,
                        const dora_bf16* beta, const dora_bf16* bias, dora_bf16* w_out,
                        float* colsum, float* colbias, dora_stream_t stream) {
  DORA_CHECK_ARG(n >= 0 && n <= (1 << 16) && k > 0 && k % 8 == 0 && k <= (1 << 16));
  DORA_CHECK_ARG(n == 0 || (w && gamma && beta && w_out && colsum && colbias));
  DORA_CHECK_ARG(aligned16(w) && aligned16(gamma) && aligned16(beta) && aligned16(w_out) &&
                 aligned16(colsum) && aligned16(colbias));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_fold_ln(w, n, k, gamma, beta, bias, w_out, colsum, colbias,
                                    reinterpret_cast<cudaStream_t>(stream)));
}

int dora_linear_ln(const dora_bf16* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                   const float* mv, float eps, const dora_bf16* w_folded, int32_t n,
                   const float* colsum, const float* colbias, int32_t gelu, dora_bf16* y,
                   int32_t* status, dora_stream_t stream) {
  DORA_CHECK_ARG(m_cap >= 0 && m_cap <= (1 << 30));
  DORA_CHECK_ARG(k > 0 && k % 64 == 0 && k <= kMaxDimRow);
  DORA_CHECK_ARG(n > 0 && n % 32 == 0 && n <= (1 << 16));
  DORA_CHECK_ARG(eps >= 0.f && isfinite(eps));
  DORA_CHECK_ARG(w_folded && y && colsum && colbias && (m_cap == 0 || (x && mv)));
  DORA_CHECK_ARG(aligned16(x) && aligned16(w_folded) && aligned16(y) && aligned16(colsum) &&
                 aligned16(colbias) && aligned8(mv));
  DORA_CHECK_DEVICE();
  LinearEpi ep;
  ep.stats_in = mv;
  ep.colsum = colsum;
  ep.colbias = colbias;
  ep.eps = eps;
  return cuda_status(launch_linear(x, m_cap, m_dev, k, w_folded, n, gelu ? kEpiLnGelu : kEpiLn, ep,
                                   y, status, reinterpret_cast<cudaStream_t>(stream)));
}

int dora_varlen_attn(const dora_bf16* qkv, const int32_t* cu_seqlens, int32_t batch,
                     int32_t max_seqlen, int32_t t_cap, int32_t heads, int32_t head_dim,
                     float softmax_scale, dora_bf16* out, int32_t* status, dora_stream_t stream) {
  if (head_dim != 64) return DORA_ERR_UNSUPPORTED;
  DORA_CHECK_ARG(batch >= 0 && batch <= 65535);
  DORA_CHECK_ARG(heads > 0 && heads <= 65535 && heads * 64 * 3 <= (1 << 16));
  DORA_CHECK_ARG(max_seqlen >= 0 && t_cap >= 0);
  DORA_CHECK_ARG(softmax_scale >= 0.f && isfinite(softmax_scale));
  DORA_CHECK_ARG(cu_seqlens && (t_cap == 0 || (qkv && out)));
  DORA_CHECK_ARG(aligned16(qkv) && aligned16(out));
  DORA_CHECK_DEVICE();
  const float scale = softmax_scale == 0.f ? 0.125f : softmax_scale;
  return cuda_status(launch_varlen_attn(qkv, cu_seqlens, batch, max_seqlen, t_cap, heads, scale,
                                        out, status, reinterpret_cast<cudaStream_t>(stream)));
}

int dora_gather_scores(const float* table, int32_t table_stride, const int32_t* ids,
                       const int32_t* cu, int32_t batch, float* scores, int32_t* status,
                       dora_stream_t stream) {
  DORA_CHECK_ARG(batch >= 0 && table_stride > 0);
  DORA_CHECK_ARG(cu && (batch == 0 || (table && ids && scores)));
  DORA_CHECK_DEVICE();
  return cuda_status(launch_gather_scores(table, table_stride, ids, cu, batch, scores, status,
                                          reinterpret_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------------------------
// workspace and the pruned block
// ---------------------------------------------------------------------------
namespace {
size_t up256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

// The two linears with a LayerNorm folded in: W' = W diag(gamma) (bf16),
// c = W' 1 and d = W beta + b (fp32).
struct FoldLayout {
  size_t wqkv, cqkv, dqkv, wfc1, cfc1, dfc1, total;
};

FoldLayout fold_layout(const dora_block_weights* w) {
  FoldLayout F{};
  const size_t d = static_cast<size_t>(w->dim), f = static_cast<size_t>(w->mlp_dim);
  size_t off = 0;
  F.wqkv = off; off += up256(3 * d * d * 2);
  F.cqkv = off; off += up256(3 * d * 4);
  F.dqkv = off; off += up256(3 * d * 4);
  F.wfc1 = off; off += up256(f * d * 2);
  F.cfc1 = off; off += up256(f * 4);
  F.dfc1 = off; off += up256(f * 4);
  F.total = off;
  return F;
}

cudaError_t fold_block(const dora_block_weights* w, uint8_t* fold, cudaStream_t stream) {
  const FoldLayout F = fold_layout(w);
  const int d = w->dim;
  cudaError_t e = launch_fold_ln(w->w_qkv, 3 * d, d, w->ln1_w, w->ln1_b, w->b_qkv,
                                 reinterpret_cast<uint16_t*>(fold + F.wqkv),
                                 reinterpret_cast<float*>(fold + F.cqkv),
                                 reinterpret_cast<float*>(fold + F.dqkv), stream);
  if (e != cudaSuccess) return e;
  return launch_fold_ln(w->w_fc1, w->mlp_dim, d, w->ln2_w, w->ln2_b, w->b_fc1,
                        reinterpret_cast<uint16_t*>(fold + F.wfc1),
                        reinterpret_cast<float*>(fold + F.cfc1),
                        reinterpret_cast<float*>(fold + F.dfc1), stream);
}

struct WsLayout {
  size_t status, sm, mv, mv2, qkv, o, hattn, hkeep, kept, u, fold, total;
};

WsLayout ws_layout(int32_t t_cap, const dora_block_weights* w) {
  WsLayout L{};
  const size_t t = static_cast<size_t>(t_cap), d = static_cast<size_t>(w->dim);
  size_t off = 0;
  L.status = off; off += 256;
  L.sm = off;     off += up256(t * (d / kSliceCols) * 8);
  L.mv = off;     off += up256(t * 8);
  L.mv2 = off;    off += up256(t * 8);
  L.qkv = off;    off += up256(t * 3 * d * 2);
  L.o = off;      off += up256(t * d * 2);
  L.hattn = off;  off += up256(t * d * 2);
  L.hkeep = off;  off += up256(t * d * 2);
  L.kept = off;   off += up256(t * 4);
  L.u = off;      off += up256(t * static_cast<size_t>(w->mlp_dim) * 2);
  L.fold = off;   off += w->folded != nullptr ? 0 : fold_layout(w).total;
  L.total = off;
  return L;
}

bool weights_ok(const dora_block_weights* w) {
  if (!w) return false;
  if (w->dim <= 0 || w->heads <= 0 || w->dim != w->heads * 64) return false;
  if (w->dim > kMaxDimRow || w->mlp_dim <= 0 || w->mlp_dim % 64 != 0) return false;
  if (!(w->ln_eps >= 0.f)) return false;
  const void* req[] = {w->ln1_w, w->ln1_b, w->w_qkv, w->w_proj, w->ln2_w, w->ln2_b, w->w_fc1,
                       w->w_fc2};
  for (const void* p : req)
    if (!p || !aligned16(p)) return false;
  const void* opt[] = {w->b_qkv, w->b_proj, w->b_fc1, w->b_fc2};
  for (const void* p : opt)
    if (!aligned16(p)) return false;
  if ((reinterpret_cast<uintptr_t>(w->folded) & 255u) != 0) return false;
  return true;
}
}  // namespace

size_t dora_folded_weights_size(const dora_block_weights* w) {
  if (!w || w->dim <= 0 || w->mlp_dim <= 0) return 0;
  return fold_layout(w).total;
}

int dora_fold_block_weights(const dora_block_weights* w, void* folded, size_t folded_bytes,
                            dora_stream_t stream) {
  DORA_CHECK_ARG(weights_ok(w) && folded != nullptr);
  DORA_CHECK_ARG((reinterpret_cast<uintptr_t>(folded) & 255u) == 0);
  DORA_CHECK_ARG(folded_bytes >= fold_layout(w).total);
  DORA_CHECK_DEVICE();
  return cuda_status(fold_block(w, static_cast<uint8_t*>(folded),
                                reinterpret_cast<cudaStream_t>(stream)));
}

size_t dora_workspace_size(int32_t t_cap, int32_t batch, const dora_block_weights* w) {
  (void)batch;
  if (t_cap < 0 || !w || w->dim <= 0 || w->mlp_dim <= 0) return 0;
  return ws_layout(t_cap, w).total;
}

int32_t* dora_workspace_status(void* workspace) { return static_cast<int32_t*>(workspace); }

// The actor run inside the block (dora_pruned_block_actor): its scores and,
// unless the caller gives keep counts, its keep counts drive the deletion.
struct ActorHook {
  const dora_actor_weights* aw;
  int32_t block;
  const float* rho;
  const int32_t* interventions;
  int32_t *gate, *budget, *k, *keep;
  float* scores;
  float* rho_next;
  int32_t* interventions_next;
  void* ws;
  size_t ws_bytes;
};

static int pruned_block_impl(const dora_bf16* x_in, const int32_t* cu_in, const int32_t* ids_in,
                             int32_t batch, int32_t max_seqlen, int32_t t_cap,
                             const dora_block_weights* w, const float* scores,
                             const int32_t* keep_counts, dora_bf16* x_out, int32_t* cu_out,
                             int32_t* ids_out, int32_t* kept_idx, const float* x_in_moments,
                             float* x_out_moments, void* workspace, size_t workspace_bytes,
                             dora_stream_t stream_, const ActorHook* hook) {
  DORA_CHECK_ARG(weights_ok(w));
  DORA_CHECK_ARG(batch >= 0 && batch <= 65535 && t_cap >= 0 && max_seqlen >= 0);
  DORA_CHECK_ARG(max_seqlen <= kMaxSeqlenSelect);
  DORA_CHECK_ARG(x_in && x_out && cu_in && workspace && x_in != x_out);
  DORA_CHECK_ARG(aligned16(x_in) && aligned16(x_out));
  DORA_CHECK_ARG((reinterpret_cast<uintptr_t>(workspace) & 255u) == 0);
  DORA_CHECK_ARG(aligned8(x_in_moments) && aligned8(x_out_moments));
  if (scores) DORA_CHECK_ARG(keep_counts && cu_out && ids_in && ids_out);
  if (hook) DORA_CHECK_ARG(!scores && cu_out && ids_in && ids_out && hook->scores && hook->keep);
  const WsLayout L = ws_layout(t_cap, w);
  DORA_CHECK_ARG(workspace_bytes >= L.total);
  DORA_CHECK_DEVICE();
  if (t_cap == 0 || batch == 0) return DORA_OK;

  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* status = reinterpret_cast<int32_t*>(ws + L.status);
  float* sm = reinterpret_cast<float*>(ws + L.sm);
  float* mv = reinterpret_cast<float*>(ws + L.mv);
  float* mv2 = reinterpret_cast<float*>(ws + L.mv2);
  uint16_t* qkv = reinterpret_cast<uint16_t*>(ws + L.qkv);
  uint16_t* o = reinterpret_cast<uint16_t*>(ws + L.o);
  uint16_t* hattn = reinterpret_cast<uint16_t*>(ws + L.hattn);
  uint16_t* hkeep = reinterpret_cast<uint16_t*>(ws + L.hkeep);
  int32_t* kept = kept_idx ? kept_idx : reinterpret_cast<int32_t*>(ws + L.kept);
  uint16_t* u = reinterpret_cast<uint16_t*>(ws + L.u);
  const int d = w->dim;
  const int32_t* rows_in = cu_in + batch;

  // LayerNorm and LayerNorm' ride in the QKV and fc1 linears (folded weights,
  // made here unless the caller folded them once with dora_fold_block_weights)
  uint8_t* fold = ws + L.fold;
  if (w->folded != nullptr) fold = static_cast<uint8_t*>(const_cast<void*>(w->folded));
  else if (fold_block(w, fold, stream) != cudaSuccess) return DORA_ERR_CUDA;
  const FoldLayout F = fold_layout(w);
  LinearEpi e_qkv, e_proj, e_fc1, e_fc2;
  e_qkv.stats_in = x_in_moments ? x_in_moments : mv;
  e_fc1.stats_in = (scores || hook) ? mv2 : mv;      // the kept rows' moments after a deletion
  e_qkv.eps = e_fc1.eps = w->ln_eps;
  e_proj.slices = d / kSliceCols;
  e_qkv.colsum = reinterpret_cast<const float*>(fold + F.cqkv);
  e_qkv.colbias = reinterpret_cast<const float*>(fold + F.dqkv);
  e_fc1.colsum = reinterpret_cast<const float*>(fold + F.cfc1);
  e_fc1.colbias = reinterpret_cast<const float*>(fold + F.dfc1);
  e_proj.bias = w->b_proj;
  e_proj.residual = x_in;
  e_proj.stats_out = sm;
  e_fc2.bias = w->b_fc2;
  e_fc2.stats_out = x_out_moments ? sm : nullptr;   // merged into x_out_moments
  e_fc2.slices = d / kSliceCols;
  // Each linear walks its row blocks the other way from the one whose output
  // it reads (QKV and fc1 forward, proj and fc2 from the last row block): the
  // rows written last are still in L2 when the reader starts.  1% of the
  // DeiT-B forward, same results.
  e_proj.m_reverse = 1;
  e_fc2.m_reverse = 1;

  // H_attn = H + Attention(LayerNorm(H))
  if (x_in_moments == nullptr &&
      launch_row_stats(x_in, t_cap, rows_in, d, mv, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  if (launch_linear(x_in, t_cap, rows_in, d, reinterpret_cast<const uint16_t*>(fold + F.wqkv),
                    3 * d, kEpiLn, e_qkv, qkv, status, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  if (launch_varlen_attn(qkv, cu_in, batch, max_seqlen, t_cap, w->heads, 0.125f, o, status,
                         stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  if (launch_linear(o, t_cap, rows_in, d, w->w_proj, d, DORA_EPI_BIAS_RESIDUAL, e_proj, hattn,
                    status, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  // LayerNorm' reads the row moments of H_attn; with a deletion only the kept
  // rows', which the compaction merges from the slice moments itself
  const bool deleting = scores != nullptr || hook != nullptr;
  if (!deleting &&
      launch_merge_moments(sm, t_cap, rows_in, d / kSliceCols, mv, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  // the actor reads this block's keys (Sec. 3.2; deletion follows the
  // attention residual, Eq. 1)
  if (hook != nullptr) {
    const int rc = dora_actor(qkv, cu_in, batch, max_seqlen, t_cap, hook->block, hook->aw,
                              hook->rho, hook->interventions, nullptr, hook->gate, hook->budget,
                              hook->k, hook->keep, hook->scores, hook->rho_next,
                              hook->interventions_next, nullptr, hook->ws, hook->ws_bytes,
                              stream_);
    if (rc != DORA_OK) return rc;
    scores = hook->scores;
    if (keep_counts == nullptr) keep_counts = hook->keep;
  }
  // H_keep: delete and compact, carrying the row moments of LayerNorm'
  const uint16_t* hk = hattn;
  const int32_t* rows_mid = rows_in;
  if (scores) {
    if (launch_select_compact(scores, cu_in, keep_counts, batch, max_seqlen, hattn, d, t_cap,
                              ids_in, sm, kept, cu_out, hkeep, ids_out, mv2, status, stream,
                              d / kSliceCols) != cudaSuccess)
      return DORA_ERR_CUDA;
    hk = hkeep;
    rows_mid = cu_out + batch;
  }
  // H_next = H_keep + MLP(LayerNorm'(H_keep))
  e_fc2.residual = hk;
  if (launch_linear(hk, t_cap, rows_mid, d, reinterpret_cast<const uint16_t*>(fold + F.wfc1),
                    w->mlp_dim, kEpiLnGelu, e_fc1, u, status, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  if (launch_linear(u, t_cap, rows_mid, w->mlp_dim, w->w_fc2, d, DORA_EPI_BIAS_RESIDUAL, e_fc2,
                    x_out, status, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  if (x_out_moments != nullptr &&
      launch_merge_moments(sm, t_cap, rows_mid, d / kSliceCols, x_out_moments, stream) !=
          cudaSuccess)
    return DORA_ERR_CUDA;
  return DORA_OK;
}

int dora_pruned_block(const dora_bf16* x_in, const int32_t* cu_in, const int32_t* ids_in,
                      int32_t batch, int32_t max_seqlen, int32_t t_cap,
                      const dora_block_weights* w, const float* scores,
                      const int32_t* keep_counts, dora_bf16* x_out, int32_t* cu_out,
                      int32_t* ids_out, int32_t* kept_idx, const float* x_in_moments,
                      float* x_out_moments, void* workspace, size_t workspace_bytes,
                      dora_stream_t stream) {
  return pruned_block_impl(x_in, cu_in, ids_in, batch, max_seqlen, t_cap, w, scores, keep_counts,
                           x_out, cu_out, ids_out, kept_idx, x_in_moments, x_out_moments,
                           workspace, workspace_bytes, stream, nullptr);
}

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
                            dora_stream_t stream) {
  DORA_CHECK_ARG(aw != nullptr && aw->dim == (w ? w->dim : -1));
  const ActorHook hook{aw, block, rho, interventions, gate, budget, k, actor_keep, scores,
                       rho_next, interventions_next, actor_workspace, actor_workspace_bytes};
  return pruned_block_impl(x_in, cu_in, ids_in, batch, max_seqlen, t_cap, w, nullptr,
                           keep_counts, x_out, cu_out, ids_out, kept_idx, x_in_moments,
                           x_out_moments, workspace, workspace_bytes, stream, &hook);
}

int dora_read_status(const int32_t* status_dev, int32_t* code) {
  DORA_CHECK_ARG(status_dev && code);
  if (cudaDeviceSynchronize() != cudaSuccess) return DORA_ERR_CUDA;
  if (cudaMemcpy(code, status_dev, sizeof(int32_t), cudaMemcpyDeviceToHost) != cudaSuccess)
    return DORA_ERR_CUDA;
  return DORA_OK;
}

}  // extern "C"
