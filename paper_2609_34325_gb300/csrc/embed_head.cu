// The two ends of the ViT forward, which the paper's GFLOPs and throughput
// include (App. E.4 "GFLOPs accounting"; backbones of Sec. 4.1):
//   patch embedding   a patch x patch convolution with stride patch, as
//                     patchify (a pure relayout) + one tcgen05 GEMM, then each
//                     image's CLS token prepended and the position embeddings
//                     added, into the packed token layout of the blocks;
//   classifier head   the final LayerNorm on each image's CLS row and the
//                     linear layer to the class logits (tcgen05 GEMM).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dora.h"
#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace embed {

__device__ __forceinline__ float lo_f(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_f(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ uint4 add8(uint4 a, uint4 b) {
  return make_uint4(pack2(lo_f(a.x) + lo_f(b.x), hi_f(a.x) + hi_f(b.x)),
                    pack2(lo_f(a.y) + lo_f(b.y), hi_f(a.y) + hi_f(b.y)),
                    pack2(lo_f(a.z) + lo_f(b.z), hi_f(a.z) + hi_f(b.z)),
                    pack2(lo_f(a.w) + lo_f(b.w), hi_f(a.w) + hi_f(b.w)));
}

// images [B, C, H, W] -> patches [B * gh * gw, C * p * p], 8 pixels (16 bytes)
// a thread: row = b * gh * gw + (y / p) * gw + x / p, column = c * p * p +
// (y % p) * p + x % p.  The weights [d, C, p, p] flattened are the GEMM's B.
__global__ void patchify_kernel(const uint4* __restrict__ img, int batch, int ch, int h, int w,
                                int p, uint4* __restrict__ out) {
  const int gw = w / p, gh = h / p;
  const long long segs = static_cast<long long>(batch) * ch * h * (w / 8);
  const int kcols8 = ch * p * p / 8;
  for (long long s = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; s < segs;
       s += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int xs = static_cast<int>(s % (w / 8));
    long long r = s / (w / 8);
    const int y = static_cast<int>(r % h);
    r /= h;
    const int c = static_cast<int>(r % ch);
    const int b = static_cast<int>(r / ch);
    const int x = xs * 8;
    const long long row = (static_cast<long long>(b) * gh + y / p) * gw + x / p;
    const int col8 = (c * p * p + (y % p) * p + x % p) / 8;
    out[row * kcols8 + col8] = img[s];
  }
}

// x0 row b * (g + 1) + j: j = 0 -> cls + pos[0]; else emb[b * g + j - 1] + pos[j].
__global__ void assemble_kernel(const uint4* __restrict__ emb, const uint4* __restrict__ cls,
                                const uint4* __restrict__ pos, int batch, int g, int dim8,
                                uint4* __restrict__ x0) {
  const long long total = static_cast<long long>(batch) * (g + 1) * dim8;
  for (long long s = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; s < total;
       s += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(s % dim8);
    const long long row = s / dim8;
    const int j = static_cast<int>(row % (g + 1));
    const long long b = row / (g + 1);
    const uint4 base = j == 0 ? cls[c] : emb[(b * g + j - 1) * dim8 + c];
    x0[s] = add8(base, pos[static_cast<long long>(j) * dim8 + c]);
  }
}

// LayerNorm of each image's CLS row (row cu[i]) into u [batch, dim]: one warp
// per image, fp32, biased variance.
__global__ void cls_ln_kernel(const uint16_t* __restrict__ x, const int32_t* __restrict__ cu,
                              int batch, int t_cap, int dim, const uint16_t* __restrict__ gam,
                              const uint16_t* __restrict__ bet, float eps,
                              uint16_t* __restrict__ u, int32_t* status) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= batch) return;
  const int r = cu[warp];
  uint16_t* ur = u + static_cast<size_t>(warp) * dim;
  if (r < 0 || r >= t_cap || cu[warp + 1] <= r) {   // empty image or outside the buffer
    if (lane == 0 && (r < 0 || r > t_cap)) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    for (int c = lane; c < dim; c += 32) ur[c] = 0;
    return;
  }
  const uint16_t* xr = x + static_cast<size_t>(r) * dim;
  float s = 0.f;
  for (int c = lane; c < dim; c += 32) s += __uint_as_float(static_cast<uint32_t>(xr[c]) << 16);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  const float mean = s / dim;
  float q = 0.f;
  for (int c = lane; c < dim; c += 32) {
    const float v = __uint_as_float(static_cast<uint32_t>(xr[c]) << 16) - mean;
    q += v * v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
  const float rstd = rsqrtf(q / dim + eps);
  for (int c = lane; c < dim; c += 32) {
    const float v = (__uint_as_float(static_cast<uint32_t>(xr[c]) << 16) - mean) * rstd *
                        __uint_as_float(static_cast<uint32_t>(gam[c]) << 16) +
                    __uint_as_float(static_cast<uint32_t>(bet[c]) << 16);
    const __nv_bfloat16 hv = __float2bfloat16_rn(v);
    ur[c] = *reinterpret_cast<const uint16_t*>(&hv);
  }
}

size_t up256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

int grid_for(long long work) {
  const long long g = (work + 255) / 256;
  return static_cast<int>(g < 152LL * 16 ? (g > 0 ? g : 1) : 152LL * 16);
}

}  // namespace embed
}  // namespace dora

using namespace dora;

extern "C" {

size_t dora_embed_workspace_size(int32_t batch, int32_t channels, int32_t height, int32_t width,
                                 int32_t patch, int32_t dim) {
  if (batch < 0 || channels <= 0 || patch <= 0 || height <= 0 || width <= 0 || dim <= 0) return 0;
  const size_t tok = static_cast<size_t>(batch) * (height / patch) * (width / patch);
  return 256 + embed::up256(tok * channels * patch * patch * 2) + embed::up256(tok * dim * 2);
}

int dora_patch_embed(const dora_bf16* images, int32_t batch, int32_t channels, int32_t height,
                     int32_t width, int32_t patch, int32_t dim, const dora_bf16* w_pe,
                     const dora_bf16* b_pe, const dora_bf16* cls, const dora_bf16* pos,
                     dora_bf16* x0, void* workspace, size_t workspace_bytes,
                     dora_stream_t stream_) {
  if (batch < 0 || batch > 65535 || channels <= 0 || patch <= 0 || patch % 8 != 0 ||
      height <= 0 || width <= 0 || height % patch != 0 || width % patch != 0 || dim <= 0 ||
      dim % 64 != 0 || dim > (1 << 16) || (channels * patch * patch) % 64 != 0)
    return DORA_ERR_INVALID_ARG;
  const void* req[] = {images, w_pe, cls, pos, x0, workspace};
  for (const void* p : req)
    if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0) return DORA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(b_pe) & 15u) != 0) return DORA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return DORA_ERR_INVALID_ARG;
  if (workspace_bytes < dora_embed_workspace_size(batch, channels, height, width, patch, dim))
    return DORA_ERR_INVALID_ARG;
  const long long g = static_cast<long long>(height / patch) * (width / patch);
  const long long tok = static_cast<long long>(batch) * g;
  if (tok > (1 << 30)) return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  if (batch == 0) return DORA_OK;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  const int k = channels * patch * patch;
  uint16_t* patches = reinterpret_cast<uint16_t*>(ws + 256);
  uint16_t* emb = reinterpret_cast<uint16_t*>(ws + 256 + embed::up256(tok * k * 2));
  const long long segs = static_cast<long long>(batch) * channels * height * (width / 8);
  embed::patchify_kernel<<<embed::grid_for(segs), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(images), batch, channels, height, width, patch,
      reinterpret_cast<uint4*>(patches));
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  LinearEpi ep;
  ep.bias = b_pe;
  if (launch_linear(patches, static_cast<int32_t>(tok), nullptr, k, w_pe, dim, DORA_EPI_BIAS, ep,
                    emb, status, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  const long long total = static_cast<long long>(batch) * (g + 1) * (dim / 8);
  embed::assemble_kernel<<<embed::grid_for(total), 256, 0, stream>>>(
      reinterpret_cast<const uint4*>(emb), reinterpret_cast<const uint4*>(cls),
      reinterpret_cast<const uint4*>(pos), batch, static_cast<int>(g), dim / 8,
      reinterpret_cast<uint4*>(x0));
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

size_t dora_head_workspace_size(int32_t batch, int32_t dim) {
  if (batch < 0 || dim <= 0) return 0;
  return 256 + embed::up256(static_cast<size_t>(batch) * dim * 2);
}

int dora_classifier_head(const dora_bf16* x, const int32_t* cu, int32_t batch, int32_t t_cap,
                         int32_t dim, const dora_bf16* norm_w, const dora_bf16* norm_b,
                         float eps, const dora_bf16* w_head, const dora_bf16* b_head,
                         int32_t classes, dora_bf16* logits, void* workspace,
                         size_t workspace_bytes, dora_stream_t stream_) {
  if (batch < 0 || batch > 65535 || t_cap < 0 || dim <= 0 || dim % 64 != 0 ||
      dim > (1 << 16) || classes <= 0 || classes % 32 != 0 || classes > (1 << 16) ||
      !(eps >= 0.f))
    return DORA_ERR_INVALID_ARG;
  const void* req[] = {x, cu, norm_w, norm_b, w_head, logits, workspace};
  for (const void* p : req)
    if (p == nullptr) return DORA_ERR_INVALID_ARG;
  const void* al[] = {x, norm_w, norm_b, w_head, b_head, logits};
  for (const void* p : al)
    if ((reinterpret_cast<uintptr_t>(p) & 15u) != 0) return DORA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 ||
      workspace_bytes < dora_head_workspace_size(batch, dim))
    return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  if (batch == 0) return DORA_OK;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  uint16_t* u = reinterpret_cast<uint16_t*>(ws + 256);
  embed::cls_ln_kernel<<<(batch + 7) / 8, 256, 0, stream>>>(x, cu, batch, t_cap, dim, norm_w,
                                                            norm_b, eps, u, status);
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  LinearEpi ep;
  ep.bias = b_head;
  return launch_linear(u, batch, nullptr, dim, w_head, classes, DORA_EPI_BIAS, ep, logits, status,
                       stream) == cudaSuccess
             ? DORA_OK
             : DORA_ERR_CUDA;
}

}  // extern "C"
