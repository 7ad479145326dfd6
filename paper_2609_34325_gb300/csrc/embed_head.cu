// The two ends of the ViT forward, which the paper's GFLOPs and throughput
// include (App. E.4 "GFLOPs accounting"; backbones of Sec. 4.1):
//   patch embedding   a patch x patch convolution with stride patch, as
//                     patchify (a pure relayout) + one tcgen05 GEMM, then each
//                     image's CLS token prepended and the position embeddings
//                     added, into the packed token layout of the blocks;
//   classifier head   the final LayerNorm on each image's CLS row and the
//                     linear layer to the class logits (tcgen05 GEMM);
//   LC1 head          DINOv2's readout (App. E.3): the final LayerNorm on every
//                     surviving token, normalised CLS ++ the mean of the
//                     normalised visual rows of each image, then the linear
//                     layer on the 2 d features;
//   LayerScale fold   DINOv2's per-channel branch scales folded once into the
//                     rows of the attention output and fc2 linears.
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

// Any patch side: one thread writes 8 consecutive columns of one row of the
// K-padded patch matrix [B gh gw, kpad] (2-byte gathers; columns >= C p^2 are
// zero).  Column order as above: c * p * p + dy * p + dx.
__global__ void patchify_any_kernel(const uint16_t* __restrict__ img, int batch, int ch, int h,
                                    int w, int p, int kpad, uint4* __restrict__ out) {
  const int gw = w / p, gh = h / p, pp = p * p, k = ch * pp, kp8 = kpad / 8;
  const long long total = static_cast<long long>(batch) * gh * gw * kp8;
  for (long long s = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; s < total;
       s += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int c8 = static_cast<int>(s % kp8);
    long long r = s / kp8;
    const int gx = static_cast<int>(r % gw);
    r /= gw;
    const int gy = static_cast<int>(r % gh);
    const long long b = r / gh;
    uint32_t v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      uint32_t pair = 0;
#pragma unroll
      for (int hlf = 0; hlf < 2; ++hlf) {
        const int col = c8 * 8 + 2 * e + hlf;
        if (col < k) {
          const int c = col / pp, rem = col - c * pp, dy = rem / p, dx = rem - dy * p;
          const long long pix =
              ((b * ch + c) * h + gy * p + dy) * static_cast<long long>(w) + gx * p + dx;
          pair |= static_cast<uint32_t>(img[pix]) << (16 * hlf);
        }
      }
      v[e] = pair;
    }
    out[s] = make_uint4(v[0], v[1], v[2], v[3]);
  }
}

// Even patch side (DINOv2's 14): one thread writes one 4-byte pixel pair of
// the K-padded patch matrix, consecutive threads consecutive pairs of a
// token row, so every store is coalesced; the pair (an even pair never
// straddles two patches) is read from the image, pad pairs are zero.  All
// counts fit in 32 bits (checked by the caller).
__global__ void patchify_even_kernel(const uint32_t* __restrict__ img, int batch, int ch, int h,
                                     int w, int p, int kpad, uint32_t* __restrict__ out) {
  const int gw = w / p, gh = h / p, p2 = p / 2, row2 = p * p2, k2 = ch * row2, w2 = w / 2;
  const int kp2 = kpad / 2;
  const int total = batch * gh * gw * kp2;
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < total; s += gridDim.x * blockDim.x) {
    const int q = s % kp2, tok = s / kp2;
    uint32_t v = 0u;
    if (q < k2) {
      const int c = q / row2, rem = q - c * row2, dy = rem / p2, e = rem - dy * p2;
      const int gx = tok % gw, t2 = tok / gw, gy = t2 % gh, b = t2 / gh;
      v = __ldg(img + (static_cast<size_t>((b * ch + c) * h + gy * p + dy) * w2 + gx * p2 + e));
    }
    out[s] = v;
  }
}

// The same relayout with the patch side and channel count fixed at compile
// time (DINOv2-B/14 on RGB), staged through shared memory: one block per
// band of patches (image b, patch row gy).  The band's CH x P image rows are
// read with coalesced 16-byte loads, then its gw token rows are written with
// coalesced 16-byte stores, each 8-column piece gathered from shared memory
// (column c P^2 + dy P + dx, zero past CH P^2).  Needs w % 8 == 0.
template <int P, int CH>
__global__ void __launch_bounds__(256)
    patchify_band_kernel(const uint4* __restrict__ img, int gh, int gw, int h, int w,
                         uint4* __restrict__ out) {
  extern __shared__ uint16_t band[];                   // [CH][P][w]
  constexpr int kK = CH * P * P, kKp8 = (kK + 63) / 64 * 8;
  const int gy = blockIdx.x % gh, b = blockIdx.x / gh;
  const int w8 = w / 8;
  uint4* band4 = reinterpret_cast<uint4*>(band);
  for (int i = threadIdx.x; i < CH * P * w8; i += blockDim.x) {
    const int x8 = i % w8, r = i / w8, dy = r % P, c = r / P;
    band4[i] = __ldg(img + (static_cast<size_t>((b * CH + c) * h + gy * P + dy) * w8 + x8));
  }
  __syncthreads();
  uint4* dst = out + static_cast<size_t>(blockIdx.x) * gw * kKp8;
  for (int i = threadIdx.x; i < gw * kKp8; i += blockDim.x) {
    const int gx = i / kKp8, c8 = i - gx * kKp8;
    uint32_t v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      uint32_t pr = 0u;
#pragma unroll
      for (int hlf = 0; hlf < 2; ++hlf) {
        const int col = c8 * 8 + 2 * e + hlf;
        if (col < kK) {
          const int c = col / (P * P), rem = col - c * (P * P), dy = rem / P, dx = rem - dy * P;
          pr |= static_cast<uint32_t>(band[(c * P + dy) * w + gx * P + dx]) << (16 * hlf);
        }
      }
      v[e] = pr;
    }
    dst[i] = make_uint4(v[0], v[1], v[2], v[3]);
  }
}

// w [d, k] -> [d, kpad] with zero columns k..kpad-1 (the GEMM's B for K-padded patches).
__global__ void pad_cols_kernel(const uint16_t* __restrict__ w, int d, int k, int kpad,
                                uint16_t* __restrict__ out) {
  const long long total = static_cast<long long>(d) * kpad;
  for (long long s = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; s < total;
       s += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int j = static_cast<int>(s % kpad);
    out[s] = j < k ? w[(s / kpad) * k + j] : static_cast<uint16_t>(0);
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

// LC1 readout of one image per CTA (8 warps): rows lo..hi-1 of x are layer-
// normalised (fp32, biased variance, row held in registers: dim <= 2048); the
// CLS row goes to u[i, 0:d], the others are summed per lane in registers and
// their mean goes to u[i, d:2d] (zero for an image without visual rows).
constexpr int kLc1Warps = 8;
constexpr int kLc1MaxDim = 2048;

// kChunks = 16-byte pieces of a row per lane (dim <= 256 kChunks).
template <int kChunks>
__global__ void __launch_bounds__(kLc1Warps * 32)
    lc1_pool_kernel(const uint16_t* __restrict__ x, const int32_t* __restrict__ cu, int t_cap,
                    int dim, const uint16_t* __restrict__ gam, const uint16_t* __restrict__ bet,
                    float eps, uint16_t* __restrict__ u, int32_t* status) {
  extern __shared__ float acc[];                 // [kLc1Warps][dim]
  const int img = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int d8 = dim / 8;
  const int lo = cu[img], hi = cu[img + 1];
  uint16_t* ur = u + static_cast<size_t>(img) * 2 * dim;
  const bool bad = lo < 0 || hi < lo || hi > t_cap;
  if (bad || hi == lo) {
    if (bad && threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    for (int c = threadIdx.x; c < 2 * dim; c += blockDim.x) ur[c] = 0;
    return;
  }
  // Each lane owns the columns of its chunks c8 = lane + 32 i in every row,
  // so the visual rows' normalised values x^ = (x - mean) rstd are summed in
  // its registers; the affine map is applied once at the end, to the mean
  // (mean of g x^ + b = g mean(x^) + b).  Each warp walks rows lo + warp,
  // lo + warp + 8, ...; the next row's loads are issued before the current
  // row is reduced.
  float accr[kChunks][8];
#pragma unroll
  for (int i = 0; i < kChunks; ++i)
#pragma unroll
    for (int e = 0; e < 8; ++e) accr[i][e] = 0.f;
  uint4 nxt[kChunks];
  auto load_row = [&](int j, uint4 (&q)[kChunks]) {
    const uint4* xr = reinterpret_cast<const uint4*>(x + static_cast<size_t>(j) * dim);
#pragma unroll
    for (int i = 0; i < kChunks; ++i) {
      const int c8 = lane + 32 * i;
      q[i] = (j < hi && c8 < d8) ? xr[c8] : make_uint4(0, 0, 0, 0);
    }
  };
  load_row(lo + warp, nxt);
  for (int j = lo + warp; j < hi; j += kLc1Warps) {
    uint4 q[kChunks];
#pragma unroll
    for (int i = 0; i < kChunks; ++i) q[i] = nxt[i];
    load_row(j + kLc1Warps, nxt);
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < kChunks; ++i)
      s += lo_f(q[i].x) + hi_f(q[i].x) + lo_f(q[i].y) + hi_f(q[i].y) + lo_f(q[i].z) +
           hi_f(q[i].z) + lo_f(q[i].w) + hi_f(q[i].w);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = s / dim;
    float v2 = 0.f;
#pragma unroll
    for (int i = 0; i < kChunks; ++i) {
      if (lane + 32 * i >= d8) continue;
      const uint32_t wv[4] = {q[i].x, q[i].y, q[i].z, q[i].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = lo_f(wv[e]) - mean, b = hi_f(wv[e]) - mean;
        v2 += a * a + b * b;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v2 += __shfl_xor_sync(0xffffffffu, v2, o);
    const float rstd = rsqrtf(v2 / dim + eps);
    if (j == lo) {                                       // CLS row: LN(x) itself
#pragma unroll
      for (int i = 0; i < kChunks; ++i) {
        const int c8 = lane + 32 * i;
        if (c8 >= d8) continue;
        const uint32_t wv[4] = {q[i].x, q[i].y, q[i].z, q[i].w};
        const uint4 g4 = reinterpret_cast<const uint4*>(gam)[c8];
        const uint4 b4 = reinterpret_cast<const uint4*>(bet)[c8];
        const uint32_t gv[4] = {g4.x, g4.y, g4.z, g4.w}, bv[4] = {b4.x, b4.y, b4.z, b4.w};
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e)
          o[e] = pack2((lo_f(wv[e]) - mean) * rstd * lo_f(gv[e]) + lo_f(bv[e]),
                       (hi_f(wv[e]) - mean) * rstd * hi_f(gv[e]) + hi_f(bv[e]));
        reinterpret_cast<uint4*>(ur)[c8] = make_uint4(o[0], o[1], o[2], o[3]);
      }
    } else {
#pragma unroll
      for (int i = 0; i < kChunks; ++i) {
        const uint32_t wv[4] = {q[i].x, q[i].y, q[i].z, q[i].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          accr[i][2 * e] += (lo_f(wv[e]) - mean) * rstd;
          accr[i][2 * e + 1] += (hi_f(wv[e]) - mean) * rstd;
        }
      }
    }
  }
#pragma unroll
  for (int i = 0; i < kChunks; ++i) {
    const int c8 = lane + 32 * i;
    if (c8 >= d8) continue;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[warp * dim + c8 * 8 + e] = accr[i][e];
  }
  __syncthreads();
  const int n_vis = hi - lo - 1;
  const float inv = n_vis > 0 ? 1.f / static_cast<float>(n_vis) : 0.f;
  for (int c = threadIdx.x; c < dim; c += blockDim.x) {
    float t = 0.f;
#pragma unroll
    for (int wp = 0; wp < kLc1Warps; ++wp) t += acc[wp * dim + c];
    const float g = __uint_as_float(static_cast<uint32_t>(gam[c]) << 16);
    const float b = __uint_as_float(static_cast<uint32_t>(bet[c]) << 16);
    const __nv_bfloat16 hv = __float2bfloat16_rn(n_vis > 0 ? t * inv * g + b : 0.f);
    ur[dim + c] = *reinterpret_cast<const uint16_t*>(&hv);
  }
}

// LayerScale fold: out[i, :] = bf16(gamma_i * w[i, :]) and bout[i] =
// bf16(gamma_i * b_i).  A product of two bf16 values is exact in fp32, so each
// output is the round-to-nearest-even of the exact product.
__global__ void layerscale_fold_kernel(const uint4* __restrict__ w, const uint16_t* __restrict__ b,
                                       const uint16_t* __restrict__ gam, int n, int k8,
                                       uint4* __restrict__ out, uint16_t* __restrict__ bout) {
  const long long total = static_cast<long long>(n) * k8;
  for (long long s = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; s < total;
       s += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int row = static_cast<int>(s / k8);
    const float g = __uint_as_float(static_cast<uint32_t>(gam[row]) << 16);
    const uint4 v = w[s];
    out[s] = make_uint4(pack2(g * lo_f(v.x), g * hi_f(v.x)), pack2(g * lo_f(v.y), g * hi_f(v.y)),
                        pack2(g * lo_f(v.z), g * hi_f(v.z)), pack2(g * lo_f(v.w), g * hi_f(v.w)));
    if (b != nullptr && s % k8 == 0) {
      const __nv_bfloat16 hv = __float2bfloat16_rn(g * __uint_as_float(
                                                           static_cast<uint32_t>(b[row]) << 16));
      bout[row] = *reinterpret_cast<const uint16_t*>(&hv);
    }
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
  const size_t k = static_cast<size_t>(channels) * patch * patch, kpad = (k + 63) / 64 * 64;
  return 256 + embed::up256(tok * kpad * 2) + embed::up256(tok * dim * 2) +
         (kpad != k ? embed::up256(static_cast<size_t>(dim) * kpad * 2) : 0);
}

int dora_patch_embed(const dora_bf16* images, int32_t batch, int32_t channels, int32_t height,
                     int32_t width, int32_t patch, int32_t dim, const dora_bf16* w_pe,
                     const dora_bf16* b_pe, const dora_bf16* cls, const dora_bf16* pos,
                     dora_bf16* x0, void* workspace, size_t workspace_bytes,
                     dora_stream_t stream_) {
  if (batch < 0 || batch > 65535 || channels <= 0 || channels > 64 || patch <= 0 ||
      patch > 64 || height <= 0 || width <= 0 || height % patch != 0 || width % patch != 0 ||
      dim <= 0 || dim % 64 != 0 || dim > (1 << 16))
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
  const int k = channels * patch * patch, kpad = (k + 63) / 64 * 64;
  uint16_t* patches = reinterpret_cast<uint16_t*>(ws + 256);
  uint16_t* emb = reinterpret_cast<uint16_t*>(ws + 256 + embed::up256(tok * kpad * 2));
  const uint16_t* w_gemm = w_pe;
  if (patch % 8 == 0 && kpad == k) {
    const long long segs = static_cast<long long>(batch) * channels * height * (width / 8);
    embed::patchify_kernel<<<embed::grid_for(segs), 256, 0, stream>>>(
        reinterpret_cast<const uint4*>(images), batch, channels, height, width, patch,
        reinterpret_cast<uint4*>(patches));
  } else {
    // K padded to a multiple of the GEMM's 64-wide K step: zero patch columns
    // and a zero-padded copy of the weights in the workspace
    uint16_t* wp = reinterpret_cast<uint16_t*>(ws + 256 + embed::up256(tok * kpad * 2) +
                                               embed::up256(tok * dim * 2));
    const long long items = tok * (kpad / 2);
    const int band_smem = 3 * 14 * width * 2;
    if (patch == 14 && channels == 3 && width % 8 == 0 && band_smem <= 160 * 1024 &&
        static_cast<long long>(batch) * (height / patch) < (1LL << 31)) {
      auto kern = embed::patchify_band_kernel<14, 3>;
      if (band_smem > 48 * 1024 &&
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, band_smem) !=
              cudaSuccess)
        return DORA_ERR_CUDA;
      kern<<<static_cast<unsigned>(batch * (height / patch)), 256, band_smem, stream>>>(
          reinterpret_cast<const uint4*>(images), height / patch, width / patch, height, width,
          reinterpret_cast<uint4*>(patches));
    } else if (patch % 2 == 0 && items < (1LL << 31) &&
               static_cast<long long>(batch) * channels * height * width / 2 < (1LL << 31)) {
      embed::patchify_even_kernel<<<embed::grid_for(items), 256, 0, stream>>>(
          reinterpret_cast<const uint32_t*>(images), batch, channels, height, width, patch, kpad,
          reinterpret_cast<uint32_t*>(patches));
    } else {
      const long long segs = tok * (kpad / 8);
      embed::patchify_any_kernel<<<embed::grid_for(segs), 256, 0, stream>>>(
          images, batch, channels, height, width, patch, kpad, reinterpret_cast<uint4*>(patches));
    }
    if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
    if (kpad != k) {
      embed::pad_cols_kernel<<<embed::grid_for(static_cast<long long>(dim) * kpad), 256, 0,
                               stream>>>(w_pe, dim, k, kpad, wp);
      w_gemm = wp;
    }
  }
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  LinearEpi ep;
  ep.bias = b_pe;
  if (launch_linear(patches, static_cast<int32_t>(tok), nullptr, kpad, w_gemm, dim, DORA_EPI_BIAS,
                    ep, emb, status, stream) != cudaSuccess)
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

size_t dora_head_lc1_workspace_size(int32_t batch, int32_t dim) {
  if (batch < 0 || dim <= 0) return 0;
  return 256 + embed::up256(static_cast<size_t>(batch) * 2 * dim * 2);
}

int dora_classifier_head_lc1(const dora_bf16* x, const int32_t* cu, int32_t batch, int32_t t_cap,
                             int32_t dim, const dora_bf16* norm_w, const dora_bf16* norm_b,
                             float eps, const dora_bf16* w_head, const dora_bf16* b_head,
                             int32_t classes, dora_bf16* logits, void* workspace,
                             size_t workspace_bytes, dora_stream_t stream_) {
  if (batch < 0 || batch > 65535 || t_cap < 0 || dim <= 0 || dim % 64 != 0 ||
      dim > embed::kLc1MaxDim || classes <= 0 || classes % 32 != 0 || classes > (1 << 16) ||
      !(eps >= 0.f))
    return DORA_ERR_INVALID_ARG;
  const void* req[] = {x, cu, norm_w, norm_b, w_head, logits, workspace};
  for (const void* p : req)
    if (p == nullptr) return DORA_ERR_INVALID_ARG;
  const void* al[] = {x, norm_w, norm_b, w_head, b_head, logits};
  for (const void* p : al)
    if ((reinterpret_cast<uintptr_t>(p) & 15u) != 0) return DORA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 ||
      workspace_bytes < dora_head_lc1_workspace_size(batch, dim))
    return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  if (batch == 0) return DORA_OK;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* status = reinterpret_cast<int32_t*>(ws);
  uint16_t* u = reinterpret_cast<uint16_t*>(ws + 256);
  const int smem = embed::kLc1Warps * dim * 4;
  const int chunks = (dim / 8 + 31) / 32;
  auto kern = chunks <= 1   ? embed::lc1_pool_kernel<1>
              : chunks <= 2 ? embed::lc1_pool_kernel<2>
              : chunks <= 3 ? embed::lc1_pool_kernel<3>
              : chunks <= 4 ? embed::lc1_pool_kernel<4>
                            : embed::lc1_pool_kernel<8>;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
          cudaSuccess)
    return DORA_ERR_CUDA;
  kern<<<batch, embed::kLc1Warps * 32, smem, stream>>>(x, cu, t_cap, dim, norm_w, norm_b, eps, u,
                                                      status);
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  LinearEpi ep;
  ep.bias = b_head;
  return launch_linear(u, batch, nullptr, 2 * dim, w_head, classes, DORA_EPI_BIAS, ep, logits,
                       status, stream) == cudaSuccess
             ? DORA_OK
             : DORA_ERR_CUDA;
}

int dora_fold_layerscale(const dora_bf16* w, const dora_bf16* b, const dora_bf16* gamma,
                         int32_t n, int32_t k, dora_bf16* w_out, dora_bf16* b_out,
                         dora_stream_t stream_) {
  if (n <= 0 || k <= 0 || k % 8 != 0 || static_cast<long long>(n) * k > (1LL << 34))
    return DORA_ERR_INVALID_ARG;
  const void* al[] = {w, gamma, w_out};
  for (const void* p : al)
    if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0) return DORA_ERR_INVALID_ARG;
  if ((b == nullptr) != (b_out == nullptr)) return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  embed::layerscale_fold_kernel<<<embed::grid_for(static_cast<long long>(n) * (k / 8)), 256, 0,
                                  stream>>>(reinterpret_cast<const uint4*>(w), b, gamma, n, k / 8,
                                            reinterpret_cast<uint4*>(w_out), b_out);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

}  // extern "C"
