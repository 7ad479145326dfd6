// Token selection, stream compaction (optionally fused with LayerNorm', or
// carrying the row moments of a LayerNorm folded into the next linear), row
// LayerNorm, row moments and their merge from slice moments, the LayerNorm
// fold of a linear's weights and the synthetic score gather.  All are bandwidth- or
// latency-bound integer/copy work: no tensor cores.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {

// ---------------------------------------------------------------------------
// helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_sumf(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide sum; `scratch` holds >= 32 ints.  All threads get the result.
__device__ int block_sum(int v, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  int t = (threadIdx.x < nw) ? scratch[threadIdx.x] : 0;
  if (warp == 0) t = warp_sum(t);
  if (threadIdx.x == 0) scratch[0] = t;
  __syncthreads();
  const int r = scratch[0];
  __syncthreads();
  return r;
}

// Block-wide exclusive prefix sum of one int per thread (thread order).
__device__ int block_exclusive_scan(int v, int* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = (blockDim.x + 31) >> 5;
  int inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += t;
  }
  __syncthreads();
  if (lane == 31) scratch[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    int w = (lane < nw) ? scratch[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += t;
    }
    if (lane < nw) scratch[lane] = w;   // inclusive over warps
  }
  __syncthreads();
  const int warp_base = (warp == 0) ? 0 : scratch[warp - 1];
  const int r = warp_base + inc - v;
  __syncthreads();
  return r;
}

// Monotone map of fp32 scores to uint32: unsigned order of keys equals the
// order of the values, -0 == +0, every NaN above +inf.
__device__ __forceinline__ uint32_t score_key(float s) {
  uint32_t b = __float_as_uint(s);
  if (b == 0x80000000u) b = 0u;
  uint32_t k = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  if (s != s) k = 0xFFFFFFFFu;
  return k;
}

// Tokens image i keeps after clamping; every CTA evaluates it identically.
__device__ __forceinline__ int clamped_keep(int n, int m, int max_seqlen) {
  if (n > max_seqlen || n <= 0) return 0;
  return m < 1 ? 1 : (m > n ? n : m);
}

// ---------------------------------------------------------------------------
// K1: per-image deterministic top-k deletion
// ---------------------------------------------------------------------------
// One CTA per image.  Each visual candidate j counts how many candidates
// precede it in the order (score key, index); it is kept when that rank is
// below m - 1.  Kept flags are then scanned to write ascending indices.
__global__ void __launch_bounds__(kSelectThreads) select_keep_kernel(
    const float* __restrict__ scores, const int32_t* __restrict__ cu_in,
    const int32_t* __restrict__ keep_counts, int32_t batch, int32_t max_seqlen,
    int32_t* __restrict__ kept_idx, int32_t* __restrict__ cu_out, int32_t* status) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint32_t keys[];            // [max_seqlen]
  __shared__ int scratch[33];
  const int i = blockIdx.x;
  const int tid = threadIdx.x;

  // output offset of this image: sum of the clamped keep counts before it
  int part = 0;
  for (int t = tid; t < i; t += blockDim.x)
    part += clamped_keep(cu_in[t + 1] - cu_in[t], keep_counts[t], max_seqlen);
  const int off = block_sum(part, scratch);

  const int lo = cu_in[i];
  const int n = cu_in[i + 1] - lo;
  const int m = keep_counts[i];
  const int me = clamped_keep(n, m, max_seqlen);
  if (tid == 0) {
    if (n > max_seqlen) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    else if (n < 0 || (n > 0 && me != m) || (n == 0 && m != 0))
      record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
    cu_out[i + 1] = off + me;
    if (i == 0) cu_out[0] = 0;
  }
  if (me == 0) return;

  for (int j = tid; j < n; j += blockDim.x) keys[j] = score_key(scores[lo + j]);
  __syncthreads();

  // Each thread owns a contiguous segment of candidate indices so that the
  // flag scan below preserves index order.
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int j0 = tid * per;
  const int j1 = min(n, j0 + per);
  uint32_t keepmask = 0;     // bit q set when index j0 + q is kept (per <= 32)
  int cnt = 0;
  const int need = me - 1;   // visual tokens to keep
  for (int j = j0; j < j1; ++j) {
    bool kept;
    if (j == 0) {
      kept = true;           // CLS
    } else {
      const uint32_t kj = keys[j];
      int rank = 0;
      for (int t = 1; t < n; ++t) {
        const uint32_t kt = keys[t];
        rank += (kt < kj) | ((kt == kj) & (t < j));
      }
      kept = rank < need;
    }
    if (kept) {
      keepmask |= 1u << (j - j0);
      ++cnt;
    }
  }
  const int pos = block_exclusive_scan(cnt, scratch);
  int w = off + pos;
  for (int j = j0; j < j1; ++j)
    if (keepmask & (1u << (j - j0))) kept_idx[w++] = lo + j;
}

// ---------------------------------------------------------------------------
// K2: compaction (+ LayerNorm' or + row moments), one warp per output row
// ---------------------------------------------------------------------------
template <bool kLN, bool kStats>
__global__ void __launch_bounds__(kRowThreads) compact_kernel(
    const uint4* __restrict__ x, int32_t chunks /* dim / 8 */, const int32_t* __restrict__ kept_idx,
    const int32_t* __restrict__ cu_out, int32_t batch, int32_t t_in_cap,
    const int32_t* __restrict__ ids_in, const uint4* __restrict__ ln_w,
    const uint4* __restrict__ ln_b, float eps, uint4* __restrict__ packed,
    int32_t* __restrict__ ids_out, uint4* __restrict__ ln_out, const float2* __restrict__ mv_in,
    float2* __restrict__ mv_out, int32_t* status) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  int t_out = cu_out[batch];
  if (t_out > t_in_cap || t_out < 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    t_out = t_out < 0 ? 0 : t_in_cap;
  }
  const float inv_dim = 1.0f / static_cast<float>(chunks * 8);
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < t_out; r += warps) {
    const int src = kept_idx[r];
    if (src < 0 || src >= t_in_cap) {
      if (lane == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
      continue;
    }
    if (lane == 0) {
      if (ids_out != nullptr) ids_out[r] = ids_in[src];
      if constexpr (kStats) mv_out[r] = mv_in[src];
    }
    const uint4* srow = x + static_cast<size_t>(src) * chunks;
    uint4* drow = packed + static_cast<size_t>(r) * chunks;
    uint4 v[kMaxChunksPerLane];
#pragma unroll
    for (int q = 0; q < kMaxChunksPerLane; ++q) {
      const int c = lane + 32 * q;
      if (c < chunks) v[q] = __ldg(srow + c);
    }
#pragma unroll
    for (int q = 0; q < kMaxChunksPerLane; ++q) {
      const int c = lane + 32 * q;
      if (c < chunks) drow[c] = v[q];
    }
    if constexpr (kLN) {
      float sum = 0.f;
#pragma unroll
      for (int q = 0; q < kMaxChunksPerLane; ++q) {
        if (lane + 32 * q < chunks) {
          const uint32_t* w = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
          for (int e = 0; e < 4; ++e) sum += bf16_lo(w[e]) + bf16_hi(w[e]);
        }
      }
      const float mean = warp_sumf(sum) * inv_dim;
      float sq = 0.f;
#pragma unroll
      for (int q = 0; q < kMaxChunksPerLane; ++q) {
        if (lane + 32 * q < chunks) {
          const uint32_t* w = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float a = bf16_lo(w[e]) - mean, b = bf16_hi(w[e]) - mean;
            sq += a * a + b * b;
          }
        }
      }
      const float rstd = rsqrtf(warp_sumf(sq) * inv_dim + eps);
      uint4* lrow = ln_out + static_cast<size_t>(r) * chunks;
#pragma unroll
      for (int q = 0; q < kMaxChunksPerLane; ++q) {
        const int c = lane + 32 * q;
        if (c < chunks) {
          const uint4 gw = __ldg(ln_w + c), gb = __ldg(ln_b + c);
          const uint32_t* w = reinterpret_cast<const uint32_t*>(&v[q]);
          const uint32_t* g = reinterpret_cast<const uint32_t*>(&gw);
          const uint32_t* bb = reinterpret_cast<const uint32_t*>(&gb);
          uint4 o;
          uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float a = (bf16_lo(w[e]) - mean) * rstd * bf16_lo(g[e]) + bf16_lo(bb[e]);
            const float b = (bf16_hi(w[e]) - mean) * rstd * bf16_hi(g[e]) + bf16_hi(bb[e]);
            ow[e] = pack_bf16x2(a, b);
          }
          lrow[c] = o;
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------
// K5: LayerNorm, one warp per row
// ---------------------------------------------------------------------------
// Row statistics and normalisation of CPL 16-byte chunks per lane (the row
// length is chunks * 8 <= 256 * CPL); two rows per warp at a time, so that
// twice the bytes are in flight.
template <int CPL>
__device__ __forceinline__ void ln_row_stats(const uint4 (&v)[CPL], int lane, int chunks,
                                             float inv_dim, float eps, float& mean, float& rstd) {
  float sum = 0.f;
#pragma unroll
  for (int q = 0; q < CPL; ++q) {
    if (lane + 32 * q < chunks) {
      const uint32_t* u = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
      for (int e = 0; e < 4; ++e) sum += bf16_lo(u[e]) + bf16_hi(u[e]);
    }
  }
  mean = warp_sumf(sum) * inv_dim;
  float sq = 0.f;
#pragma unroll
  for (int q = 0; q < CPL; ++q) {
    if (lane + 32 * q < chunks) {
      const uint32_t* u = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = bf16_lo(u[e]) - mean, c2 = bf16_hi(u[e]) - mean;
        sq += a * a + c2 * c2;
      }
    }
  }
  rstd = rsqrtf(warp_sumf(sq) * inv_dim + eps);
}

template <int CPL>
__device__ __forceinline__ void ln_row_store(const uint4 (&v)[CPL], int lane, int chunks,
                                             float mean, float rstd, const uint4* __restrict__ w,
                                             const uint4* __restrict__ b, uint4* __restrict__ drow) {
#pragma unroll
  for (int q = 0; q < CPL; ++q) {
    const int c = lane + 32 * q;
    if (c < chunks) {
      const uint4 gw = __ldg(w + c), gb = __ldg(b + c);
      const uint32_t* u = reinterpret_cast<const uint32_t*>(&v[q]);
      const uint32_t* g = reinterpret_cast<const uint32_t*>(&gw);
      const uint32_t* bb = reinterpret_cast<const uint32_t*>(&gb);
      uint4 o;
      uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = (bf16_lo(u[e]) - mean) * rstd * bf16_lo(g[e]) + bf16_lo(bb[e]);
        const float c2 = (bf16_hi(u[e]) - mean) * rstd * bf16_hi(g[e]) + bf16_hi(bb[e]);
        ow[e] = pack_bf16x2(a, c2);
      }
      drow[c] = o;
    }
  }
}

template <int CPL>
__global__ void __launch_bounds__(kRowThreads) layernorm_kernel(
    const uint4* __restrict__ x, int32_t rows_cap, const int32_t* __restrict__ rows_dev,
    int32_t chunks, const uint4* __restrict__ w, const uint4* __restrict__ b, float eps,
    uint4* __restrict__ y) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  int rows = rows_cap;
  if (rows_dev != nullptr) rows = min(rows_cap, max(0, *rows_dev));
  const float inv_dim = 1.0f / static_cast<float>(chunks * 8);
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += 2 * warps) {
    const int r2 = r + warps;                         // second row of this warp, if any
    const bool two = r2 < rows;                       // warp-uniform
    uint4 v[CPL], v2[CPL];
#pragma unroll
    for (int q = 0; q < CPL; ++q) {
      const int c = lane + 32 * q;
      if (c < chunks) {
        v[q] = __ldg(x + static_cast<size_t>(r) * chunks + c);
        if (two) v2[q] = __ldg(x + static_cast<size_t>(r2) * chunks + c);
      }
    }
    float mean, rstd;
    ln_row_stats<CPL>(v, lane, chunks, inv_dim, eps, mean, rstd);
    ln_row_store<CPL>(v, lane, chunks, mean, rstd, w, b, y + static_cast<size_t>(r) * chunks);
    if (two) {
      ln_row_stats<CPL>(v2, lane, chunks, inv_dim, eps, mean, rstd);
      ln_row_store<CPL>(v2, lane, chunks, mean, rstd, w, b, y + static_cast<size_t>(r2) * chunks);
    }
  }
}

// ---------------------------------------------------------------------------
// K6: row moments (mean, biased variance) for a folded LayerNorm, one warp
// per row (two rows at a time), and their merge from slice moments
// ---------------------------------------------------------------------------
template <int CPL>
__device__ __forceinline__ float2 row_moments(const uint4 (&v)[CPL], int lane, int chunks,
                                              float inv_dim) {
  float sum = 0.f;
#pragma unroll
  for (int q = 0; q < CPL; ++q) {
    if (lane + 32 * q < chunks) {
      const uint32_t* u = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
      for (int e = 0; e < 4; ++e) sum += bf16_lo(u[e]) + bf16_hi(u[e]);
    }
  }
  const float mean = warp_sumf(sum) * inv_dim;
  float sq = 0.f;
#pragma unroll
  for (int q = 0; q < CPL; ++q) {
    if (lane + 32 * q < chunks) {
      const uint32_t* u = reinterpret_cast<const uint32_t*>(&v[q]);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float a = bf16_lo(u[e]) - mean, c2 = bf16_hi(u[e]) - mean;
        sq += a * a + c2 * c2;
      }
    }
  }
  return make_float2(mean, warp_sumf(sq) * inv_dim);
}

template <int CPL>
__global__ void __launch_bounds__(kRowThreads) row_stats_kernel(
    const uint4* __restrict__ x, int32_t rows_cap, const int32_t* __restrict__ rows_dev,
    int32_t chunks, float2* __restrict__ mv) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  int rows = rows_cap;
  if (rows_dev != nullptr) rows = min(rows_cap, max(0, *rows_dev));
  const float inv_dim = 1.0f / static_cast<float>(chunks * 8);
  for (int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < rows; r += 2 * warps) {
    const int r2 = r + warps;                         // second row of this warp, if any
    const bool two = r2 < rows;                       // warp-uniform
    uint4 v[CPL], v2[CPL];
#pragma unroll
    for (int q = 0; q < CPL; ++q) {
      const int c = lane + 32 * q;
      if (c < chunks) {
        v[q] = __ldg(x + static_cast<size_t>(r) * chunks + c);
        if (two) v2[q] = __ldg(x + static_cast<size_t>(r2) * chunks + c);
      }
    }
    const float2 a = row_moments<CPL>(v, lane, chunks, inv_dim);
    if (lane == 0) mv[r] = a;
    if (two) {
      const float2 b = row_moments<CPL>(v2, lane, chunks, inv_dim);
      if (lane == 0) mv[r2] = b;
    }
  }
}

// One thread per row: mean = (1/S) sum mean_s, M2 = sum (M2_s + 64 (mean_s -
// mean)^2) over the row's S slices of 64 (the pairwise update of Chan, Golub
// & LeVeque with equal counts), var = M2 / (64 S).
__global__ void __launch_bounds__(256) merge_moments_kernel(const float2* __restrict__ sm,
                                                            int32_t rows_cap,
                                                            const int32_t* __restrict__ rows_dev,
                                                            int32_t slices,
                                                            float2* __restrict__ mv) {
  pdl_trigger();
  pdl_wait();
  int rows = rows_cap;
  if (rows_dev != nullptr) rows = min(rows_cap, max(0, *rows_dev));
  const size_t stride = static_cast<size_t>(rows_cap);
  const float inv_s = 1.0f / static_cast<float>(slices);
  constexpr int kHeld = 16;     // slices held in registers (dim <= 1024): one round of loads
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += gridDim.x * blockDim.x) {
    const float2* p = sm + r;
    float mean, m2 = 0.f;
    if (slices <= kHeld) {
      float2 t[kHeld];
#pragma unroll
      for (int j = 0; j < kHeld; ++j)
        if (j < slices) t[j] = __ldg(p + j * stride);
      float sum = 0.f;
#pragma unroll
      for (int j = 0; j < kHeld; ++j)
        if (j < slices) sum += t[j].x;
      mean = sum * inv_s;
#pragma unroll
      for (int j = 0; j < kHeld; ++j)
        if (j < slices) {
          const float d = t[j].x - mean;
          m2 += t[j].y + static_cast<float>(kSliceCols) * d * d;
        }
    } else {
      float sum = 0.f;
      for (int j = 0; j < slices; ++j) sum += __ldg(p + j * stride).x;
      mean = sum * inv_s;
      for (int j = 0; j < slices; ++j) {
        const float2 t = __ldg(p + j * stride);
        const float d = t.x - mean;
        m2 += t.y + static_cast<float>(kSliceCols) * d * d;
      }
    }
    mv[r] = make_float2(mean, m2 * inv_s * (1.0f / kSliceCols));
  }
}

// ---------------------------------------------------------------------------
// K7: LayerNorm affine folded into the next linear, one warp per weight row
// ---------------------------------------------------------------------------
// w_out[n, :] = bf16(w[n, :] * gamma) (the product of two bf16 values is
// exact in fp32, so this is one rounding), colsum[n] = sum of the rounded
// w_out[n, :] (the values the GEMM multiplies), colbias[n] = w[n, :] . beta
// + bias[n], both accumulated in fp32.
__global__ void __launch_bounds__(kRowThreads) fold_ln_kernel(
    const uint4* __restrict__ w, int32_t n, int32_t chunks, const uint4* __restrict__ gamma,
    const uint4* __restrict__ beta, const uint16_t* __restrict__ bias, uint4* __restrict__ w_out,
    float* __restrict__ colsum, float* __restrict__ colbias) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  for (int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < n; row += warps) {
    float cs = 0.f, cb = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      const uint4 wv = __ldg(w + static_cast<size_t>(row) * chunks + c);
      const uint4 gv = __ldg(gamma + c), bv = __ldg(beta + c);
      const uint32_t* wu = reinterpret_cast<const uint32_t*>(&wv);
      const uint32_t* gu = reinterpret_cast<const uint32_t*>(&gv);
      const uint32_t* bu = reinterpret_cast<const uint32_t*>(&bv);
      uint4 o;
      uint32_t* ou = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        ou[e] = pack_bf16x2(bf16_lo(wu[e]) * bf16_lo(gu[e]), bf16_hi(wu[e]) * bf16_hi(gu[e]));
        cs += bf16_lo(ou[e]) + bf16_hi(ou[e]);
        cb += bf16_lo(wu[e]) * bf16_lo(bu[e]) + bf16_hi(wu[e]) * bf16_hi(bu[e]);
      }
      w_out[static_cast<size_t>(row) * chunks + c] = o;
    }
    cs = warp_sumf(cs);
    cb = warp_sumf(cb);
    if (lane == 0) {
      colsum[row] = cs;
      colbias[row] = cb + (bias != nullptr ? __uint_as_float(static_cast<uint32_t>(bias[row]) << 16)
                                           : 0.f);
    }
  }
}

// ---------------------------------------------------------------------------
// synthetic actor stand-in: row-aligned scores from per-image id tables
// ---------------------------------------------------------------------------
__global__ void gather_scores_kernel(const float* __restrict__ table, int32_t stride,
                                     const int32_t* __restrict__ ids,
                                     const int32_t* __restrict__ cu, float* __restrict__ scores,
                                     int32_t* status) {
  pdl_trigger();
  pdl_wait();
  const int i = blockIdx.x;
  const int lo = cu[i], hi = cu[i + 1];
  const float* row = table + static_cast<size_t>(i) * stride;
  for (int r = lo + threadIdx.x; r < hi; r += blockDim.x) {
    const int id = ids[r];
    float s;
    if (id >= 0 && id < stride) {
      s = row[id];
    } else {
      s = __int_as_float(0x7FC00000);
      record_status(status, DORA_ERR_DEVICE_SEQLEN);
    }
    scores[r] = s;
  }
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
static int row_grid(int64_t rows) {
  const int64_t warps_per_cta = kRowThreads / 32;
  int64_t g = (rows + warps_per_cta - 1) / warps_per_cta;
  const int64_t cap = 152LL * 16;       // grid-stride beyond ~16 CTAs per SM
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  return static_cast<int>(g);
}

cudaError_t launch_select_keep(const float* scores, const int32_t* cu_in,
                               const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                               int32_t* kept_idx, int32_t* cu_out, int32_t* status,
                               cudaStream_t stream) {
  if (batch == 0) return cudaSuccess;
  const size_t smem = static_cast<size_t>(max_seqlen) * sizeof(uint32_t);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(select_keep_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  return launch_pdl(select_keep_kernel, dim3(batch), dim3(kSelectThreads), smem, stream, scores,
                    cu_in, keep_counts, batch, max_seqlen, kept_idx, cu_out, status);
}

cudaError_t launch_compact(const uint16_t* x, int32_t dim, const int32_t* kept_idx,
                           const int32_t* cu_out, int32_t batch, int32_t t_in_cap,
                           const int32_t* ids_in, const uint16_t* ln_w, const uint16_t* ln_b,
                           float eps, uint16_t* packed, int32_t* ids_out, uint16_t* ln_out,
                           const float* mv_in, float* mv_out, int32_t* status,
                           cudaStream_t stream) {
  const int grid = row_grid(t_in_cap);
  const int chunks = dim / 8;
  const uint4* xx = reinterpret_cast<const uint4*>(x);
  const uint4* ww = reinterpret_cast<const uint4*>(ln_w);
  const uint4* bb = reinterpret_cast<const uint4*>(ln_b);
  uint4* pp = reinterpret_cast<uint4*>(packed);
  uint4* ll = reinterpret_cast<uint4*>(ln_out);
  const float2* mi = reinterpret_cast<const float2*>(mv_in);
  float2* mo = reinterpret_cast<float2*>(mv_out);
  if (ln_out != nullptr)
    return launch_pdl(compact_kernel<true, false>, dim3(grid), dim3(kRowThreads), 0, stream,
                      xx, chunks, kept_idx, cu_out, batch, t_in_cap, ids_in, ww, bb, eps, pp, ids_out, ll,
        nullptr, nullptr, status);
  if (mv_out != nullptr)
    return launch_pdl(compact_kernel<false, true>, dim3(grid), dim3(kRowThreads), 0, stream,
        xx, chunks, kept_idx, cu_out, batch, t_in_cap, ids_in, nullptr, nullptr, 0.f, pp, ids_out,
        nullptr, mi, mo, status);
  return launch_pdl(compact_kernel<false, false>, dim3(grid), dim3(kRowThreads), 0, stream,
        xx, chunks, kept_idx, cu_out, batch, t_in_cap, ids_in, nullptr, nullptr, 0.f, pp, ids_out,
        nullptr, nullptr, nullptr, status);
}

cudaError_t launch_layernorm(const uint16_t* x, int32_t rows_cap, const int32_t* rows_dev,
                             int32_t dim, const uint16_t* w, const uint16_t* b, float eps,
                             uint16_t* y, cudaStream_t stream) {
  if (rows_cap == 0) return cudaSuccess;
  const int chunks = dim / 8;
  const int grid = row_grid((rows_cap + 1) / 2);
  const uint4* xx = reinterpret_cast<const uint4*>(x);
  const uint4* ww = reinterpret_cast<const uint4*>(w);
  const uint4* bb = reinterpret_cast<const uint4*>(b);
  uint4* yy = reinterpret_cast<uint4*>(y);
  // registers sized to the row: 16-byte chunks per lane
  cudaError_t e;
  switch ((chunks + 31) / 32) {
    case 1: e = launch_pdl(layernorm_kernel<1>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ww, bb, eps, yy); break;
    case 2: e = launch_pdl(layernorm_kernel<2>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ww, bb, eps, yy); break;
    case 3: e = launch_pdl(layernorm_kernel<3>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ww, bb, eps, yy); break;
    case 4: e = launch_pdl(layernorm_kernel<4>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ww, bb, eps, yy); break;
    default: e = launch_pdl(layernorm_kernel<kMaxChunksPerLane>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ww, bb, eps, yy); break;
  }
  return e;
}

cudaError_t launch_row_stats(const uint16_t* x, int32_t rows_cap, const int32_t* rows_dev,
                             int32_t dim, float* mv, cudaStream_t stream) {
  if (rows_cap == 0) return cudaSuccess;
  const int chunks = dim / 8;
  const int grid = row_grid((rows_cap + 1) / 2);
  const uint4* xx = reinterpret_cast<const uint4*>(x);
  float2* ss = reinterpret_cast<float2*>(mv);
  cudaError_t e;
  switch ((chunks + 31) / 32) {
    case 1: e = launch_pdl(row_stats_kernel<1>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ss); break;
    case 2: e = launch_pdl(row_stats_kernel<2>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ss); break;
    case 3: e = launch_pdl(row_stats_kernel<3>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ss); break;
    case 4: e = launch_pdl(row_stats_kernel<4>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ss); break;
    default: e = launch_pdl(row_stats_kernel<kMaxChunksPerLane>, dim3(grid), dim3(kRowThreads), 0, stream, xx, rows_cap, rows_dev, chunks, ss); break;
  }
  return e;
}

cudaError_t launch_merge_moments(const float* sm, int32_t rows_cap, const int32_t* rows_dev,
                                 int32_t slices, float* mv, cudaStream_t stream) {
  if (rows_cap == 0) return cudaSuccess;
  int64_t g = (static_cast<int64_t>(rows_cap) + 255) / 256;
  if (g > 152LL * 8) g = 152LL * 8;
  return launch_pdl(merge_moments_kernel, dim3(static_cast<unsigned>(g)), dim3(256), 0, stream,
                    reinterpret_cast<const float2*>(sm), rows_cap, rows_dev, slices,
                    reinterpret_cast<float2*>(mv));
}

cudaError_t launch_fold_ln(const uint16_t* w, int32_t n, int32_t k, const uint16_t* gamma,
                           const uint16_t* beta, const uint16_t* bias, uint16_t* w_out,
                           float* colsum, float* colbias, cudaStream_t stream) {
  if (n == 0) return cudaSuccess;
  return launch_pdl(fold_ln_kernel, dim3(row_grid(n)), dim3(kRowThreads), 0, stream,
                    reinterpret_cast<const uint4*>(w), n, k / 8,
                    reinterpret_cast<const uint4*>(gamma), reinterpret_cast<const uint4*>(beta),
                    bias, reinterpret_cast<uint4*>(w_out), colsum, colbias);
}

cudaError_t launch_gather_scores(const float* table, int32_t stride, const int32_t* ids,
                                 const int32_t* cu, int32_t batch, float* scores, int32_t* status,
                                 cudaStream_t stream) {
  if (batch == 0) return cudaSuccess;
  return launch_pdl(gather_scores_kernel, dim3(batch), dim3(256), 0, stream, table, stride, ids, cu,
                    scores, status);
}

}  // namespace dora
