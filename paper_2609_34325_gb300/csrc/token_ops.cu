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
// An image whose rows do not lie inside [0, t_cap) keeps nothing.
__device__ __forceinline__ int clamped_keep(int lo, int n, int m, int max_seqlen, int t_cap) {
  if (n > max_seqlen || n <= 0 || lo < 0 || lo > t_cap - n) return 0;
  return m < 1 ? 1 : (m > n ? n : m);
}

// ---------------------------------------------------------------------------
// K1: per-image deterministic top-k deletion, optionally fused with the
// compaction of the kept rows
// ---------------------------------------------------------------------------
// Work of one CTA (kSelectThreads threads) for image i = blockIdx.x / splits:
//  1. its output offset, the sum of the clamped keep counts of images < i,
//  2. and, with those loads in flight, the image's candidate keys (ordered
//     uint32 of the deletion scores) in shared memory;
//  3. radix select, 8 bits a pass from the top: the key T of the
//     (m-1)-th smallest candidate and how many candidates equal to T are
//     kept (the lowest-indexed ones: ties are broken by index); once a
//     single candidate has T's prefix, its key is T and the passes stop;
//  4. one block-wide scan over contiguous index segments of the packed
//     counts (candidates below T, candidates equal to T), which gives every
//     kept token its output position in index order;
//  5. the kept list in shared memory (and, by the image's first CTA, in
//     kept_idx and cu_out).
// With CPL > 0, the `splits` CTAs of the image then copy its kept rows
// (16-byte vector loads and stores, one warp per row, two rows in flight a
// warp), their ids and their row moments: every CTA selects (the scores are
// read from L2 after the first), and the row copies are spread over all of
// them.  Selection and compaction are one launch, and no kept_idx round trip
// through global memory stands between them.  CPL is the number of 16-byte
// chunks of a row per lane (registers sized to the row); 0 = selection only.
constexpr int kRadixBins = 256;
static_assert(kSelectThreads == kRadixBins, "one histogram bin per thread");

// Row moments (mean, var) of one row from its S slice moments (mean_s, M2_s)
// over 64 columns each, stored slice-major with `stride` rows between slices:
// mean = (1/S) sum mean_s, M2 = sum (M2_s + 64 (mean_s - mean)^2) (the
// pairwise update of Chan, Golub & LeVeque with equal counts), var = M2 / (64 S).
// Every rounding is explicit, so each caller gets the same bits.
__device__ __forceinline__ float2 merge_slice_moments(const float2* __restrict__ p, size_t stride,
                                                      int slices) {
  constexpr int kHeld = 16;     // slice means held in registers (dim <= 1024)
  const float inv_s = __frcp_rn(static_cast<float>(slices));
  float mean, m2 = 0.f;
  if (slices <= kHeld) {
    float mu[kHeld];
#pragma unroll
    for (int j = 0; j < kHeld; ++j)
      if (j < slices) mu[j] = __ldg(&p[j * stride].x);
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j < kHeld; ++j)
      if (j < slices) sum = __fadd_rn(sum, mu[j]);
    mean = __fmul_rn(sum, inv_s);
#pragma unroll
    for (int j = 0; j < kHeld; ++j)
      if (j < slices) {             // the M2 halves are read again (L1)
        const float d = __fsub_rn(mu[j], mean);
        m2 = __fadd_rn(m2, __fmaf_rn(__fmul_rn(static_cast<float>(kSliceCols), d), d,
                                     __ldg(&p[j * stride].y)));
      }
  } else {
    float sum = 0.f;
    for (int j = 0; j < slices; ++j) sum = __fadd_rn(sum, __ldg(&p[j * stride].x));
    mean = __fmul_rn(sum, inv_s);
    for (int j = 0; j < slices; ++j) {
      const float2 t = __ldg(p + j * stride);
      const float d = __fsub_rn(t.x, mean);
      m2 = __fadd_rn(m2, __fmaf_rn(__fmul_rn(static_cast<float>(kSliceCols), d), d, t.y));
    }
  }
  return make_float2(mean, __fmul_rn(__fmul_rn(m2, inv_s), 1.0f / kSliceCols));
}

template <int CPL>
__global__ void __launch_bounds__(kSelectThreads) select_keep_kernel(
    const float* __restrict__ scores, const int32_t* __restrict__ cu_in,
    const int32_t* __restrict__ keep_counts, int32_t batch, int32_t max_seqlen, int32_t t_cap,
    int32_t splits, int32_t* __restrict__ kept_idx, int32_t* __restrict__ cu_out,
    const uint4* __restrict__ x, int32_t chunks, const int32_t* __restrict__ ids_in,
    const float2* __restrict__ mv_in, int32_t mv_slices, uint4* __restrict__ packed,
    int32_t* __restrict__ ids_out, float2* __restrict__ mv_out, int32_t* status) {
  pdl_trigger();
  pdl_wait();
  extern __shared__ uint32_t keys[];            // [max_seqlen] keys, then [max_seqlen] kept rows
  int32_t* kept_rows = reinterpret_cast<int32_t*>(keys + max_seqlen);
  __shared__ int scratch[33];
  __shared__ int hist[kRadixBins];
  __shared__ uint32_t sel_prefix;
  __shared__ int sel_rank;
  __shared__ int sel_count;
  __shared__ uint32_t sel_key;
  const int i = blockIdx.x / splits;
  const int part = blockIdx.x - i * splits;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  // rows of the input (and capacity of the outputs): t_cap, or cu_in[batch]
  // when the caller gives none
  const int cap = t_cap >= 0 ? t_cap : cu_in[batch];

  // 1-2. the image's own bounds and keep count (every thread reads the same
  // three words), its candidate keys into shared memory, and its output
  // offset, the sum of the clamped keep counts of the images before it: the
  // keys' loads and the offset's are in flight together, and the offset's
  // block reduction is also the barrier that publishes the keys
  const int lo = cu_in[i];
  const int n = cu_in[i + 1] - lo;
  const int m = keep_counts[i];
  const int me = clamped_keep(lo, n, m, max_seqlen, cap);
  if (me > 0)                                   // the rows lie inside the input
    for (int j = tid; j < n; j += blockDim.x) keys[j] = score_key(scores[lo + j]);
  int acc = 0;
  for (int t = tid; t < i; t += blockDim.x) {
    const int l0 = cu_in[t];
    acc += clamped_keep(l0, cu_in[t + 1] - l0, keep_counts[t], max_seqlen, cap);
  }
  const int off = block_sum(acc, scratch);   // its barriers also publish the keys
  if (part == 0 && tid == 0) {
    // rows outside the input, or (boundaries not increasing) outputs past it
    if (n > max_seqlen || (n > 0 && (lo < 0 || lo > cap - n)) || off > cap - me)
      record_status(status, DORA_ERR_DEVICE_SEQLEN);
    else if (n < 0 || (n > 0 && me != m) || (n == 0 && m != 0))
      record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
    cu_out[i + 1] = off + me;
    if (i == 0) cu_out[0] = 0;
  }
  if (me == 0) return;

  // 3. threshold key T and the number of candidates equal to T that are kept
  const int need = me - 1;                       // visual tokens kept
  uint32_t thr;
  int ties_keep;
  if (need == 0) {
    thr = 0u;                                    // no candidate is below key 0 ...
    ties_keep = 0;                               // ... and none equal to it is kept
  } else if (need == n - 1) {
    thr = 0xFFFFFFFFu;                           // every candidate is kept
    ties_keep = n;
  } else {
    uint32_t prefix = 0u, hi_mask = 0u;
    int rank = need;                             // 1-based rank among the remaining
#pragma unroll 1
    for (int shift = 24; shift >= 0; shift -= 8) {
      hist[tid] = 0;
      __syncthreads();
      // warp-uniform trip count: every lane reaches the match below
      for (int base = 0; base < n; base += blockDim.x) {
        const int j = base + tid;
        const uint32_t k = (j >= 1 && j < n) ? keys[j] : 0u;
        const bool in = j >= 1 && j < n && ((k ^ prefix) & hi_mask) == 0u;
        const uint32_t digit = in ? ((k >> shift) & 0xFFu) : 0x100u;
        const uint32_t peers = __match_any_sync(0xffffffffu, digit);
        if (in && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], __popc(peers));
      }
      __syncthreads();
      const int c = hist[tid];
      const int below = block_exclusive_scan(c, scratch);
      if (below < rank && rank <= below + c) {
        sel_prefix = prefix | (static_cast<uint32_t>(tid) << shift);
        sel_rank = rank - below;
        sel_count = c;
      }
      __syncthreads();
      prefix = sel_prefix;
      rank = sel_rank;
      hi_mask |= 0xFFu << shift;
      if (shift > 0 && sel_count == 1) {
        // one candidate has this prefix: its key is the threshold (no other
        // key equals it, so rank is 1) and the lower bytes need no pass
        for (int j = tid; j < n; j += blockDim.x)
          if (j >= 1 && ((keys[j] ^ prefix) & hi_mask) == 0u) sel_key = keys[j];
        __syncthreads();
        prefix = sel_key;
        break;
      }
    }
    thr = prefix;
    ties_keep = rank;
  }

  // 4. output positions: each thread owns a contiguous segment of indices;
  // CLS (index 0) counts as a token below the threshold
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int j0 = tid * per;
  const int j1 = min(n, j0 + per);
  int below = 0, equal = 0;
  for (int j = j0; j < j1; ++j) {
    if (j == 0) {
      ++below;
    } else {
      const uint32_t k = keys[j];
      below += k < thr;
      equal += k == thr;
    }
  }
  const int pre = block_exclusive_scan((equal << 16) | below, scratch);   // both < 2^16
  int ties_before = pre >> 16;
  int pos = (pre & 0xFFFF) + min(ties_before, ties_keep);
  // 5. the kept list
  for (int j = j0; j < j1; ++j) {
    bool kept = j == 0;
    if (!kept) {
      const uint32_t k = keys[j];
      if (k == thr) kept = ties_before++ < ties_keep;
      else kept = k < thr;
    }
    if (kept) {
      if (part == 0 && off + pos < cap) kept_idx[off + pos] = lo + j;
      if constexpr (CPL > 0) kept_rows[pos] = lo + j;
      ++pos;
    }
  }
  if constexpr (CPL > 0) {
    __syncthreads();
    // rows r = part * 8 + warp, + splits * 8, ... of this image: two per pass
    const int warps = blockDim.x >> 5;
    const int stride = splits * warps;
    const int rows = min(me, cap - off);        // outputs past the capacity are dropped
    int r = part * warps + (tid >> 5);
    for (; r < rows; r += 2 * stride) {
      const int r2 = r + stride;
      const bool two = r2 < rows;
      const int s1 = kept_rows[r];
      const int s2 = two ? kept_rows[r2] : s1;
      const uint4* src1 = x + static_cast<size_t>(s1) * chunks;
      const uint4* src2 = x + static_cast<size_t>(s2) * chunks;
      uint4 v1[CPL], v2[CPL];
#pragma unroll
      for (int q = 0; q < CPL; ++q) {
        const int c = lane + 32 * q;
        if (c < chunks) {
          v1[q] = __ldg(src1 + c);
          if (two) v2[q] = __ldg(src2 + c);
        }
      }
      uint4* dst1 = packed + static_cast<size_t>(off + r) * chunks;
      uint4* dst2 = packed + static_cast<size_t>(off + r2) * chunks;
#pragma unroll
      for (int q = 0; q < CPL; ++q) {
        const int c = lane + 32 * q;
        if (c < chunks) {
          dst1[c] = v1[q];
          if (two) dst2[c] = v2[q];
        }
      }
      if (lane == 0) {
        if (ids_out != nullptr) ids_out[off + r] = ids_in[s1];
        if (mv_out != nullptr && mv_slices == 0) mv_out[off + r] = mv_in[s1];
      } else if (lane == 1 && two) {
        if (ids_out != nullptr) ids_out[off + r2] = ids_in[s2];
        if (mv_out != nullptr && mv_slices == 0) mv_out[off + r2] = mv_in[s2];
      }
    }
    // row moments merged from the slice moments the producing linear wrote
    // (mv_slices > 0): one thread per kept row, apart from the row copies so
    // that the merge's registers do not weigh on them
    if (mv_out != nullptr && mv_slices > 0)
      for (int q = part * blockDim.x + tid; q < rows; q += splits * blockDim.x)
        mv_out[off + q] = merge_slice_moments(mv_in + kept_rows[q], cap, mv_slices);
  }
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

// One thread per row: the row's slice moments merged (merge_slice_moments).
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
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += gridDim.x * blockDim.x)
    mv[r] = merge_slice_moments(sm + r, stride, slices);
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

// Shared memory of the selection: keys and the kept list, [max_seqlen] each.
static cudaError_t select_smem(const void* kern, int32_t max_seqlen, size_t* smem) {
  *smem = static_cast<size_t>(max_seqlen) * 2 * sizeof(uint32_t);
  if (*smem > 48 * 1024)
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(*smem));
  return cudaSuccess;
}

cudaError_t launch_select_keep(const float* scores, const int32_t* cu_in,
                               const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                               int32_t* kept_idx, int32_t* cu_out, int32_t* status,
                               cudaStream_t stream) {
  if (batch == 0) return cudaSuccess;
  size_t smem = 0;
  cudaError_t e = select_smem(reinterpret_cast<const void*>(select_keep_kernel<0>),
                              max_seqlen, &smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(select_keep_kernel<0>, dim3(batch), dim3(kSelectThreads), smem, stream,
                    scores, cu_in, keep_counts, batch, max_seqlen, -1, 1, kept_idx,
                    cu_out, static_cast<const uint4*>(nullptr), 0,
                    static_cast<const int32_t*>(nullptr), static_cast<const float2*>(nullptr), 0,
                    static_cast<uint4*>(nullptr), static_cast<int32_t*>(nullptr),
                    static_cast<float2*>(nullptr), status);
}

// CTAs per image of the fused kernel: about kSelectCtas CTAs in all (a
// measured sweep at 256 x 197, 64 x 577 and 1024 x 197 tokens put the best
// split near 512 CTAs), at most kSelectMaxSplits, and no more than one per
// 16 tokens of the longest image.
int select_compact_splits(int32_t batch, int32_t max_seqlen) {
  if (batch <= 0) return 1;
  int s = (kSelectCtas + batch - 1) / batch;
  const int by_rows = (max_seqlen + 15) / 16;
  if (s > by_rows) s = by_rows;
  return s < 1 ? 1 : (s > kSelectMaxSplits ? kSelectMaxSplits : s);
}

template <int CPL>
static cudaError_t select_compact_cpl(const float* scores, const int32_t* cu_in,
                                      const int32_t* keep_counts, int32_t batch,
                                      int32_t max_seqlen, const uint16_t* x, int32_t chunks,
                                      int32_t t_in_cap, const int32_t* ids_in,
                                      const float* mv_in, int32_t mv_slices, int32_t* kept_idx,
                                      int32_t* cu_out, uint16_t* packed, int32_t* ids_out,
                                      float* mv_out, int32_t* status, cudaStream_t stream) {
  size_t smem = 0;
  cudaError_t e = select_smem(reinterpret_cast<const void*>(select_keep_kernel<CPL>),
                              max_seqlen, &smem);
  if (e != cudaSuccess) return e;
  const int splits = select_compact_splits(batch, max_seqlen);
  const long long grid = static_cast<long long>(batch) * splits;
  if (grid > 0x7fffffffLL) return cudaErrorInvalidValue;
  return launch_pdl(select_keep_kernel<CPL>, dim3(static_cast<unsigned>(grid)),
                    dim3(kSelectThreads), smem, stream, scores, cu_in, keep_counts, batch,
                    max_seqlen, t_in_cap, splits, kept_idx, cu_out,
                    reinterpret_cast<const uint4*>(x), chunks, ids_in,
                    reinterpret_cast<const float2*>(mv_in), mv_slices,
                    reinterpret_cast<uint4*>(packed), ids_out, reinterpret_cast<float2*>(mv_out),
                    status);
}

cudaError_t launch_select_compact(const float* scores, const int32_t* cu_in,
                                  const int32_t* keep_counts, int32_t batch, int32_t max_seqlen,
                                  const uint16_t* x, int32_t dim, int32_t t_in_cap,
                                  const int32_t* ids_in, const float* mv_in, int32_t* kept_idx,
                                  int32_t* cu_out, uint16_t* packed, int32_t* ids_out,
                                  float* mv_out, int32_t* status, cudaStream_t stream,
                                  int32_t mv_slices) {
  if (batch == 0) return cudaSuccess;
  const int chunks = dim / 8;
  switch ((chunks + 31) / 32) {
    case 1: return select_compact_cpl<1>(scores, cu_in, keep_counts, batch, max_seqlen, x, chunks,
                                         t_in_cap, ids_in, mv_in, mv_slices, kept_idx, cu_out, packed, ids_out,
                                         mv_out, status, stream);
    case 2: return select_compact_cpl<2>(scores, cu_in, keep_counts, batch, max_seqlen, x, chunks,
                                         t_in_cap, ids_in, mv_in, mv_slices, kept_idx, cu_out, packed, ids_out,
                                         mv_out, status, stream);
    case 3: return select_compact_cpl<3>(scores, cu_in, keep_counts, batch, max_seqlen, x, chunks,
                                         t_in_cap, ids_in, mv_in, mv_slices, kept_idx, cu_out, packed, ids_out,
                                         mv_out, status, stream);
    case 4: return select_compact_cpl<4>(scores, cu_in, keep_counts, batch, max_seqlen, x, chunks,
                                         t_in_cap, ids_in, mv_in, mv_slices, kept_idx, cu_out, packed, ids_out,
                                         mv_out, status, stream);
    default: return select_compact_cpl<kMaxChunksPerLane>(
        scores, cu_in, keep_counts, batch, max_seqlen, x, chunks, t_in_cap, ids_in, mv_in,
        mv_slices, kept_idx, cu_out, packed, ids_out, mv_out, status, stream);
  }
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
