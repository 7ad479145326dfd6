// Training-side pieces of DORA on the packed token layout:
//   Plackett-Luce ordered sampling   App. A.3: the removal sequence drawn
//                                    without replacement from the selector's
//                                    scores, as the Gumbel-top-k of s + g
//                                    (the noise g is an input);
//   Plackett-Luce log-probability    App. A.3: sum_t s_{i_t} - log sum_{R_t}
//                                    exp(s_j), and its gradient for PPO;
//   branching                        App. B.2: complete-prefix shadows leave
//                                    the rollout after each pruning block and
//                                    run the remaining blocks unpruned, as
//                                    extra sequences of the same packed batch;
//   fidelity cost                    App. B.2: tau^2 KL(softmax(z^N / tau) ||
//                                    softmax(z^(l) / tau)) per shadow.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "dora.h"
#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace train {

constexpr int kMaxVisual = 2048;    // visual tokens per image held in shared memory
constexpr int kThreads = 256;

// fp32 -> uint32 whose unsigned order is the value order: -0 == +0, NaN above +inf.
__device__ __forceinline__ uint32_t order_key(float v) {
  uint32_t b = __float_as_uint(v);
  if (b == 0x80000000u) b = 0;
  if (v != v) return 0xFFFFFFFFu;
  return (b >> 31) ? ~b : (b | 0x80000000u);
}

// ---------------------------------------------------------------------------
// Gumbel-top-k: one CTA per image.  Visual token j's rank is the number of
// tokens whose key s + g (fp32) is larger, or equal with a higher index (the
// deployment selection's tie rule, so the first k_i are what it deletes given
// the keys); ranks below k_i give order[i, rank] = j, entries k_i..k_cap-1
// are -1, and the keys go to keys_out (row-aligned, nullable).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads)
    pl_sample_kernel(const float* __restrict__ scores, const float* __restrict__ gumbel,
                     const int32_t* __restrict__ cu, int t_cap, const int32_t* __restrict__ kreq,
                     int k_cap, int32_t* __restrict__ order, float* __restrict__ keys_out,
                     int32_t* status) {
  __shared__ uint32_t keys[kMaxVisual];
  const int img = blockIdx.x;
  const int lo = cu[img], hi = cu[img + 1];
  int32_t* out = order + static_cast<size_t>(img) * k_cap;
  int n = hi - lo - 1;
  if (lo < 0 || hi > t_cap || n > kMaxVisual) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    n = 0;
  }
  if (n < 0) n = 0;
  int k = kreq[img];
  if (k < 0 || k > n || k > k_cap) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
    k = k < 0 ? 0 : (k > n ? n : k);
    k = k > k_cap ? k_cap : k;
  }
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    const float key = scores[lo + 1 + j] + gumbel[lo + 1 + j];
    keys[j] = order_key(key);
    if (keys_out != nullptr) keys_out[lo + 1 + j] = key;
  }
  if (keys_out != nullptr && threadIdx.x == 0 && hi > lo && lo >= 0 && lo < t_cap)
    keys_out[lo] = scores[lo];
  __syncthreads();
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    const uint32_t kj = keys[j];
    int rank = 0;
    for (int u = 0; u < n; ++u) {
      const uint32_t ku = keys[u];
      rank += (ku > kj) | ((ku == kj) & (u > j));
    }
    if (rank < k) out[rank] = j;
  }
  for (int t = k + threadIdx.x; t < k_cap; t += blockDim.x) out[t] = -1;
}

// ---------------------------------------------------------------------------
// log-sum-exp pairs: (m, s) stands for log(s) + m, s = sum exp(x - m).
// ---------------------------------------------------------------------------
struct Lse {
  float m, s;
};
__device__ __forceinline__ Lse lse_id() { return {-INFINITY, 0.f}; }
__device__ __forceinline__ Lse lse_of(float x) { return {x, 1.f}; }
__device__ __forceinline__ Lse lse_merge(Lse a, Lse b) {
  if (a.s == 0.f) return b;
  if (b.s == 0.f) return a;
  const float m = fmaxf(a.m, b.m);
  return {m, a.s * __expf(a.m - m) + b.s * __expf(b.m - m)};
}
__device__ __forceinline__ float lse_val(Lse a) { return a.m + __logf(a.s); }
__device__ __forceinline__ Lse shfl_lse_down(Lse a, int off) {
  return {__shfl_down_sync(0xffffffffu, a.m, off), __shfl_down_sync(0xffffffffu, a.s, off)};
}
__device__ __forceinline__ Lse shfl_lse_up(Lse a, int off) {
  return {__shfl_up_sync(0xffffffffu, a.m, off), __shfl_up_sync(0xffffffffu, a.s, off)};
}

// ---------------------------------------------------------------------------
// Log-probability and gradient: one CTA per image.
//   rest   = LSE of the scores never removed;
//   L_t    = LSE over R_t = rest (+) LSE(s_{i_t}, ..., s_{i_k}) (a suffix scan
//            over the sequence in one warp: no cancellation, every term is
//            added, never subtracted);
//   log pi = sum_t s_{i_t} - L_t;
//   P_u    = log sum_{t<=u} exp(-L_t) (a prefix scan);
//   d log pi / d s_j = 1[j = i_u] - exp(s_j + P_u) for removed j = i_u, and
//                      -exp(s_j + P_k) for the others (each exp <= u since
//                      s_j <= L_t whenever j is in R_t).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads)
    pl_logprob_kernel(const float* __restrict__ scores, const int32_t* __restrict__ cu, int t_cap,
                      const int32_t* __restrict__ kreq, const int32_t* __restrict__ order,
                      int k_cap, float* __restrict__ logp, float* __restrict__ grad,
                      const float* __restrict__ dlogp, int32_t* status) {
  __shared__ float s[kMaxVisual];
  __shared__ int32_t pos[kMaxVisual];     // 1 + the step that removes j, 0 if kept
  __shared__ float lt[kMaxVisual];        // L_t, then P_t
  __shared__ Lse part[kThreads / 32];
  __shared__ int bad;
  const int img = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int lo = cu[img], hi = cu[img + 1];
  int n = hi - lo - 1;
  if (threadIdx.x == 0) bad = 0;
  if (lo < 0 || hi > t_cap || n > kMaxVisual) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    n = 0;
  }
  if (n < 0) n = 0;
  int k = kreq[img];
  if (k < 0 || k > n || k > k_cap) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
    k = k < 0 ? 0 : (k > n ? n : k);
    k = k > k_cap ? k_cap : k;
  }
  const int32_t* seq = order + static_cast<size_t>(img) * k_cap;
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    s[j] = scores[lo + 1 + j];
    pos[j] = 0;
  }
  __syncthreads();
  for (int t = threadIdx.x; t < k; t += blockDim.x) {
    const int j = seq[t];
    if (j < 0 || j >= n || atomicCAS(&pos[j], 0, t + 1) != 0) bad = 1;   // range, repeats
  }
  __syncthreads();
  if (bad) {
    if (threadIdx.x == 0) {
      record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
      logp[img] = NAN;
    }
    if (grad != nullptr)
      for (int r = lo + threadIdx.x; r < hi && lo >= 0 && hi <= t_cap; r += blockDim.x)
        grad[r] = NAN;
    return;
  }
  // LSE of the kept scores
  Lse rest = lse_id();
  for (int j = threadIdx.x; j < n; j += blockDim.x)
    if (pos[j] == 0) rest = lse_merge(rest, lse_of(s[j]));
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) rest = lse_merge(rest, shfl_lse_down(rest, off));
  if (lane == 0) part[warp] = rest;
  __syncthreads();
  if (warp == 0) {
    Lse r = lane < kThreads / 32 ? part[lane] : lse_id();
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) r = lse_merge(r, shfl_lse_down(r, off));
    r = Lse{__shfl_sync(0xffffffffu, r.m, 0), __shfl_sync(0xffffffffu, r.s, 0)};
    // suffix scan over the sequence: lane handles steps [c0, c1)
    const int chunk = (k + 31) / 32;
    const int c0 = min(lane * chunk, k), c1 = min(c0 + chunk, k);
    Lse tot = lse_id();
    for (int t = c0; t < c1; ++t) tot = lse_merge(tot, lse_of(s[seq[t]]));
    Lse inc = tot;                                       // inclusive suffix over lanes
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const Lse o = shfl_lse_down(inc, off);
      if (lane + off < 32) inc = lse_merge(inc, o);
    }
    Lse above = shfl_lse_down(inc, 1);
    if (lane == 31) above = lse_id();
    Lse acc = lse_merge(r, above);
    float part_lp = 0.f;
    for (int t = c1 - 1; t >= c0; --t) {
      const float v = s[seq[t]];
      acc = lse_merge(acc, lse_of(v));
      const float L = lse_val(acc);
      lt[t] = L;
      part_lp += v - L;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) part_lp += __shfl_down_sync(0xffffffffu, part_lp, off);
    if (lane == 0) logp[img] = part_lp;
    if (grad != nullptr) {
      // prefix scan of -L_t: P_t = log sum_{u<=t} exp(-L_u)
      __syncwarp();
      Lse ptot = lse_id();
      for (int t = c0; t < c1; ++t) ptot = lse_merge(ptot, lse_of(-lt[t]));
      Lse pinc = ptot;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const Lse o = shfl_lse_up(pinc, off);
        if (lane >= off) pinc = lse_merge(o, pinc);
      }
      Lse below = shfl_lse_up(pinc, 1);
      if (lane == 0) below = lse_id();
      __syncwarp();
      Lse pacc = below;
      for (int t = c0; t < c1; ++t) {
        pacc = lse_merge(pacc, lse_of(-lt[t]));
        lt[t] = lse_val(pacc);                           // now P_t
      }
    }
  }
  __syncthreads();
  if (grad == nullptr) return;
  const float up = dlogp != nullptr ? dlogp[img] : 1.f;
  const float pk = k > 0 ? lt[k - 1] : -INFINITY;
  if (threadIdx.x == 0 && hi > lo && lo >= 0 && lo < t_cap) grad[lo] = 0.f;   // CLS
  for (int j = threadIdx.x; j < n; j += blockDim.x) {
    const int u = pos[j];
    const float g = u > 0 ? 1.f - __expf(s[j] + lt[u - 1]) : (k > 0 ? -__expf(s[j] + pk) : 0.f);
    grad[lo + 1 + j] = up * g;
  }
}

// ---------------------------------------------------------------------------
// Branching: the rows of sequences src[0..nb-1] appended after row cu[batch]
// (in place), with their ids and row moments; cu[batch + 1 + s] and the
// appended sequences' lengths (len_out) written by the single scan CTA.
// ---------------------------------------------------------------------------
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads)
    branch_cu_kernel(const int32_t* __restrict__ cu, int batch, const int32_t* __restrict__ src,
                     int nb, int t_cap, int32_t* __restrict__ cu_out,
                     int32_t* __restrict__ len_out, int32_t* status) {
  // one CTA: the appended lengths in chunks of 1024, a block-wide exclusive
  // scan per chunk carried across chunks (64-bit sums)
  __shared__ long long warp_sum[kScanThreads / 32];
  __shared__ int warp_fit[kScanThreads / 32];
  __shared__ long long carry;
  __shared__ int last_fit;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (cu_out != cu)
    for (int i = threadIdx.x; i <= batch; i += blockDim.x) cu_out[i] = cu[i];
  if (threadIdx.x == 0) {
    carry = cu[batch];
    last_fit = cu[batch] < t_cap ? cu[batch] : t_cap;
  }
  __syncthreads();
  for (int base = 0; base < nb; base += kScanThreads) {
    const int s = base + threadIdx.x;
    long long len = 0;
    if (s < nb) {
      const int b = src[s];
      if (b >= 0 && b < batch) len = cu[b + 1] - cu[b];
      else record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
      if (len < 0) len = 0;
    }
    long long inc = len;                                 // inclusive warp scan
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const long long o = __shfl_up_sync(0xffffffffu, inc, off);
      if (lane >= off) inc += o;
    }
    if (lane == 31) warp_sum[warp] = inc;
    __syncthreads();
    if (warp == 0) {
      long long w = warp_sum[lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const long long o = __shfl_up_sync(0xffffffffu, w, off);
        if (lane >= off) w += o;
      }
      warp_sum[lane] = w;                                // inclusive over warps
    }
    __syncthreads();
    const long long end = carry + (warp > 0 ? warp_sum[warp - 1] : 0) + inc;
    const bool fits = end <= t_cap;
    // the ends only grow: the last one that fits is the largest fitting end
    const int fm = __reduce_max_sync(0xffffffffu, (s < nb && fits) ? static_cast<int>(end) : 0);
    if (lane == 0) warp_fit[warp] = fm;
    __syncthreads();                                     // carry and warp_fit are read
    if (threadIdx.x == 0) {
      int m = last_fit;
      for (int w = 0; w < kScanThreads / 32; ++w) m = warp_fit[w] > m ? warp_fit[w] : m;
      last_fit = m;
    }
    __syncthreads();
    if (s < nb) {
      // the first sequence that does not fit in t_cap, and every one after
      // it, gets length 0 (its end is the last end that fits)
      if (!fits && len > 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
      cu_out[batch + 1 + s] = fits ? static_cast<int32_t>(end) : last_fit;
      if (len_out != nullptr) len_out[s] = fits ? static_cast<int32_t>(len) : 0;
    }
    if (threadIdx.x == kScanThreads - 1) carry = end;
    __syncthreads();
  }
}

__global__ void branch_rows_kernel(uint4* __restrict__ x, int32_t* __restrict__ ids,
                                   float2* __restrict__ mv, const int32_t* __restrict__ cu_out,
                                   int batch, const int32_t* __restrict__ src, int nb, int t_cap,
                                   int d8) {
  const int warps = gridDim.x * (blockDim.x >> 5);
  const int lane = threadIdx.x & 31;
  const int r0 = cu_out[batch], r1 = min(cu_out[batch + nb], t_cap);
  for (int r = r0 + blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < r1; r += warps) {
    int a = 0, b = nb - 1;                               // sequence holding row r
    while (a < b) {
      const int m = (a + b + 1) >> 1;
      if (cu_out[batch + m] <= r) a = m; else b = m - 1;
    }
    const int from = cu_out[src[a]] + (r - cu_out[batch + a]);
    const uint4* xs = x + static_cast<size_t>(from) * d8;
    uint4* xd = x + static_cast<size_t>(r) * d8;
    for (int c = lane; c < d8; c += 32) xd[c] = xs[c];
    if (lane == 0) {
      if (ids != nullptr) ids[r] = ids[from];
      if (mv != nullptr) mv[r] = mv[from];
    }
  }
}

// ---------------------------------------------------------------------------
// Fidelity cost: one warp per shadow, fp32, two passes over the true classes.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf(uint16_t v) { return __uint_as_float(static_cast<uint32_t>(v) << 16); }

__global__ void kd_cost_kernel(const uint16_t* __restrict__ zn, const uint16_t* __restrict__ z,
                               const int32_t* __restrict__ map, int shadows, int batch,
                               int classes, int ld, float inv_tau, float tau2,
                               float* __restrict__ cost, int32_t* status) {
  const int sh = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (sh >= shadows) return;
  const int img = map != nullptr ? map[sh] : sh;
  if (img < 0 || img >= batch) {
    if (lane == 0) {
      record_status(status, DORA_ERR_DEVICE_BAD_COUNT);
      cost[sh] = NAN;
    }
    return;
  }
  const uint16_t* a = zn + static_cast<size_t>(img) * ld;
  const uint16_t* b = z + static_cast<size_t>(sh) * ld;
  Lse la = lse_id(), lb = lse_id();
  for (int c = lane; c < classes; c += 32) {
    la = lse_merge(la, lse_of(bf(a[c]) * inv_tau));
    lb = lse_merge(lb, lse_of(bf(b[c]) * inv_tau));
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    la = lse_merge(la, shfl_lse_down(la, off));
    lb = lse_merge(lb, shfl_lse_down(lb, off));
  }
  const float za = __shfl_sync(0xffffffffu, lse_val(la), 0);
  const float zb = __shfl_sync(0xffffffffu, lse_val(lb), 0);
  float kl = 0.f;
  for (int c = lane; c < classes; c += 32) {
    const float lpa = bf(a[c]) * inv_tau - za, lpb = bf(b[c]) * inv_tau - zb;
    kl += __expf(lpa) * (lpa - lpb);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) kl += __shfl_down_sync(0xffffffffu, kl, off);
  if (lane == 0) cost[sh] = tau2 * kl;
}

// ---------------------------------------------------------------------------
// Local rewards: one thread per image.  D_j of pruning block j < P - 1 is the
// cost of its shadow, cost[(2 + j) B + i]; the last pruning block's prefix is
// the whole rollout, cost[i]; D_{-1} = 0.
// ---------------------------------------------------------------------------
__global__ void step_rewards_kernel(const float* __restrict__ cost,
                                    const int32_t* __restrict__ removals,
                                    const int32_t* __restrict__ blocks, int n_blocks, int batch,
                                    int depth, int n0, float a, float* __restrict__ reward,
                                    float* __restrict__ ret) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= batch) return;
  const float inv = 25.f / (static_cast<float>(depth) * static_cast<float>(n0));
  float prev = 0.f, total = 0.f;
  for (int j = 0; j < n_blocks; ++j) {
    const float d = j + 1 < n_blocks ? cost[static_cast<size_t>(2 + j) * batch + i] : cost[i];
    const float dc = static_cast<float>(removals[static_cast<size_t>(j) * batch + i]) *
                     static_cast<float>(depth - blocks[j]) * inv;
    const float r = dc - a * (d - prev);
    reward[static_cast<size_t>(j) * batch + i] = r;
    total += r;
    prev = d;
  }
  if (ret != nullptr) ret[i] = total;
}

}  // namespace train
}  // namespace dora

using namespace dora;

namespace {
int device_or_error() {
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  return DORA_OK;
}
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

extern "C" {

int dora_pl_sample(const float* scores, const float* gumbel, const int32_t* cu, int32_t batch,
                   int32_t t_cap, const int32_t* k, int32_t k_cap, int32_t* order,
                   float* keys_out, int32_t* status, dora_stream_t stream) {
  if (batch < 0 || batch > (1 << 24) || t_cap < 0 || k_cap < 1 || k_cap > train::kMaxVisual)
    return DORA_ERR_INVALID_ARG;
  if (scores == nullptr || gumbel == nullptr || cu == nullptr || k == nullptr || order == nullptr)
    return DORA_ERR_INVALID_ARG;
  const int e = device_or_error();
  if (e != DORA_OK) return e;
  if (batch == 0) return DORA_OK;
  train::pl_sample_kernel<<<batch, train::kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      scores, gumbel, cu, t_cap, k, k_cap, order, keys_out, status);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

int dora_pl_logprob(const float* scores, const int32_t* cu, int32_t batch, int32_t t_cap,
                    const int32_t* k, const int32_t* order, int32_t k_cap, float* logp,
                    float* grad, const float* dlogp, int32_t* status, dora_stream_t stream) {
  if (batch < 0 || batch > (1 << 24) || t_cap < 0 || k_cap < 1 || k_cap > train::kMaxVisual)
    return DORA_ERR_INVALID_ARG;
  if (scores == nullptr || cu == nullptr || k == nullptr || order == nullptr || logp == nullptr)
    return DORA_ERR_INVALID_ARG;
  const int e = device_or_error();
  if (e != DORA_OK) return e;
  if (batch == 0) return DORA_OK;
  train::pl_logprob_kernel<<<batch, train::kThreads, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      scores, cu, t_cap, k, order, k_cap, logp, grad, dlogp, status);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

int dora_branch(dora_bf16* x, int32_t* ids, float* x_moments, const int32_t* cu, int32_t batch,
                int32_t t_cap, int32_t dim, const int32_t* src, int32_t n_branch,
                int32_t* cu_out, int32_t* len_out, int32_t* status, dora_stream_t stream_) {
  if (batch < 1 || batch > (1 << 24) || t_cap < 0 || dim <= 0 || dim % 8 != 0 || n_branch < 0 ||
      n_branch > (1 << 20))
    return DORA_ERR_INVALID_ARG;
  if (x == nullptr || cu == nullptr || cu_out == nullptr || (n_branch > 0 && src == nullptr) ||
      !aligned16(x) || (x_moments != nullptr && (reinterpret_cast<uintptr_t>(x_moments) & 7u)))
    return DORA_ERR_INVALID_ARG;
  const int e = device_or_error();
  if (e != DORA_OK) return e;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  train::branch_cu_kernel<<<1, train::kScanThreads, 0, stream>>>(cu, batch, src, n_branch, t_cap,
                                                                  cu_out, len_out, status);
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  if (n_branch == 0) return DORA_OK;
  train::branch_rows_kernel<<<152 * 8, 256, 0, stream>>>(
      reinterpret_cast<uint4*>(x), ids, reinterpret_cast<float2*>(x_moments), cu_out, batch, src,
      n_branch, t_cap, dim / 8);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

int dora_kd_cost(const dora_bf16* z_native, const dora_bf16* z, const int32_t* shadow_image,
                 int32_t shadows, int32_t batch, int32_t classes, int32_t ld, float tau,
                 float* cost, int32_t* status, dora_stream_t stream) {
  if (shadows < 0 || batch < 1 || classes < 1 || ld < classes || !(tau > 0.f))
    return DORA_ERR_INVALID_ARG;
  if (z_native == nullptr || z == nullptr || cost == nullptr) return DORA_ERR_INVALID_ARG;
  const int e = device_or_error();
  if (e != DORA_OK) return e;
  if (shadows == 0) return DORA_OK;
  const int blocks = (shadows * 32 + 255) / 256;
  train::kd_cost_kernel<<<blocks, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(
      z_native, z, shadow_image, shadows, batch, classes, ld, 1.f / tau, tau * tau, cost, status);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

int dora_step_rewards(const float* cost, const int32_t* removals, const int32_t* blocks,
                      int32_t n_blocks, int32_t batch, int32_t depth, int32_t n0, float a,
                      float* reward, float* ret, dora_stream_t stream) {
  if (n_blocks < 1 || batch < 1 || depth < 1 || n0 < 1 || !(a == a))
    return DORA_ERR_INVALID_ARG;
  if (cost == nullptr || removals == nullptr || blocks == nullptr || reward == nullptr)
    return DORA_ERR_INVALID_ARG;
  const int e = device_or_error();
  if (e != DORA_OK) return e;
  train::step_rewards_kernel<<<(batch + 255) / 256, 256, 0,
                               reinterpret_cast<cudaStream_t>(stream)>>>(
      cost, removals, blocks, n_blocks, batch, depth, n0, a, reward, ret);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

}  // extern "C"
