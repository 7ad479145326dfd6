// The deterministic actor of DORA at deployment (Sec. 3.2 "The actor";
// Appendix A.1-A.3), at one block, for every image of a packed batch:
//   gate      p = sigmoid(MLP_G([K_CLS, e^G_l, h_l])), a (d + 19) -> 64 -> 1
//             SiLU MLP: one CTA per image;
//   encoder   X = W_in K + b_in + e^C_l (+ W_h h_l on the CLS row), then one
//             pre-LayerNorm Transformer block of width 128 (four heads of 32,
//             GELU feed-forward 128 -> 256 -> 128), run on the library's
//             tcgen05 GEMMs (LayerNorms folded in) and varlen attention;
//   budget    the highest logit of MLP_B(LayerNorm(Z_CLS)) among the budgets
//             k <= N_l - 4 (ties to the smaller), and
//   selector  s_j = MLP_S(Z_j + W_k k / N_l), a 128 -> 64 -> 1 SiLU MLP,
//             written W_1 Z_j + b_1 + (k / N_l) W_1 W_k: the first term is one
//             tcgen05 GEMM over all tokens, W_1 W_k is made once per set of
//             weights, and the rest runs per token.
// The attention kernel works on heads of 64 lanes.  The encoder's heads of 32
// are zero-padded to 64: the padded QKV rows and W_o columns are zero, so
// every score, softmax weight and head output equals that of the 32-wide head
// (the softmax scale stays 1/sqrt(32)).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "dora.h"
#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace actor {

constexpr int W = 128;          // encoder width
constexpr int HEADS = 4;
constexpr int HD = 32;          // encoder head width
constexpr int HDP = 64;         // padded head width
constexpr int FF = 256;         // feed-forward width
constexpr int GH = 64;          // gate hidden units
constexpr int GE = 16;          // gate block embedding
constexpr int SH = 64;          // selector hidden units
constexpr int kMaxDim = 2048;
constexpr int kMaxN0 = 1028;    // budget-head outputs (n0 - 4) / 2 <= 512
constexpr int kMaxBudgets = (kMaxN0 - 4) / 2;
constexpr int kGateStagedInputs = 1536;   // gate weights staged in shared memory up to d + 19 = 1536

__device__ __forceinline__ float ld(const uint16_t* __restrict__ p, size_t i) {
  return __uint_as_float(static_cast<uint32_t>(p[i]) << 16);
}
__device__ __forceinline__ uint16_t to_bf16(float v) {
  const __nv_bfloat16 h = __float2bfloat16_rn(v);
  return *reinterpret_cast<const uint16_t*>(&h);
}
__device__ __forceinline__ float silu(float x) { return x / (1.f + expf(-x)); }
__device__ __forceinline__ float gelu(float x) {
  return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ---------------------------------------------------------------------------
// preparation (once per set of weights)
// ---------------------------------------------------------------------------
// Padded QKV [768, 128]: row part * 256 + head * 64 + j takes folded row
// part * 128 + head * 32 + j for j < 32 and is zero otherwise (so are its c, d).
__global__ void pad_qkv_kernel(const uint16_t* __restrict__ wf, const float* __restrict__ cf,
                               const float* __restrict__ df, uint16_t* __restrict__ wp,
                               float* __restrict__ cp, float* __restrict__ dp) {
  const int p = blockIdx.x;
  const int part = p / (HEADS * HDP), head = (p / HDP) % HEADS, j = p % HDP;
  const bool live = j < HD;
  const int src = part * W + head * HD + j;
  for (int c = threadIdx.x; c < W; c += blockDim.x)
    wp[static_cast<size_t>(p) * W + c] = live ? wf[static_cast<size_t>(src) * W + c] : 0;
  if (threadIdx.x == 0) {
    cp[p] = live ? cf[src] : 0.f;
    dp[p] = live ? df[src] : 0.f;
  }
}

// Padded W_o [128, 256]: column head * 64 + j takes column head * 32 + j for
// j < 32 and is zero otherwise.
__global__ void pad_wo_kernel(const uint16_t* __restrict__ wo, uint16_t* __restrict__ wp) {
  const int r = blockIdx.x;
  for (int c = threadIdx.x; c < HEADS * HDP; c += blockDim.x) {
    const int head = c / HDP, j = c % HDP;
    wp[static_cast<size_t>(r) * HEADS * HDP + c] =
        j < HD ? wo[static_cast<size_t>(r) * W + head * HD + j] : 0;
  }
}

// The selector's W_1 W_k (fp32 [64]).
__global__ void sel_wk_kernel(const uint16_t* __restrict__ w1, const uint16_t* __restrict__ w_k,
                              float* __restrict__ out) {
  const int h = threadIdx.x;
  float a = 0.f;
  for (int c = 0; c < W; ++c) a = fmaf(ld(w1, static_cast<size_t>(h) * W + c), ld(w_k, c), a);
  out[h] = a;
}

// The input projection's bias at every block: bf16(b_in + e^C_l).
__global__ void bias_in_kernel(const uint16_t* __restrict__ b_in, const uint16_t* __restrict__ emb,
                               uint16_t* __restrict__ out) {
  const int l = blockIdx.x;
  for (int c = threadIdx.x; c < W; c += blockDim.x)
    out[static_cast<size_t>(l) * W + c] = to_bf16(ld(b_in, c) + ld(emb, static_cast<size_t>(l) * W + c));
}

// ---------------------------------------------------------------------------
// gate (Appendix A.1) and budget head (Sec. 3.2; Appendix A.1-A.3): one CTA per
// image.  Their weights are transposed once ([inputs, outputs]), so the
// threads computing neighbouring outputs read each input's weights together,
// and every thread keeps several independent loads in flight.
// ---------------------------------------------------------------------------
__global__ void transpose_kernel(const uint16_t* __restrict__ w, int rows, int cols,
                                 uint16_t* __restrict__ wt) {
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < rows * cols;
       idx += gridDim.x * blockDim.x) {
    const int c = idx / rows, r = idx % rows;    // wt [cols, rows]
    wt[idx] = w[static_cast<size_t>(r) * cols + c];
  }
}

// Copy n16 16-byte words from global to shared memory, 8 loads in flight.
__device__ __forceinline__ void stage(uint4* __restrict__ dst, const uint4* __restrict__ src,
                                      int n16) {
  int i = threadIdx.x;
  for (; i + 7 * static_cast<int>(blockDim.x) < n16; i += 8 * blockDim.x) {
    uint4 v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = src[i + e * blockDim.x];
#pragma unroll
    for (int e = 0; e < 8; ++e) dst[i + e * blockDim.x] = v[e];
  }
  for (; i < n16; i += blockDim.x) dst[i] = src[i];
}

// sum_c wt[c * stride + o] * v[c] over c in [c0, c1), 8 loads in flight
__device__ __forceinline__ float dot_t(const uint16_t* __restrict__ wt, int stride, int o,
                                       const float* __restrict__ v, int c0, int c1) {
  float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  int c = c0;
  for (; c + 7 < c1; c += 8) {
#pragma unroll
    for (int e = 0; e < 8; ++e) a[e] = fmaf(ld(wt, static_cast<size_t>(c + e) * stride + o), v[c + e], a[e]);
  }
  for (; c < c1; ++c) a[0] = fmaf(ld(wt, static_cast<size_t>(c) * stride + o), v[c], a[0]);
  return ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
}

// h_l = [N_l / N0, rho_l, E_<l / (L - 1)]; the gate logit and p^G; and W_h h_l
// added to the image's CLS row of the encoder input x [rows, 128].  256
// threads: hidden unit t % 64 over a quarter t / 64 of the d + 19 inputs.
__global__ void __launch_bounds__(256) gate_kernel(
    const uint16_t* __restrict__ qkv, int dim, const int32_t* __restrict__ cu, int t_cap,
    int block, int depth, int n0, const float* __restrict__ rho,
    const int32_t* __restrict__ interventions, const uint16_t* __restrict__ w1t,
    const uint16_t* __restrict__ b1, const uint16_t* __restrict__ w2,
    const uint16_t* __restrict__ b2, const uint16_t* __restrict__ emb,
    const uint16_t* __restrict__ w_h, uint16_t* __restrict__ x, float* __restrict__ glogit,
    float* __restrict__ p_gate) {
  __shared__ float z[kMaxDim + GE + 3];
  __shared__ float part[4][GH];
  extern __shared__ __align__(16) uint4 wsm[];          // W_1^T when it fits (else empty)
  const int i = blockIdx.x, t = threadIdx.x;
  const int lo = cu[i], hi = cu[i + 1];
  const int n = (lo < 0 || hi > t_cap) ? -1 : hi - lo - 1;   // visual tokens
  const int kin_ = dim + GE + 3;
  const bool staged = kin_ <= kGateStagedInputs;
  if (staged && n >= 0) stage(wsm, reinterpret_cast<const uint4*>(w1t), kin_ * GH * 2 / 16);
  if (n < 0) {                                       // empty (or outside the buffer): closed
    if (t == 0) {
      glogit[i] = -INFINITY;
      if (p_gate != nullptr) p_gate[i] = 0.f;
    }
    return;
  }
  const float h0 = static_cast<float>(n) / static_cast<float>(n0);
  const float h1 = rho[i];
  const float h2 = static_cast<float>(interventions[i]) / static_cast<float>(max(depth - 1, 1));
  const int kin = dim + GE + 3;
  const size_t krow = static_cast<size_t>(lo) * 3 * dim + dim;   // the CLS key
  for (int c = t; c < dim; c += blockDim.x) z[c] = ld(qkv, krow + c);
  if (t < GE) z[dim + t] = ld(emb, static_cast<size_t>(block) * GE + t);
  if (t == 0) {
    z[dim + GE] = h0;
    z[dim + GE + 1] = h1;
    z[dim + GE + 2] = h2;
  }
  __syncthreads();
  {
    const int h = t % GH, q = t / GH;
    const int c0 = (kin * q) / 4, c1 = (kin * (q + 1)) / 4;
    part[q][h] = dot_t(staged ? reinterpret_cast<const uint16_t*>(wsm) : w1t, GH, h, z, c0, c1);
  }
  __syncthreads();
  if (t < 32) {
    float s = 0.f;
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int h = t + 32 * e;
      s += ld(w2, h) * silu(((part[0][h] + part[1][h]) + (part[2][h] + part[3][h])) + ld(b1, h));
    }
    s = warp_sum(s);
    if (t == 0) {
      const float lg = s + ld(b2, 0);
      glogit[i] = lg;
      if (p_gate != nullptr) p_gate[i] = 1.f / (1.f + expf(-lg));
    }
  }
  // the history enters the encoder on the CLS token only
  if (t < W) {
    uint16_t* xr = x + static_cast<size_t>(lo) * W;
    const float v = ld(w_h, t * 3) * h0 + ld(w_h, t * 3 + 1) * h1 + ld(w_h, t * 3 + 2) * h2;
    xr[t] = to_bf16(ld(xr, t) + v);
  }
}

// LayerNorm(Z_CLS) -> 128 -> 128 GELU -> M logits; the highest feasible logit
// (k <= N_l - 4, ties to the smaller k) is the budget.  128 threads.
__global__ void __launch_bounds__(128) budget_kernel(
    const uint16_t* __restrict__ z, const int32_t* __restrict__ cu, int t_cap, int n0, float eps,
    const uint16_t* __restrict__ ln_w, const uint16_t* __restrict__ ln_b,
    const uint16_t* __restrict__ bw1t, const uint16_t* __restrict__ bb1,
    const uint16_t* __restrict__ bw2t, const uint16_t* __restrict__ bb2,
    const float* __restrict__ glogit, const int32_t* __restrict__ interventions,
    int32_t* __restrict__ gate, int32_t* __restrict__ budget, int32_t* __restrict__ k_out,
    int32_t* __restrict__ keep, float* __restrict__ rho_next, int32_t* __restrict__ e_next,
    float* __restrict__ scores) {
  __shared__ float u[W], hb[W], logit[kMaxBudgets];
  extern __shared__ __align__(16) uint4 bsm[];          // W_1^T [128, 128], W_2^T [128, M]
  const int i = blockIdx.x, t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int lo = cu[i], hi = cu[i + 1];
  const int n = (lo < 0 || hi > t_cap) ? -1 : hi - lo - 1;
  const int m_out = (n0 - 4) / 2;
  uint16_t* const w1s = reinterpret_cast<uint16_t*>(bsm);
  uint16_t* const w2s = w1s + W * W;
  if (n >= 0) {
    stage(bsm, reinterpret_cast<const uint4*>(bw1t), W * W * 2 / 16);
    stage(reinterpret_cast<uint4*>(w2s), reinterpret_cast<const uint4*>(bw2t), W * m_out * 2 / 16);
  }
  if (n < 0) {
    if (t == 0) {
      gate[i] = budget[i] = k_out[i] = keep[i] = 0;
      if (rho_next != nullptr) rho_next[i] = 0.f;
      if (e_next != nullptr) e_next[i] = interventions[i];
    }
    return;
  }
  const size_t zc = static_cast<size_t>(lo) * W;
  if (warp == 0) {                                   // LayerNorm(Z_CLS)
    float v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = ld(z, zc + lane + 32 * q);
    const float mean = warp_sum(v[0] + v[1] + v[2] + v[3]) * (1.f / W);
    float d2 = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) d2 += (v[q] - mean) * (v[q] - mean);
    const float rstd = rsqrtf(warp_sum(d2) * (1.f / W) + eps);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int c = lane + 32 * q;
      u[c] = (v[q] - mean) * rstd * ld(ln_w, c) + ld(ln_b, c);
    }
  }
  __syncthreads();
  hb[t] = gelu(dot_t(w1s, W, t, u, 0, W) + ld(bb1, t));
  __syncthreads();
  for (int m = t; m < m_out; m += blockDim.x) logit[m] = dot_t(w2s, m_out, m, hb, 0, W) + ld(bb2, m);
  __syncthreads();
  if (t == 0) {
    int best = -1;
    float bv = 0.f;
    for (int m = 0; m < m_out; ++m)
      if (2 * (m + 1) <= n - 4 && (best < 0 || logit[m] > bv)) {
        best = m;
        bv = logit[m];
      }
    const int bud = best < 0 ? 0 : 2 * (best + 1);
    const int g = (glogit[i] >= 0.f && bud > 0) ? 1 : 0;
    const int kk = g ? bud : 0;
    budget[i] = bud;
    gate[i] = g;
    k_out[i] = kk;
    keep[i] = n + 1 - kk;
    if (rho_next != nullptr) rho_next[i] = n > 0 ? static_cast<float>(kk) / n : 0.f;
    if (e_next != nullptr) e_next[i] = interventions[i] + g;
    scores[lo] = 0.f;
  }
}

// ---------------------------------------------------------------------------
// selector tail (Eq. 2): one thread per visual token, s = w_2 . silu(S1_j +
// (k / N_l) W_1 W_k) + b_2, with S1_j = W_1 Z_j + b_1 from the GEMM and k the
// image's budget
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) selector_kernel(
    const uint16_t* __restrict__ s1, const int32_t* __restrict__ cu, int t_cap,
    const int32_t* __restrict__ budget, const float* __restrict__ sel_wk,
    const uint16_t* __restrict__ sw2, const uint16_t* __restrict__ sb2,
    float* __restrict__ scores) {
  __shared__ float sck[SH], sw2s[SH];
  const int i = blockIdx.x, t = threadIdx.x;
  const int lo = cu[i], hi = cu[i + 1];
  const int n = (lo < 0 || hi > t_cap) ? -1 : hi - lo - 1;
  if (n <= 0) return;
  const float kr = static_cast<float>(budget[i]) / n;
  if (t < SH) {
    sck[t] = kr * sel_wk[t];
    sw2s[t] = ld(sw2, t);
  }
  __syncthreads();
  const float b2 = ld(sb2, 0);
  for (int j = 1 + t; j <= n; j += blockDim.x) {
    const uint4* sr = reinterpret_cast<const uint4*>(s1 + static_cast<size_t>(lo + j) * SH);
    float acc = 0.f;
#pragma unroll 2
    for (int q = 0; q < SH / 8; ++q) {
      const uint4 v = sr[q];
      const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int hh = 8 * q + 2 * e;
        acc = fmaf(sw2s[hh], silu(__uint_as_float(wv[e] << 16) + sck[hh]), acc);
        acc = fmaf(sw2s[hh + 1], silu(__uint_as_float(wv[e] & 0xFFFF0000u) + sck[hh + 1]), acc);
      }
    }
    scores[lo + j] = acc + b2;
  }
}

// ---------------------------------------------------------------------------
// host side: layouts
// ---------------------------------------------------------------------------
size_t up256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

struct Prep {
  size_t bias_in, wqkv_f, cqkv_f, dqkv_f, wqkv_p, cqkv_p, dqkv_p, wo_p, wfc1, cfc1, dfc1, sel_wk,
      gate_w1t, bud_w1t, bud_w2t, total;
};

Prep prep_layout(const dora_actor_weights* w) {
  Prep P{};
  size_t off = 0;
  P.bias_in = off; off += up256(static_cast<size_t>(w->depth) * W * 2);
  P.wqkv_f = off;  off += up256(3 * W * W * 2);
  P.cqkv_f = off;  off += up256(3 * W * 4);
  P.dqkv_f = off;  off += up256(3 * W * 4);
  P.wqkv_p = off;  off += up256(3 * HEADS * HDP * W * 2);
  P.cqkv_p = off;  off += up256(3 * HEADS * HDP * 4);
  P.dqkv_p = off;  off += up256(3 * HEADS * HDP * 4);
  P.wo_p = off;    off += up256(W * HEADS * HDP * 2);
  P.wfc1 = off;    off += up256(FF * W * 2);
  P.cfc1 = off;    off += up256(FF * 4);
  P.dfc1 = off;    off += up256(FF * 4);
  P.sel_wk = off;  off += up256(SH * 4);
  P.gate_w1t = off; off += up256(static_cast<size_t>(w->dim + GE + 3) * GH * 2);
  P.bud_w1t = off; off += up256(W * W * 2);
  P.bud_w2t = off; off += up256(static_cast<size_t>(W) * ((w->n0 - 4) / 2) * 2);
  P.total = off;
  return P;
}

struct Ws {
  size_t status, x, mv, qkv, o, z1, sm, f, z, s1, glogit, prep, total;
};

Ws ws_layout(int32_t t_cap, int32_t batch, const dora_actor_weights* w) {
  Ws L{};
  const size_t t = static_cast<size_t>(t_cap), b = static_cast<size_t>(batch);
  size_t off = 0;
  L.status = off; off += 256;
  L.x = off;      off += up256(t * W * 2);
  L.mv = off;     off += up256(t * 8);
  L.qkv = off;    off += up256(t * 3 * HEADS * HDP * 2);
  L.o = off;      off += up256(t * HEADS * HDP * 2);
  L.z1 = off;     off += up256(t * W * 2);
  L.sm = off;     off += up256(t * 2 * 8);
  L.f = off;      off += up256(t * FF * 2);
  L.z = off;      off += up256(t * W * 2);
  L.s1 = off;     off += up256(t * SH * 2);
  L.glogit = off; off += up256(b * 4);
  L.prep = off;   off += w->prepared != nullptr ? 0 : prep_layout(w).total;
  L.total = off;
  return L;
}

bool weights_ok(const dora_actor_weights* w) {
  if (w == nullptr) return false;
  if (w->dim <= 0 || w->dim % 64 != 0 || w->dim > kMaxDim) return false;
  if (w->depth <= 0 || w->n0 < 6 || w->n0 > kMaxN0) return false;
  if (!(w->eps >= 0.f) || !isfinite(w->eps)) return false;
  const void* req[] = {w->gate_w1, w->gate_b1, w->gate_w2, w->gate_b2, w->gate_emb,
                       w->enc_w_in, w->enc_b_in, w->enc_emb, w->enc_w_h, w->enc_ln1_w,
                       w->enc_ln1_b, w->enc_w_qkv, w->enc_b_qkv, w->enc_w_o, w->enc_b_o,
                       w->enc_ln2_w, w->enc_ln2_b, w->enc_w_fc1, w->enc_b_fc1, w->enc_w_fc2,
                       w->enc_b_fc2, w->bud_ln_w, w->bud_ln_b, w->bud_w1, w->bud_b1,
                       w->bud_w2, w->bud_b2, w->sel_w_k, w->sel_w1, w->sel_b1, w->sel_w2,
                       w->sel_b2};
  for (const void* p : req)
    if (p == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0) return false;
  return (reinterpret_cast<uintptr_t>(w->prepared) & 255u) == 0;
}

cudaError_t prepare(const dora_actor_weights* w, uint8_t* prep, cudaStream_t stream) {
  const Prep P = prep_layout(w);
  cudaError_t e = launch_fold_ln(w->enc_w_qkv, 3 * W, W, w->enc_ln1_w, w->enc_ln1_b,
                                 w->enc_b_qkv, reinterpret_cast<uint16_t*>(prep + P.wqkv_f),
                                 reinterpret_cast<float*>(prep + P.cqkv_f),
                                 reinterpret_cast<float*>(prep + P.dqkv_f), stream);
  if (e != cudaSuccess) return e;
  pad_qkv_kernel<<<3 * HEADS * HDP, 128, 0, stream>>>(
      reinterpret_cast<const uint16_t*>(prep + P.wqkv_f),
      reinterpret_cast<const float*>(prep + P.cqkv_f),
      reinterpret_cast<const float*>(prep + P.dqkv_f), reinterpret_cast<uint16_t*>(prep + P.wqkv_p),
      reinterpret_cast<float*>(prep + P.cqkv_p), reinterpret_cast<float*>(prep + P.dqkv_p));
  pad_wo_kernel<<<W, 256, 0, stream>>>(w->enc_w_o, reinterpret_cast<uint16_t*>(prep + P.wo_p));
  bias_in_kernel<<<w->depth, W, 0, stream>>>(w->enc_b_in, w->enc_emb,
                                             reinterpret_cast<uint16_t*>(prep + P.bias_in));
  sel_wk_kernel<<<1, SH, 0, stream>>>(w->sel_w1, w->sel_w_k, reinterpret_cast<float*>(prep + P.sel_wk));
  transpose_kernel<<<64, 256, 0, stream>>>(w->gate_w1, GH, w->dim + GE + 3,
                                           reinterpret_cast<uint16_t*>(prep + P.gate_w1t));
  transpose_kernel<<<64, 256, 0, stream>>>(w->bud_w1, W, W,
                                           reinterpret_cast<uint16_t*>(prep + P.bud_w1t));
  transpose_kernel<<<64, 256, 0, stream>>>(w->bud_w2, (w->n0 - 4) / 2, W,
                                           reinterpret_cast<uint16_t*>(prep + P.bud_w2t));
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_fold_ln(w->enc_w_fc1, FF, W, w->enc_ln2_w, w->enc_ln2_b, w->enc_b_fc1,
                        reinterpret_cast<uint16_t*>(prep + P.wfc1),
                        reinterpret_cast<float*>(prep + P.cfc1),
                        reinterpret_cast<float*>(prep + P.dfc1), stream);
}

}  // namespace actor
}  // namespace dora

using namespace dora;

extern "C" {

size_t dora_actor_prepared_size(const dora_actor_weights* w) {
  if (w == nullptr || w->depth <= 0) return 0;
  return actor::prep_layout(w).total;
}

size_t dora_actor_workspace_size(int32_t t_cap, int32_t batch, const dora_actor_weights* w) {
  if (w == nullptr || t_cap < 0 || batch < 0 || w->depth <= 0) return 0;
  return actor::ws_layout(t_cap, batch, w).total;
}

int dora_actor_prepare(const dora_actor_weights* w, void* prepared, size_t prepared_bytes,
                       dora_stream_t stream) {
  if (!actor::weights_ok(w) || prepared == nullptr ||
      (reinterpret_cast<uintptr_t>(prepared) & 255u) != 0 ||
      prepared_bytes < actor::prep_layout(w).total)
    return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  return actor::prepare(w, static_cast<uint8_t*>(prepared),
                        reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DORA_OK
             : DORA_ERR_CUDA;
}

int dora_actor(const dora_bf16* qkv, const int32_t* cu, int32_t batch, int32_t max_seqlen,
               int32_t t_cap, int32_t block, const dora_actor_weights* w, const float* rho,
               const int32_t* interventions, float* p_gate, int32_t* gate, int32_t* budget,
               int32_t* k, int32_t* keep_counts, float* scores, float* rho_next,
               int32_t* interventions_next, dora_bf16* z_out, void* workspace,
               size_t workspace_bytes, dora_stream_t stream_) {
  using namespace actor;
  if (!weights_ok(w)) return DORA_ERR_INVALID_ARG;
  if (batch < 0 || batch > 65535 || t_cap < 0 || max_seqlen < 0 || max_seqlen > 65535)
    return DORA_ERR_INVALID_ARG;
  if (block < 0 || block >= w->depth) return DORA_ERR_INVALID_ARG;
  if (cu == nullptr || workspace == nullptr ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return DORA_ERR_INVALID_ARG;
  if (batch > 0 && (qkv == nullptr || rho == nullptr || interventions == nullptr ||
                    gate == nullptr || budget == nullptr || k == nullptr ||
                    keep_counts == nullptr || scores == nullptr))
    return DORA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(qkv) & 15u) != 0 ||
      (reinterpret_cast<uintptr_t>(z_out) & 15u) != 0)
    return DORA_ERR_INVALID_ARG;
  const Ws L = ws_layout(t_cap, batch, w);
  if (workspace_bytes < L.total) return DORA_ERR_INVALID_ARG;
  const int dev = checked_device();
  if (dev == -1) return DORA_ERR_CUDA;
  if (dev < 0) return DORA_ERR_UNSUPPORTED;
  if (t_cap == 0 || batch == 0) return DORA_OK;

  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* status = reinterpret_cast<int32_t*>(ws + L.status);
  uint16_t* x = reinterpret_cast<uint16_t*>(ws + L.x);
  float* mv = reinterpret_cast<float*>(ws + L.mv);
  uint16_t* qkv_e = reinterpret_cast<uint16_t*>(ws + L.qkv);
  uint16_t* o_e = reinterpret_cast<uint16_t*>(ws + L.o);
  uint16_t* z1 = reinterpret_cast<uint16_t*>(ws + L.z1);
  float* sm = reinterpret_cast<float*>(ws + L.sm);
  uint16_t* f = reinterpret_cast<uint16_t*>(ws + L.f);
  uint16_t* z = z_out != nullptr ? z_out : reinterpret_cast<uint16_t*>(ws + L.z);
  float* glogit = reinterpret_cast<float*>(ws + L.glogit);
  uint8_t* prep = ws + L.prep;
  if (w->prepared != nullptr) prep = static_cast<uint8_t*>(const_cast<void*>(w->prepared));
  else if (prepare(w, prep, stream) != cudaSuccess) return DORA_ERR_CUDA;
  const Prep P = prep_layout(w);
  const int32_t* rows = cu + batch;
  const int d = w->dim;

  // X = W_in K + (b_in + e^C_l), K read in place from the block's qkv rows
  LinearEpi e_in;
  e_in.bias = reinterpret_cast<const uint16_t*>(prep + P.bias_in) + static_cast<size_t>(block) * W;
  if (launch_linear(qkv + d, t_cap, rows, d, w->enc_w_in, W, DORA_EPI_BIAS, e_in, x, status,
                    stream, 3 * d) != cudaSuccess)
    return DORA_ERR_CUDA;
  // gate, and the history term on every CLS row
  const int kin = d + GE + 3;
  const size_t gate_smem = kin <= kGateStagedInputs ? static_cast<size_t>(kin) * GH * 2 : 0;
  const size_t bud_smem = static_cast<size_t>(W) * (W + (w->n0 - 4) / 2) * 2;
  if (cudaFuncSetAttribute(gate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(gate_smem)) != cudaSuccess ||
      cudaFuncSetAttribute(budget_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(bud_smem)) != cudaSuccess)
    return DORA_ERR_CUDA;
  gate_kernel<<<batch, 256, gate_smem, stream>>>(
      qkv, d, cu, t_cap, block, w->depth, w->n0, rho, interventions,
      reinterpret_cast<const uint16_t*>(prep + P.gate_w1t), w->gate_b1, w->gate_w2, w->gate_b2,
      w->gate_emb, w->enc_w_h, x, glogit, p_gate);
  if (cudaGetLastError() != cudaSuccess) return DORA_ERR_CUDA;
  // Z1 = X + W_o Attention(LayerNorm1(X)) + b_o
  LinearEpi e_q;
  e_q.stats_in = mv;
  e_q.colsum = reinterpret_cast<const float*>(prep + P.cqkv_p);
  e_q.colbias = reinterpret_cast<const float*>(prep + P.dqkv_p);
  e_q.eps = w->eps;
  LinearEpi e_o;
  e_o.bias = w->enc_b_o;
  e_o.residual = x;
  e_o.stats_out = sm;
  e_o.slices = W / kSliceCols;
  if (launch_row_stats(x, t_cap, rows, W, mv, stream) != cudaSuccess ||
      launch_linear(x, t_cap, rows, W, reinterpret_cast<const uint16_t*>(prep + P.wqkv_p),
                    3 * HEADS * HDP, kEpiLn, e_q, qkv_e, status, stream) != cudaSuccess ||
      launch_varlen_attn(qkv_e, cu, batch, max_seqlen, t_cap, HEADS, 0.17677669529663688f, o_e,
                         status, stream) != cudaSuccess ||
      launch_linear(o_e, t_cap, rows, HEADS * HDP, reinterpret_cast<const uint16_t*>(prep + P.wo_p),
                    W, DORA_EPI_BIAS_RESIDUAL, e_o, z1, status, stream) != cudaSuccess ||
      launch_merge_moments(sm, t_cap, rows, W / kSliceCols, mv, stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  // Z = Z1 + W_2 GELU(W_1 LayerNorm2(Z1) + b_1) + b_2
  LinearEpi e_f1;
  e_f1.stats_in = mv;
  e_f1.colsum = reinterpret_cast<const float*>(prep + P.cfc1);
  e_f1.colbias = reinterpret_cast<const float*>(prep + P.dfc1);
  e_f1.eps = w->eps;
  LinearEpi e_f2;
  e_f2.bias = w->enc_b_fc2;
  e_f2.residual = z1;
  if (launch_linear(z1, t_cap, rows, W, reinterpret_cast<const uint16_t*>(prep + P.wfc1), FF,
                    kEpiLnGelu, e_f1, f, status, stream) != cudaSuccess ||
      launch_linear(f, t_cap, rows, FF, w->enc_w_fc2, W, DORA_EPI_BIAS_RESIDUAL, e_f2, z, status,
                    stream) != cudaSuccess)
    return DORA_ERR_CUDA;
  // selector's first layer on every token, then budget head and selector tail
  uint16_t* s1 = reinterpret_cast<uint16_t*>(ws + L.s1);
  LinearEpi e_s;
  e_s.bias = w->sel_b1;
  if (launch_linear(z, t_cap, rows, W, w->sel_w1, SH, DORA_EPI_BIAS, e_s, s1, status, stream) !=
      cudaSuccess)
    return DORA_ERR_CUDA;
  budget_kernel<<<batch, 128, bud_smem, stream>>>(
      z, cu, t_cap, w->n0, w->eps, w->bud_ln_w, w->bud_ln_b,
      reinterpret_cast<const uint16_t*>(prep + P.bud_w1t), w->bud_b1,
      reinterpret_cast<const uint16_t*>(prep + P.bud_w2t), w->bud_b2, glogit, interventions, gate,
      budget, k, keep_counts, rho_next,
      interventions_next, scores);
  selector_kernel<<<batch, 256, 0, stream>>>(s1, cu, t_cap, budget,
                                             reinterpret_cast<const float*>(prep + P.sel_wk),
                                             w->sel_w2, w->sel_b2, scores);
  return cudaGetLastError() == cudaSuccess ? DORA_OK : DORA_ERR_CUDA;
}

}  // extern "C"
