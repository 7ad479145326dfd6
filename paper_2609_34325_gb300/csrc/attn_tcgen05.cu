// Packed variable-length multi-head self-attention on tcgen05 tensor cores.
// For image i (rows [cu[i], cu[i+1]) of the packed buffer) and head h:
//     O = softmax(Q K^T * scale) V
// with no attention across images and no padding (Sec. 3.5 "Inference").
//
// One CTA per (128-row query tile, head, image); two CTAs share an SM.
//   warp 0     TMA: Q tile once, then K/V tiles of 128 rows into a 2-stage ring.
//   warp 1     MMA: S = Q K^T (M=128, N=valid keys rounded to 16, K=64) into
//              TMEM columns [0,128); O_j = P V (M=128, N=64, K=keys) into TMEM
//              columns [128,192).
//   warps 2-5  softmax, one thread per query row (TMEM lane): row max, exp2,
//              row sum, P written to shared memory in the 128-byte-swizzled
//              K-major layout the MMA reads; the partial O_j of every key tile
//              is folded into fp32 registers with the online-softmax rescale.
// Keys past the image end (the tile reads into the next image or past the
// buffer) are masked to -inf in S, their P entries are 0, and the matching V
// rows are zeroed in shared memory so stale data cannot leak through 0 * NaN.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace attn {

constexpr int BQ = 128;
constexpr int BKV = 128;
constexpr int HD = 64;
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kTmemO = 128;

struct Smem {
  uint16_t q[BQ * HD];          // 16 KB
  uint16_t k[2][BKV * HD];      // 2 x 16 KB
  uint16_t v[2][BKV * HD];      // 2 x 16 KB
  uint16_t p[2][BQ * 64];       // P key columns [0,64) and [64,128): 2 x 16 KB
  uint64_t q_full;
  uint64_t kv_full[2];
  uint64_t kv_empty[2];
  uint64_t s_full;
  uint64_t s_free;
  uint64_t p_full;
  uint64_t o_full;
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int issued;
  int consumed;
};

__global__ void __launch_bounds__(kThreads, 2)
    varlen_attn_kernel(const __grid_constant__ CUtensorMap tm, const int32_t* __restrict__ cu,
                       int max_seqlen, int t_cap, int heads, float scale_log2,
                       uint16_t* __restrict__ out, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const int qt = blockIdx.x;
  const int h = blockIdx.y;
  const int img = blockIdx.z;
  const int lo = cu[img];
  int n = cu[img + 1] - lo;
  if (lo < 0 || lo > t_cap || n > t_cap - lo) {      // boundaries past the buffer: clamp
    if (qt == 0 && threadIdx.x == 0) record_status(status, DORA_ERR_DEVICE_SEQLEN);
    n = (lo < 0 || lo > t_cap) ? 0 : t_cap - lo;
  }
  if (qt == 0 && threadIdx.x == 0 && n > max_seqlen) record_status(status, DORA_ERR_DEVICE_SEQLEN);
  if (n <= 0 || qt * BQ >= n) return;
  if (smem_u32(smem_raw) & 1023u) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem& s = *reinterpret_cast<Smem*>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int dim = heads * HD;
  const int n_kv = (n + BKV - 1) / BKV;
  const int q0 = lo + qt * BQ;
  const int q_rows = min(BQ, n - qt * BQ);

  if (threadIdx.x == 0) {
    mbar_init(&s.q_full, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.kv_full[i], 1);
      mbar_init(&s.kv_empty[i], 1);
    }
    mbar_init(&s.s_full, 1);
    mbar_init(&s.s_free, 128);
    mbar_init(&s.p_full, 128);
    mbar_init(&s.o_full, 1);
    mbar_init(&s.drain, 1);
    s.abort_flag = 0;
    s.issued = 0;
    s.consumed = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tm);
  }
  if (warp == 1) tmem_alloc(&s.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(&s.q_full, BQ * HD * 2);
      tma_load_2d(s.q, &tm, &s.q_full, h * HD, q0);
      int j = 0;
      for (; j < n_kv; ++j) {
        const int st = j & 1;
        const uint32_t ph = (j >> 1) & 1;
        if (!mbar_wait(&s.kv_empty[st], ph ^ 1, abort)) break;
        mbar_arrive_expect_tx(&s.kv_full[st], 2 * BKV * HD * 2);
        tma_load_2d(s.k[st], &tm, &s.kv_full[st], dim + h * HD, lo + j * BKV);
        tma_load_2d(s.v[st], &tm, &s.kv_full[st], 2 * dim + h * HD, lo + j * BKV);
      }
      s.issued = j;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int j = 0;
      if (mbar_wait(&s.q_full, 0, abort)) {
        const uint64_t qd = sdesc_sw128(smem_u32(s.q), 16, 1024);
        constexpr uint32_t id_o = idesc_bf16(BQ, HD, true);
        for (; j < n_kv; ++j) {
          const int st = j & 1;
          const uint32_t ph = (j >> 1) & 1;
          const int valid = min(BKV, n - j * BKV);
          const int nm = (valid + 15) & ~15;
          if (!mbar_wait(&s.kv_full[st], ph, abort)) break;
          if (j > 0 && !mbar_wait(&s.s_free, (j - 1) & 1, abort)) break;
          tc_fence_after();
          const uint64_t kd = sdesc_sw128(smem_u32(s.k[st]), 16, 1024);
          const uint32_t id_s = idesc_bf16(BQ, nm, false);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16_ss(tmem, qd + 2 * kk, kd + 2 * kk, id_s, kk > 0 ? 1u : 0u);
          mma_commit(&s.s_full);
          if (!mbar_wait(&s.p_full, j & 1, abort)) break;
          tc_fence_after();
          const uint32_t vbase = smem_u32(s.v[st]);
          for (int kk = 0; kk < nm / 16; ++kk) {
            const uint64_t pd =
                sdesc_sw128(smem_u32(s.p[kk >> 2]) + static_cast<uint32_t>((kk & 3) * 32), 16, 1024);
            const uint64_t vd = sdesc_sw128(vbase + static_cast<uint32_t>(kk * 16 * 128), 1024, 1024);
            mma_bf16_ss(tmem + kTmemO, pd, vd, id_o, kk > 0 ? 1u : 0u);
          }
          mma_commit(&s.o_full);
          mma_commit(&s.kv_empty[st]);
        }
      }
      s.consumed = j;
      mma_commit(&s.drain);
      mbar_wait_limited(&s.drain, 0, kWaitLimitNs);
    }
  } else {
    // softmax: thread <-> query row r of the tile (TMEM lane r)
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    float o[HD];
#pragma unroll
    for (int d = 0; d < HD; ++d) o[d] = 0.f;
    float m_run = -INFINITY, l_run = 0.f, alpha_pending = 0.f;
    bool ok = true;
    for (int j = 0; j < n_kv; ++j) {
      const int st = j & 1;
      const int valid = min(BKV, n - j * BKV);
      const int nm = (valid + 15) & ~15;
      const int nc = (valid + 31) & ~31;
      if (!mbar_wait_warp(&s.s_full, j & 1, abort)) { ok = false; break; }
      tc_fence_after();
      float mx = -INFINITY;
      for (int c = 0; c < nc; c += 32) {
        uint32_t sr[32];
        tmem_ld32(tmem + lane_sel + static_cast<uint32_t>(c), sr);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (c + e < valid) mx = fmaxf(mx, __uint_as_float(sr[e]));
      }
      const float m_new = fmaxf(m_run, mx * scale_log2);
      if (j > 0) {
        // P and O of the previous key tile are free once its PV product is done
        if (!mbar_wait_warp(&s.o_full, (j - 1) & 1, abort)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < HD; c += 32) {
          uint32_t orr[32];
          tmem_ld32(tmem + lane_sel + kTmemO + static_cast<uint32_t>(c), orr);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[c + e] = o[c + e] * alpha_pending + __uint_as_float(orr[e]);
        }
      }
      const float alpha = ex2_approx(m_run - m_new);
      float lsum = 0.f;
      for (int c = 0; c < nc; c += 32) {
        uint32_t sr[32];
        tmem_ld32(tmem + lane_sel + static_cast<uint32_t>(c), sr);
        tmem_ld_wait();
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const float p0 = (c + e < valid) ? ex2_approx(__uint_as_float(sr[e]) * scale_log2 - m_new) : 0.f;
          const float p1 =
              (c + e + 1 < valid) ? ex2_approx(__uint_as_float(sr[e + 1]) * scale_log2 - m_new) : 0.f;
          lsum += p0 + p1;
          pk[e >> 1] = pack_bf16x2(p0, p1);
        }
#pragma unroll
        for (int qd = 0; qd < 4; ++qd) {
          const int chunk = (c >> 3) + qd;          // 16-byte chunk among the 16 of a P row
          uint8_t* base = reinterpret_cast<uint8_t*>(s.p[chunk >> 3]);
          uint4* dst = reinterpret_cast<uint4*>(base + r * 128 + (((chunk & 7) ^ (r & 7)) << 4));
          *dst = make_uint4(pk[qd * 4 + 0], pk[qd * 4 + 1], pk[qd * 4 + 2], pk[qd * 4 + 3]);
        }
      }
      l_run = l_run * alpha + lsum;
      m_run = m_new;
      alpha_pending = alpha;
      // zero V rows [valid, nm) of this stage: they are read by the PV product
      bool vz_ok = true;
      if (r >= valid && r < nm) vz_ok = mbar_wait(&s.kv_full[st], (j >> 1) & 1, abort);
      if (!__all_sync(0xffffffffu, vz_ok)) { ok = false; break; }
      if (r >= valid && r < nm) {
        uint4* vrow = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(s.v[st]) + r * 128);
#pragma unroll
        for (int qd = 0; qd < 8; ++qd) vrow[qd] = make_uint4(0u, 0u, 0u, 0u);
      }
      tc_fence_before();
      mbar_arrive(&s.s_free);
      fence_proxy_async_smem();
      mbar_arrive(&s.p_full);
    }
    if (ok && mbar_wait_warp(&s.o_full, (n_kv - 1) & 1, abort)) {
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < HD; c += 32) {
        uint32_t orr[32];
        tmem_ld32(tmem + lane_sel + kTmemO + static_cast<uint32_t>(c), orr);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) o[c + e] = o[c + e] * alpha_pending + __uint_as_float(orr[e]);
      }
      if (r < q_rows) {
        const float inv = 1.0f / l_run;
        uint4* dst = reinterpret_cast<uint4*>(out + static_cast<size_t>(q0 + r) * dim + h * HD);
#pragma unroll
        for (int qd = 0; qd < 8; ++qd) {
          dst[qd] = make_uint4(pack_bf16x2(o[qd * 8 + 0] * inv, o[qd * 8 + 1] * inv),
                               pack_bf16x2(o[qd * 8 + 2] * inv, o[qd * 8 + 3] * inv),
                               pack_bf16x2(o[qd * 8 + 4] * inv, o[qd * 8 + 5] * inv),
                               pack_bf16x2(o[qd * 8 + 6] * inv, o[qd * 8 + 7] * inv));
        }
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (*abort) {
    if (threadIdx.x == 0) {
      record_status(status, DORA_ERR_TIMEOUT);
      mbar_wait_limited(&s.q_full, 0, 100ull * 1000 * 1000);
      for (int j = s.consumed; j < s.issued; ++j)
        mbar_wait_limited(&s.kv_full[j & 1], (j >> 1) & 1, 100ull * 1000 * 1000);
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace attn

cudaError_t launch_varlen_attn(const uint16_t* qkv, const int32_t* cu, int32_t batch,
                               int32_t max_seqlen, int32_t t_cap, int32_t heads, float scale,
                               uint16_t* out, int32_t* status, cudaStream_t stream) {
  if (batch == 0 || t_cap == 0 || max_seqlen == 0) return cudaSuccess;
  CUtensorMap tm;
  const uint64_t row = static_cast<uint64_t>(3) * heads * attn::HD;
  if (encode_tmap_2d_bf16(&tm, qkv, row, static_cast<uint64_t>(t_cap), row * 2, attn::HD,
                          attn::BQ) != 0)
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(attn::Smem);
  cudaError_t e = cudaFuncSetAttribute(attn::varlen_attn_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const dim3 grid((max_seqlen + attn::BQ - 1) / attn::BQ, heads, batch);
  const float scale_log2 = scale * 1.4426950408889634f;
  attn::varlen_attn_kernel<<<grid, attn::kThreads, smem, stream>>>(tm, cu, max_seqlen, t_cap,
                                                                    heads, scale_log2, out, status);
  return cudaGetLastError();
}

}  // namespace dora
