// Dense bf16 GEMM with fused epilogues on the 5th-generation tensor cores:
//   Y[M, N] = epi(X[M, K] W[N, K]^T + b)      (nn.Linear layout)
// used for the QKV, projection and MLP linears of the pruned block (Eq. 1).
//
// Design (one persistent CTA per SM):
//   warp 0     TMA producer: 128x64 X tile + BNx64 W tile per stage into a
//              4-stage shared-memory ring (128-byte swizzle).
//   warp 1     MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16)
//              into one of two TMEM accumulators (2 x BN fp32 columns), so
//              the epilogue of tile t overlaps the main loop of tile t+1.
//   warps 2-9  epilogue: tcgen05.ld the accumulator (each thread owns one
//              row, each warp half the columns), add bias, GELU or residual,
//              round to bf16, store.
// The live row count M may come from device memory (rows left after a
// deletion); tiles past it are never scheduled.  Every wait is bounded.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace gemm {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kStages = 4;
constexpr int kEpiWarps = 8;
constexpr int kThreads = 64 + 32 * kEpiWarps;

template <int BN>
struct Smem {
  uint16_t a[kStages][BM * BK];   // 16 KB per stage
  uint16_t b[kStages][BN * BK];   // BN * 128 B per stage
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int issued;
  int consumed;
};

template <int EPI>
__device__ __forceinline__ void epilogue_store(const uint32_t (&r)[32], uint16_t* __restrict__ Y,
                                               const uint16_t* __restrict__ bias,
                                               const uint16_t* __restrict__ R, int row, int gcol,
                                               int N) {
  float v[32];
#pragma unroll
  for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
  if (bias != nullptr) {
    const uint4* bp = reinterpret_cast<const uint4*>(bias + gcol);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint4 bb = __ldg(bp + q);
      const uint32_t* w = reinterpret_cast<const uint32_t*>(&bb);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[q * 8 + 2 * e] += bf16_lo(w[e]);
        v[q * 8 + 2 * e + 1] += bf16_hi(w[e]);
      }
    }
  }
  if constexpr (EPI == DORA_EPI_BIAS_GELU) {
#pragma unroll
    for (int e = 0; e < 32; ++e) v[e] = 0.5f * v[e] * (1.0f + erff(v[e] * 0.70710678118654752f));
  }
  const size_t off = static_cast<size_t>(row) * N + gcol;
  if constexpr (EPI == DORA_EPI_BIAS_RESIDUAL) {
    const uint4* rp = reinterpret_cast<const uint4*>(R + off);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint4 rr = __ldg(rp + q);
      const uint32_t* w = reinterpret_cast<const uint32_t*>(&rr);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        v[q * 8 + 2 * e] += bf16_lo(w[e]);
        v[q * 8 + 2 * e + 1] += bf16_hi(w[e]);
      }
    }
  }
  uint4* yp = reinterpret_cast<uint4*>(Y + off);
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint4 o;
    o.x = pack_bf16x2(v[q * 8 + 0], v[q * 8 + 1]);
    o.y = pack_bf16x2(v[q * 8 + 2], v[q * 8 + 3]);
    o.z = pack_bf16x2(v[q * 8 + 4], v[q * 8 + 5]);
    o.w = pack_bf16x2(v[q * 8 + 6], v[q * 8 + 7]);
    yp[q] = o;
  }
}

template <int BN, int EPI>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                uint16_t* __restrict__ Y, const uint16_t* __restrict__ bias,
                const uint16_t* __restrict__ R, int m_cap, const int32_t* __restrict__ m_dev,
                int N, int K, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {           // swizzled tiles need 1 KB alignment
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem<BN>& s = *reinterpret_cast<Smem<BN>*>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int M = m_cap;
  if (m_dev != nullptr) {
    const int v = *m_dev;
    M = v < 0 ? 0 : (v > m_cap ? m_cap : v);
  }
  const int n_tiles = (N + BN - 1) / BN;
  const int num_tiles = ((M + BM - 1) / BM) * n_tiles;
  const int kb_count = K / BK;
  constexpr uint32_t kTmemCols = 2 * BN;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.acc_full[i], 1);
      mbar_init(&s.acc_empty[i], kEpiWarps);
    }
    mbar_init(&s.drain, 1);
    s.abort_flag = 0;
    s.issued = 0;
    s.consumed = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) tmem_alloc(&s.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
        const int mt = tile / n_tiles;
        const int nt = tile - mt * n_tiles;
        for (int kb = 0; kb < kb_count; ++kb) {
          const int st = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&s.empty[st], ph ^ 1, abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&s.full[st], (BM + BN) * BK * 2);
          tma_load_2d(s.a[st], &tmA, &s.full[st], kb * BK, mt * BM);
          tma_load_2d(s.b[st], &tmB, &s.full[st], kb * BK, nt * BN);
          ++it;
        }
      }
      s.issued = it;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, false);
      int it = 0, ti = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x, ++ti) {
        const int acc = ti & 1;
        const uint32_t aph = (ti >> 1) & 1;
        if (!mbar_wait(&s.acc_empty[acc], aph ^ 1, abort)) break;
        tc_fence_after();
        const uint32_t d = tmem + static_cast<uint32_t>(acc * BN);
        for (int kb = 0; kb < kb_count; ++kb) {
          const int st = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&s.full[st], ph, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sdesc_sw128(smem_u32(s.a[st]), 16, 1024);
          const uint64_t bd = sdesc_sw128(smem_u32(s.b[st]), 16, 1024);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16_ss(d, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
          mma_commit(&s.empty[st]);
          ++it;
        }
        if (ok) mma_commit(&s.acc_full[acc]);
      }
      s.consumed = it;
      mma_commit(&s.drain);
      mbar_wait_limited(&s.drain, 0, kWaitLimitNs);
    }
  } else {
    const int q = warp & 3;                       // TMEM lanes this warp may read
    const int half = (warp - 2) >> 2;             // which half of the columns
    const uint32_t lane_sel = static_cast<uint32_t>(q * 32) << 16;
    int ti = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++ti) {
      const int acc = ti & 1;
      const uint32_t aph = (ti >> 1) & 1;
      if (!mbar_wait_warp(&s.acc_full[acc], aph, abort)) break;
      tc_fence_after();
      const int mt = tile / n_tiles;
      const int nt = tile - mt * n_tiles;
      const int row = mt * BM + q * 32 + lane;
#pragma unroll 1
      for (int c = 0; c < BN / 2; c += 32) {
        const int tcol = half * (BN / 2) + c;
        uint32_t r[32];
        tmem_ld32(tmem + lane_sel + static_cast<uint32_t>(acc * BN + tcol), r);
        tmem_ld_wait();
        const int gcol = nt * BN + tcol;
        if (row < M && gcol < N) epilogue_store<EPI>(r, Y, bias, R, row, gcol, N);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.acc_empty[acc]);
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (*abort) {
    if (threadIdx.x == 0) {
      record_status(status, DORA_ERR_TIMEOUT);
      // let every TMA load that was issued but never consumed land first
      for (int it = s.consumed; it < s.issued; ++it)
        mbar_wait_limited(&s.full[it % kStages], (it / kStages) & 1, 100ull * 1000 * 1000);
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

template <int BN, int EPI>
static cudaError_t launch_bn_epi(const CUtensorMap& ta, const CUtensorMap& tb, uint16_t* y,
                                 const uint16_t* bias, const uint16_t* residual, int m_cap,
                                 const int32_t* m_dev, int n, int k, int32_t* status,
                                 cudaStream_t stream) {
  const size_t smem = sizeof(Smem<BN>);
  auto kern = gemm_kernel<BN, EPI>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long tiles = static_cast<long>((m_cap + BM - 1) / BM) * ((n + BN - 1) / BN);
  const int grid = static_cast<int>(tiles < num_sms() ? tiles : num_sms());
  kern<<<grid, kThreads, smem, stream>>>(ta, tb, y, bias, residual, m_cap, m_dev, n, k, status);
  return cudaGetLastError();
}

template <int BN>
static cudaError_t launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, uint16_t* y,
                             const uint16_t* bias, const uint16_t* residual, int epi, int m_cap,
                             const int32_t* m_dev, int n, int k, int32_t* status,
                             cudaStream_t stream) {
  switch (epi) {
    case DORA_EPI_BIAS_GELU:
      return launch_bn_epi<BN, DORA_EPI_BIAS_GELU>(ta, tb, y, bias, residual, m_cap, m_dev, n, k,
                                                   status, stream);
    case DORA_EPI_BIAS_RESIDUAL:
      return launch_bn_epi<BN, DORA_EPI_BIAS_RESIDUAL>(ta, tb, y, bias, residual, m_cap, m_dev, n,
                                                       k, status, stream);
    default:
      return launch_bn_epi<BN, DORA_EPI_BIAS>(ta, tb, y, bias, residual, m_cap, m_dev, n, k,
                                              status, stream);
  }
}

}  // namespace gemm

cudaError_t launch_linear(const uint16_t* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                          const uint16_t* w, int32_t n, const uint16_t* bias,
                          const uint16_t* residual, int32_t epilogue, uint16_t* y,
                          int32_t* status, cudaStream_t stream) {
  if (m_cap == 0) return cudaSuccess;
  const int bn = (n % 256 == 0) ? 256 : 128;
  CUtensorMap ta, tb;
  if (encode_tmap_2d_bf16(&ta, x, static_cast<uint64_t>(k), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(k) * 2, gemm::BK, gemm::BM) != 0)
    return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&tb, w, static_cast<uint64_t>(k), static_cast<uint64_t>(n),
                          static_cast<uint64_t>(k) * 2, gemm::BK, static_cast<uint32_t>(bn)) != 0)
    return cudaErrorInvalidValue;
  if (bn == 256)
    return gemm::launch_bn<256>(ta, tb, y, bias, residual, epilogue, m_cap, m_dev, n, k, status,
                                stream);
  return gemm::launch_bn<128>(ta, tb, y, bias, residual, epilogue, m_cap, m_dev, n, k, status,
                              stream);
}

}  // namespace dora
