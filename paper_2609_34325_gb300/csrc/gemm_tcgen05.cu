// Dense bf16 GEMM with fused epilogues on the 5th-generation tensor cores:
//   Y[M, N] = epi(X[M, K] W[N, K]^T + b)      (nn.Linear layout)
// used for the QKV, projection and MLP linears of the pruned block (Eq. 1).
//
// Design (one persistent CTA per SM, CTAs paired in clusters of two):
//   The two CTAs of a cluster work on vertically adjacent output tiles
//   (M-tiles 2p and 2p+1 of the same N-tile), so they need the same W tile.
//   warp 0     TMA producer: the CTA's own 128x64 X tile, plus one half of the
//              shared BNx64 W tile multicast into both CTAs, per stage of a
//              4-stage shared-memory ring (128-byte swizzle).  Each W byte is
//              read from L2 once per pair.
//   warp 1     MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16)
//              into one of two TMEM accumulators (2 x BN fp32 columns), so
//              the epilogue of tile t overlaps the main loop of tile t+1.
//   epilogue warps (2 .. 1 + kEpiWarps): tcgen05.ld the accumulator (each
//              thread owns one row; the warps of a TMEM lane quarter split the
//              columns), release it once in registers, add bias, GELU or
//              residual, round to bf16, stage each 32x32 chunk in one of two
//              shared-memory buffers (64-byte swizzle) and write it with a TMA
//              tensor store.  The tile that straddles the live row count
//              stores row by row.
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
// Pair mode (BN = 256): one MMA of M = 256 spans both CTAs of the cluster,
// each holding its own 128 rows of X and one half of the W tile, so a stage is
// 32 KB instead of 48 and six fit; the shared memory read per MMA drops by a
// third.  Otherwise one MMA per CTA, with W halves multicast.
template <int BN, bool PAIR>
struct Mode {
  static constexpr bool kPair = PAIR;
  static constexpr int kStages = kPair ? 6 : 4;
  static constexpr int kBRows = kPair ? BN / 2 : BN;   // W rows held per CTA
};
// Epilogue warps per CTA (a multiple of 4: one per TMEM lane quarter) and
// staging buffers per warp, chosen per epilogue: the ALU-heavy GELU epilogue
// wants more warps, the others fewer warps with double-buffered stores.
template <int EPI>
struct EpiCfg {
  static constexpr int kWarps = EPI == DORA_EPI_BIAS_GELU ? 16 : 8;
  static constexpr int kBufs = kWarps == 16 ? 1 : 2;
  static constexpr int kThreads = 64 + 32 * kWarps;
};
constexpr int kCluster = 2;
constexpr uint16_t kPairMask = 0x3;

constexpr int kStageChunk = 32 * 32;   // one warp's 32 rows x 32 columns, bf16

template <int BN, int EPI, bool PAIR>
struct Smem {
  uint16_t a[Mode<BN, PAIR>::kStages][BM * BK];                 // 16 KB per stage
  uint16_t b[Mode<BN, PAIR>::kStages][Mode<BN, PAIR>::kBRows * BK];   // 16 or 32 KB per stage
  uint16_t out[EpiCfg<EPI>::kWarps][EpiCfg<EPI>::kBufs][kStageChunk];   // 2 KB each
  uint64_t full[Mode<BN, PAIR>::kStages];
  uint64_t empty[Mode<BN, PAIR>::kStages];
  uint64_t acc_full[2];
  uint64_t acc_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int issued;
  int consumed;
};

__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// GELU(x) = x * Phi(x), Phi(x) = (1 + erf(x / sqrt 2)) / 2, with erf from
// formula 7.1.26 of Abramowitz & Stegun, Handbook of Mathematical Functions
// (|erf error| <= 1.5e-7): for z >= 0,
//     erf(z) = 1 - t (a1 + t (a2 + t (a3 + t (a4 + t a5)))) exp(-z^2),
//     t = 1 / (1 + p z).
// With z = |x| / sqrt 2 and q = (1 - erf(z)) / 2:  Phi = 1 - q for x >= 0,
// q for x < 0.  The constants below fold in the 1/sqrt 2 and the 1/2.
// Evaluated on two values at once with the paired fp32 instructions
// (fma/mul.rn.f32x2): the epilogue's ALU work is what limits this GEMM.
__device__ __forceinline__ void gelu_erf2(float& x0, float& x1) {
  const uint64_t P2 = f2_pack(0.3275911f * 0.70710678118654752f, 0.3275911f * 0.70710678118654752f);
  const uint64_t ONE2 = f2_pack(1.0f, 1.0f);
  const uint64_t A1 = f2_pack(0.5f * 0.254829592f, 0.5f * 0.254829592f);
  const uint64_t A2 = f2_pack(0.5f * -0.284496736f, 0.5f * -0.284496736f);
  const uint64_t A3 = f2_pack(0.5f * 1.421413741f, 0.5f * 1.421413741f);
  const uint64_t A4 = f2_pack(0.5f * -1.453152027f, 0.5f * -1.453152027f);
  const uint64_t A5 = f2_pack(0.5f * 1.061405429f, 0.5f * 1.061405429f);
  const uint64_t C2 = f2_pack(-0.72134752044448170f, -0.72134752044448170f);
  const uint64_t X = f2_pack(x0, x1);
  float d0, d1;
  f2_unpack(f2_fma(P2, f2_pack(fabsf(x0), fabsf(x1)), ONE2), d0, d1);
  const uint64_t T = f2_pack(rcp_approx(d0), rcp_approx(d1));
  const uint64_t poly =
      f2_mul(T, f2_fma(T, f2_fma(T, f2_fma(T, f2_fma(T, A5, A4), A3), A2), A1));
  float e0, e1;
  f2_unpack(f2_mul(f2_mul(X, X), C2), e0, e1);
  float q0, q1;
  f2_unpack(f2_mul(poly, f2_pack(ex2_approx(e0), ex2_approx(e1))), q0, q1);
  f2_unpack(f2_mul(X, f2_pack(x0 >= 0.0f ? 1.0f - q0 : q0, x1 >= 0.0f ? 1.0f - q1 : q1)), x0, x1);
}

// Adds 8 bf16 values (one 16-byte piece) to v[0..7] in fp32 pairs.
__device__ __forceinline__ void add_bf16x8(float* v, const uint4& piece) {
  const uint32_t* w = reinterpret_cast<const uint32_t*>(&piece);
#pragma unroll
  for (int e = 0; e < 4; ++e)
    f2_unpack(f2_add(f2_pack(v[2 * e], v[2 * e + 1]), f2_pack(bf16_lo(w[e]), bf16_hi(w[e]))),
              v[2 * e], v[2 * e + 1]);
}

// Bias and GELU of one 32-column chunk of one row, in fp32.
template <int EPI>
__device__ __forceinline__ void epilogue_math(const uint32_t (&r)[32], float (&v)[32],
                                              const uint16_t* __restrict__ bias, int gcol) {
#pragma unroll
  for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
  if (bias != nullptr) {
    const uint4* bp = reinterpret_cast<const uint4*>(bias + gcol);
#pragma unroll
    for (int q = 0; q < 4; ++q) add_bf16x8(v + 8 * q, __ldg(bp + q));
  }
  if constexpr (EPI == DORA_EPI_BIAS_GELU) {
#pragma unroll
    for (int e = 0; e < 32; e += 2) gelu_erf2(v[e], v[e + 1]);
  }
}

__device__ __forceinline__ void pack_row(const float (&v)[32], uint32_t (&o)[16]) {
#pragma unroll
  for (int e = 0; e < 16; ++e) o[e] = pack_bf16x2(v[2 * e], v[2 * e + 1]);
}

template <int BN, int EPI, bool PAIR>
__global__ void __launch_bounds__(EpiCfg<EPI>::kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmY, uint16_t* __restrict__ Y,
                const uint16_t* __restrict__ bias,
                const uint16_t* __restrict__ R, int m_cap, const int32_t* __restrict__ m_dev,
                int N, int K, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {           // swizzled tiles need 1 KB alignment
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem<BN, EPI, PAIR>& s = *reinterpret_cast<Smem<BN, EPI, PAIR>*>(smem_raw);
  constexpr int kEpiWarps = EpiCfg<EPI>::kWarps;
  constexpr int kBufs = EpiCfg<EPI>::kBufs;
  constexpr int kColGroups = kEpiWarps / 4;
  constexpr int kStages = Mode<BN, PAIR>::kStages;
  constexpr bool kPair = Mode<BN, PAIR>::kPair;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  int M = m_cap;
  if (m_dev != nullptr) {
    const int v = *m_dev;
    M = v < 0 ? 0 : (v > m_cap ? m_cap : v);
  }
  // Work is a list of tile pairs: pair p covers M-tiles 2*(p / n_tiles) and
  // 2*(p / n_tiles) + 1 of N-tile p % n_tiles; CTA `rank` of cluster c takes
  // the M-tile 2*(p / n_tiles) + rank of pairs c, c + clusters, ...
  // Both CTAs of a cluster walk the same pairs in lockstep.
  const int rank = static_cast<int>(cluster_ctarank());
  const int cid = blockIdx.x / kCluster;
  const int n_clusters = gridDim.x / kCluster;
  const int n_tiles = (N + BN - 1) / BN;
  const int m_pairs = (M + 2 * BM - 1) / (2 * BM);
  const int num_pairs = m_pairs * n_tiles;
  const int kb_count = K / BK;
  constexpr uint32_t kTmemCols = 2 * BN;
  constexpr int kHalfB = BN / 2;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      // pair mode: the first CTA's MMAs release both CTAs' stages; otherwise
      // both CTAs' MMAs release a stage (its W halves came from both)
      mbar_init(&s.empty[i], kPair ? 1 : kCluster);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.acc_full[i], 1);
      // pair mode: the epilogues of both CTAs hand the accumulator back to the first
      mbar_init(&s.acc_empty[i], kPair ? 2 * kEpiWarps : kEpiWarps);
    }
    mbar_init(&s.drain, 1);
    s.abort_flag = 0;
    s.issued = 0;
    s.consumed = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmY);
  }
  if (warp == 1) {
    if constexpr (kPair) tmem_alloc_pair(&s.tmem_base, kTmemCols);
    else tmem_alloc(&s.tmem_base, kTmemCols);
  }
  tc_fence_before();
  cluster_sync();              // peers' barriers are initialised before any multicast
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int pr = cid; ok && pr < num_pairs; pr += n_clusters) {
        const int mt = 2 * (pr / n_tiles) + rank;
        const int nt = pr % n_tiles;
        for (int kb = 0; kb < kb_count; ++kb) {
          const int st = it % kStages;
          const uint32_t ph = (it / kStages) & 1;
          if (!mbar_wait(&s.empty[st], ph ^ 1, abort)) {
            ok = false;
            break;
          }
          if constexpr (kPair) {
            // this CTA's X rows and half of the W tile; the bytes of both CTAs
            // are counted on the first CTA's barrier, which its MMA waits on
            if (rank == 0) mbar_arrive_expect_tx(&s.full[st], 2 * (BM + Mode<BN, PAIR>::kBRows) * BK * 2);
            tma_load_2d_pair(s.a[st], &tmA, &s.full[st], 0, kb * BK, mt * BM);
            tma_load_2d_pair(s.b[st], &tmB, &s.full[st], 0, kb * BK, nt * BN + rank * kHalfB);
          } else {
            mbar_arrive_expect_tx(&s.full[st], (BM + BN) * BK * 2);
            tma_load_2d(s.a[st], &tmA, &s.full[st], kb * BK, mt * BM);
            tma_load_2d_multicast(s.b[st] + rank * kHalfB * BK, &tmB, &s.full[st], kb * BK,
                                  nt * BN + rank * kHalfB, kPairMask);
          }
          ++it;
        }
      }
      s.issued = it;
    }
  } else if (warp == 1) {
    if (lane == 0 && kPair && rank == 0) {
      // pair MMA issuer: M = 256 over both CTAs, D in both CTAs' TMEM
      constexpr uint32_t idesc = idesc_bf16(2 * BM, BN, false);
      int it = 0, ti = 0;
      bool ok = true;
      for (int pr = cid; ok && pr < num_pairs; pr += n_clusters, ++ti) {
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
            mma_bf16_ss_pair(d, ad + 2 * k, bd + 2 * k, idesc, (kb | k) != 0 ? 1u : 0u);
          mma_commit_pair(&s.empty[st], kPairMask);        // both CTAs' stages free
          ++it;
        }
        if (ok) mma_commit_pair(&s.acc_full[acc], kPairMask);
      }
      s.consumed = it;
      mma_commit_pair(&s.drain, 0x1);
      mbar_wait_limited(&s.drain, 0, kWaitLimitNs);
    } else if (lane == 0) {
     if constexpr (!kPair) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, false);
      int it = 0, ti = 0;
      bool ok = true;
      for (int pr = cid; ok && pr < num_pairs; pr += n_clusters, ++ti) {
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
          mma_commit_multicast(&s.empty[st], kPairMask);   // both CTAs' W halves free
          ++it;
        }
        if (ok) mma_commit(&s.acc_full[acc]);
      }
      s.consumed = it;
      mma_commit(&s.drain);
      mbar_wait_limited(&s.drain, 0, kWaitLimitNs);
     }
    }
  } else {
    constexpr int kCols = BN / kColGroups;        // columns per epilogue warp
    constexpr int kChunks = kCols / 32;
    constexpr int kBatch = kChunks < 2 ? kChunks : 2;   // chunks per TMEM load
    const int q = warp & 3;                       // TMEM lanes this warp may read
    const int slot = (warp - 2) >> 2;             // which column slice
    const uint32_t lane_sel = static_cast<uint32_t>(q * 32) << 16;
    int buf = 0;                                  // staging buffer to write next
    int ti = 0;
    for (int pr = cid; pr < num_pairs; pr += n_clusters, ++ti) {
      const int acc = ti & 1;
      const uint32_t aph = (ti >> 1) & 1;
      if (!mbar_wait_warp(&s.acc_full[acc], aph, abort)) break;
      tc_fence_after();
      const int mt = 2 * (pr / n_tiles) + rank;
      const int nt = pr % n_tiles;
      const int row0 = mt * BM + q * 32;          // first row of this warp
      const int row = row0 + lane;
      const bool whole = row0 + 32 <= M;          // all 32 rows live: TMA store
#pragma unroll 1
      for (int cb = 0; cb < kChunks; cb += kBatch) {
        // Residual of whole 32-row chunks: loaded by the warp together, 8 rows
        // x 64 contiguous bytes per instruction (piece p = lane + 32 i is
        // row p / 4, 16-byte piece p % 4), before the TMEM load so its
        // latency overlaps; it is transposed to rows through shared memory.
        uint4 res[kBatch][4];
        if constexpr (EPI == DORA_EPI_BIAS_RESIDUAL) {
          if (whole) {
#pragma unroll
            for (int c = 0; c < kBatch; ++c) {
              const int gcol = nt * BN + slot * kCols + (cb + c) * 32;
              if (gcol < N) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  const int pc = lane + 32 * i;
                  res[c][i] = __ldg(reinterpret_cast<const uint4*>(
                                        R + static_cast<size_t>(row0 + (pc >> 2)) * N + gcol) +
                                    (pc & 3));
                }
              }
            }
          }
        }
        uint32_t r[kBatch][32];
#pragma unroll
        for (int c = 0; c < kBatch; ++c)
          tmem_ld32(tmem + lane_sel +
                        static_cast<uint32_t>(acc * BN + slot * kCols + (cb + c) * 32),
                    r[c]);
        tmem_ld_wait();
        if (cb + kBatch == kChunks) {
          // the accumulator is in registers: hand it back to the MMA warp
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (kPair && rank != 0) mbar_arrive_remote(&s.acc_empty[acc], 0);
            else mbar_arrive(&s.acc_empty[acc]);
          }
        }
#pragma unroll
        for (int c = 0; c < kBatch; ++c) {
          const int gcol = nt * BN + slot * kCols + (cb + c) * 32;
          if (gcol >= N || row0 >= M) continue;    // warp-uniform
          float v[32];
          uint32_t o[16];
          epilogue_math<EPI>(r[c], v, bias, gcol);
          if (whole) {
            // row `lane` of the 32x32 chunk, 64-byte swizzle: 16-byte piece j
            // of row l sits at piece j ^ ((l >> 1) & 3).  The store issued
            // kBufs chunks ago from this buffer must have read it.
            uint16_t* stage = s.out[warp - 2][buf];
            uint8_t* base = reinterpret_cast<uint8_t*>(stage);
            if (lane == 0) {
              if constexpr (kBufs == 2) bulk_wait_group_read1();
              else bulk_wait_group_read0();
            }
            __syncwarp();
            uint8_t* rowp = base + lane * 64;
            if constexpr (EPI == DORA_EPI_BIAS_RESIDUAL) {
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int pc = lane + 32 * i, rr = pc >> 2, j = pc & 3;
                *reinterpret_cast<uint4*>(base + rr * 64 + ((j ^ ((rr >> 1) & 3)) << 4)) =
                    res[c][i];
              }
              __syncwarp();
#pragma unroll
              for (int j = 0; j < 4; ++j)
                add_bf16x8(v + 8 * j,
                           *reinterpret_cast<const uint4*>(rowp + ((j ^ ((lane >> 1) & 3)) << 4)));
            }
            pack_row(v, o);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              *reinterpret_cast<uint4*>(rowp + ((j ^ ((lane >> 1) & 3)) << 4)) =
                  make_uint4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmY, stage, gcol, row0);
              bulk_commit_group();
            }
            buf = (buf + 1) % kBufs;
          } else if (row < M) {
            if constexpr (EPI == DORA_EPI_BIAS_RESIDUAL) {
              const uint4* rp = reinterpret_cast<const uint4*>(R + static_cast<size_t>(row) * N + gcol);
#pragma unroll
              for (int j = 0; j < 4; ++j) add_bf16x8(v + 8 * j, __ldg(rp + j));
            }
            pack_row(v, o);
            uint4* yp = reinterpret_cast<uint4*>(Y + static_cast<size_t>(row) * N + gcol);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              yp[j] = make_uint4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
          }
        }
      }
    }
    if (lane == 0) bulk_wait_group0();             // stores done before the CTA exits
    __syncwarp();
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (*abort) {
    if (threadIdx.x == 0) {
      record_status(status, DORA_ERR_TIMEOUT);
      // let every TMA load that was issued but never consumed land first
      if (!kPair || rank == 0)
        for (int it = s.consumed; it < s.issued; ++it)
          mbar_wait_limited(&s.full[it % kStages], (it / kStages) & 1, 100ull * 1000 * 1000);
      __nanosleep(50000);      // the peer's last multicast halves
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair) tmem_dealloc_pair(tmem, kTmemCols);
    else tmem_dealloc(tmem, kTmemCols);
  }
  cluster_sync();              // no CTA leaves while its peer may still signal it
}

template <int BN, int EPI, bool PAIR>
static cudaError_t launch_bn_epi(const CUtensorMap& ta, const CUtensorMap& tb,
                                 const CUtensorMap& ty, uint16_t* y,
                                 const uint16_t* bias, const uint16_t* residual, int m_cap,
                                 const int32_t* m_dev, int n, int k, int32_t* status,
                                 cudaStream_t stream) {
  const size_t smem = sizeof(Smem<BN, EPI, PAIR>);
  auto kern = gemm_kernel<BN, EPI, PAIR>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(EpiCfg<EPI>::kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // as many co-resident clusters as fit, capped by the tile pairs of m_cap
  static int max_clusters[64] = {0};   // per instantiation and device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) dev = 0;
  if (max_clusters[dev] == 0) {
    cfg.gridDim = dim3(kCluster * (num_sms() / kCluster));
    int c = 0;
    e = cudaOccupancyMaxActiveClusters(&c, kern, &cfg);
    if (e != cudaSuccess) return e;
    max_clusters[dev] = c > 0 ? c : 1;
  }
  const long pairs =
      static_cast<long>((m_cap + 2 * BM - 1) / (2 * BM)) * ((n + BN - 1) / BN);
  const long clusters = pairs < max_clusters[dev] ? pairs : max_clusters[dev];
  cfg.gridDim = dim3(static_cast<unsigned>(kCluster * clusters));
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, ty, y, bias, residual, m_cap, m_dev, n, k,
                            status);
}

// Pair mode for BN = 256, except for the residual epilogue over a short K
// (the projection linear), whose epilogue traffic then dominates: measured
// slower in pair mode.
template <int BN>
static cudaError_t launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& ty,
                             uint16_t* y,
                             const uint16_t* bias, const uint16_t* residual, int epi, int m_cap,
                             const int32_t* m_dev, int n, int k, int32_t* status,
                             cudaStream_t stream) {
  switch (epi) {
    case DORA_EPI_BIAS_GELU:
      return launch_bn_epi<BN, DORA_EPI_BIAS_GELU, BN == 256>(ta, tb, ty, y, bias, residual, m_cap,
                                                              m_dev, n, k, status, stream);
    case DORA_EPI_BIAS_RESIDUAL:
      if (BN == 256 && k > 1024)
        return launch_bn_epi<BN, DORA_EPI_BIAS_RESIDUAL, BN == 256>(ta, tb, ty, y, bias, residual,
                                                                    m_cap, m_dev, n, k, status, stream);
      return launch_bn_epi<BN, DORA_EPI_BIAS_RESIDUAL, false>(ta, tb, ty, y, bias, residual, m_cap,
                                                              m_dev, n, k, status, stream);
    default:
      return launch_bn_epi<BN, DORA_EPI_BIAS, BN == 256>(ta, tb, ty, y, bias, residual, m_cap, m_dev,
                                                         n, k, status, stream);
  }
}

}  // namespace gemm

cudaError_t launch_linear(const uint16_t* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                          const uint16_t* w, int32_t n, const uint16_t* bias,
                          const uint16_t* residual, int32_t epilogue, uint16_t* y,
                          int32_t* status, cudaStream_t stream) {
  if (m_cap == 0) return cudaSuccess;
  const int bn = (n % 256 == 0) ? 256 : 128;
  CUtensorMap ta, tb, ty;
  if (encode_tmap_2d_bf16(&ta, x, static_cast<uint64_t>(k), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(k) * 2, gemm::BK, gemm::BM) != 0)
    return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&tb, w, static_cast<uint64_t>(k), static_cast<uint64_t>(n),
                          static_cast<uint64_t>(k) * 2, gemm::BK, static_cast<uint32_t>(bn / 2)) != 0)
    return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&ty, y, static_cast<uint64_t>(n), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(n) * 2, 32, 32, 64) != 0)
    return cudaErrorInvalidValue;
  if (bn == 256)
    return gemm::launch_bn<256>(ta, tb, ty, y, bias, residual, epilogue, m_cap, m_dev, n, k, status,
                                stream);
  return gemm::launch_bn<128>(ta, tb, ty, y, bias, residual, epilogue, m_cap, m_dev, n, k, status,
                              stream);
}

}  // namespace dora
