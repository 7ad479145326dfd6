// Dense bf16 GEMM with fused epilogues on the 5th-generation tensor cores:
//   Y[M, N] = epi(X[M, K] W[N, K]^T + b)      (nn.Linear layout)
// used for the QKV, projection and MLP linears of the pruned block (Eq. 1).
// The LayerNorm before the QKV and fc1 linears is folded in: with W' = W
// diag(gamma) (bf16), c = W' 1 and d = W beta + b,
//   LayerNorm(x) W^T + b = rstd (x W'^T - mean c) + d,
// so the GEMM reads the raw rows and the epilogue applies each row's mean and
// rstd = 1/sqrt(var + eps) from the row moments (mean, var) written with the
// rows; the residual epilogue writes the 64-column slice moments they are
// merged from.
//
// Design (one persistent CTA per SM, CTAs paired in clusters of two):
//   The two CTAs of a cluster work on vertically adjacent output tiles
//   (M-tiles 2p and 2p+1 of the same N-tile), so they need the same W tile.
//   warp 0     TMA producer: the CTA's own 128x64 X tile and its part of the
//              BNx64 W tile, per stage of a shared-memory ring (128-byte
//              swizzle).  256-wide tiles run as a CTA pair (below), each CTA
//              loading half of W; narrower tiles load the whole W tile in each
//              CTA (both CTAs of a cluster read the same W tile, so the second
//              read is an L2 hit).
//   warp 1     MMA issuer: one thread issues tcgen05.mma (M=128, N=BN, K=16,
//              or M=256 across the pair) into one of two TMEM accumulators
//              (2 x BN fp32 columns), so the epilogue of tile t overlaps the
//              main loop of tile t+1.
//   epilogue warps (2 .. 1 + kEpiWarps): tcgen05.ld the accumulator (each
//              thread owns one row; the warps of a TMEM lane quarter split the
//              columns), release it once in registers, add bias, GELU or
//              residual, round to bf16, stage each 32x32 chunk in shared
//              memory (64-byte swizzle) and write it with a TMA tensor store.
//              The residual epilogue gives each chunk its own buffer, into
//              which a TMA load brings the residual chunk while the tile's
//              MMAs still run; the result is written over it in place (a
//              long-K linear keeps two buffers a warp and reloads them within
//              the tile, for one more stage).  The tile that straddles the
//              live row count stores row by row.
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
constexpr int kCluster = 2;
constexpr int kStageChunk = 32 * 32;   // one warp's 32 rows x 32 columns, bf16
constexpr int kSmemLimit = 227 * 1024;
// The residual epilogue of a long-K linear (K >= kLongK, fc2): two staging
// buffers per epilogue warp instead of one per chunk, so the stage ring gets
// one more stage.  The residual of a tile's first two chunks is loaded a tile
// ahead as in the plain residual epilogue; that of the other two is loaded
// into the first two's buffers once their stores have read them, inside an
// epilogue that a long main loop leaves mostly idle.
constexpr int kEpiResidualLongK = 5;
constexpr int kLongK = 2048;

// Per-instantiation layout.
// Pair mode: one MMA of M = 256 spans both CTAs of the cluster, each holding
// its own 128 rows of X and one half of the W tile, so a stage is 32 KB
// instead of 48; the shared memory read per MMA drops by a third.  Otherwise
// one MMA per CTA on a whole W tile of its own.
// Epilogue warps: a multiple of 4 (one per TMEM lane quarter); the ALU-heavy
// plain GELU epilogue gets 16, the others 8 with two staging buffers per warp
// (the residual epilogue one per chunk).  The stages fill what shared memory is left.
template <int BN, int EPI, bool PAIR>
struct Cfg {
  static constexpr bool kPair = PAIR;
  static constexpr int kBRows = kPair ? BN / 2 : BN;   // W rows held per CTA
  static constexpr bool kLn = EPI == kEpiLn || EPI == kEpiLnGelu;
  // the two GELU epilogues are ALU-bound: 16 warps; the others 8
  static constexpr int kEpiWarps = (EPI == DORA_EPI_BIAS_GELU || EPI == kEpiLnGelu) ? 16 : 8;
  static constexpr int kColGroups = kEpiWarps / 4;
  static constexpr int kCols = BN / kColGroups;         // columns per epilogue warp
  static constexpr int kChunks = kCols / 32;
  // chunks per TMEM load: two (64 registers) unless 16 warps cap registers at 96
  static constexpr int kBatch = kEpiWarps == 16 ? 1 : (kChunks < 2 ? kChunks : 2);
  static constexpr bool kResTma = EPI == DORA_EPI_BIAS_RESIDUAL || EPI == kEpiResidualLongK;
  // staging buffers per epilogue warp: one per chunk for the residual (its
  // TMA load lands there; two for a long K), one with 16 warps or the folded
  // LayerNorm, else two
  static constexpr int kBufs =
      kResTma ? (EPI == kEpiResidualLongK && kChunks > 2 ? 2 : kChunks)
              : ((kEpiWarps == 16 || kLn) ? 1 : 2);
  // folded LayerNorm: each epilogue warp's c and d columns, staged per tile
  static constexpr int kCdCols = kLn ? kCols : 1;
  static constexpr int kThreads = 64 + 32 * kEpiWarps;
  static constexpr int kStageBytes = (BM + kBRows) * BK * 2;
  static constexpr int kOutBytes = kEpiWarps * (kBufs * kStageChunk * 2 + 2 * kCdCols * 4);
  static constexpr int kFit = (kSmemLimit - 1024 - kOutBytes) / kStageBytes;
  static constexpr int kStages = kFit < 6 ? kFit : 6;
  static_assert(kStages >= 2, "shared memory");
};
constexpr uint16_t kPairMask = 0x3;

template <int BN, int EPI, bool PAIR>
struct Smem {
  using C = Cfg<BN, EPI, PAIR>;
  uint16_t a[C::kStages][BM * BK];                  // 16 KB per stage
  uint16_t b[C::kStages][C::kBRows * BK];           // 16 or 32 KB per stage
  uint16_t out[C::kEpiWarps][C::kBufs][kStageChunk];   // 2 KB each
  float cd[C::kEpiWarps][2][C::kCdCols];            // colsum, colbias of the warp's columns
  uint64_t full[C::kStages];
  uint64_t empty[C::kStages];
  uint64_t res_full[C::kEpiWarps][C::kResTma ? C::kBufs : 1];
  uint64_t cd_full[C::kEpiWarps];
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
// With z = |x| / sqrt 2 and q = (1 - erf(z)) / 2, Phi = 1 - q for x >= 0 and
// q for x < 0, so in both cases GELU(x) = max(x, 0) - |x| q: no select on
// the sign.  The constants below fold in the 1/sqrt 2, the 1/2 and the sign
// of q.  Evaluated on two values at once with the paired fp32 instructions
// (fma/mul.rn.f32x2): the epilogue's ALU work is what limits this GEMM.
__device__ __forceinline__ void gelu_erf2(float& x0, float& x1) {
  const uint64_t P2 = f2_pack(0.3275911f * 0.70710678118654752f, 0.3275911f * 0.70710678118654752f);
  const uint64_t ONE2 = f2_pack(1.0f, 1.0f);
  const uint64_t A1 = f2_pack(-0.5f * 0.254829592f, -0.5f * 0.254829592f);
  const uint64_t A2 = f2_pack(-0.5f * -0.284496736f, -0.5f * -0.284496736f);
  const uint64_t A3 = f2_pack(-0.5f * 1.421413741f, -0.5f * 1.421413741f);
  const uint64_t A4 = f2_pack(-0.5f * -1.453152027f, -0.5f * -1.453152027f);
  const uint64_t A5 = f2_pack(-0.5f * 1.061405429f, -0.5f * 1.061405429f);
  const uint64_t C2 = f2_pack(-0.72134752044448170f, -0.72134752044448170f);   // -log2(e) / 2
  const uint64_t AX = f2_pack(fabsf(x0), fabsf(x1));
  float d0, d1;
  f2_unpack(f2_fma(P2, AX, ONE2), d0, d1);
  const uint64_t T = f2_pack(rcp_approx(d0), rcp_approx(d1));
  const uint64_t poly =
      f2_mul(T, f2_fma(T, f2_fma(T, f2_fma(T, f2_fma(T, A5, A4), A3), A2), A1));
  float e0, e1;
  f2_unpack(f2_mul(f2_mul(AX, AX), C2), e0, e1);
  const uint64_t neg_q = f2_mul(poly, f2_pack(ex2_approx(e0), ex2_approx(e1)));
  f2_unpack(f2_fma(AX, neg_q, f2_pack(fmaxf(x0, 0.0f), fmaxf(x1, 0.0f))), x0, x1);
}

// Adds 8 bf16 values (one 16-byte piece) to v[0..7] in fp32 pairs.
__device__ __forceinline__ void add_bf16x8(float* v, const uint4& piece) {
  const uint32_t* w = reinterpret_cast<const uint32_t*>(&piece);
#pragma unroll
  for (int e = 0; e < 4; ++e)
    f2_unpack(f2_add(f2_pack(v[2 * e], v[2 * e + 1]), f2_pack(bf16_lo(w[e]), bf16_hi(w[e]))),
              v[2 * e], v[2 * e + 1]);
}

// Bias (or the folded LayerNorm) and GELU of one 32-column chunk of one row,
// in fp32.
// For the folded LayerNorm, c and d of the chunk's 32 columns come from
// shared memory (cs, cb).
template <int EPI>
__device__ __forceinline__ void epilogue_math(const uint32_t (&r)[32], float (&v)[32],
                                              const LinearEpi& ep, int gcol, float neg_mean,
                                              float rstd, const float* cs, const float* cb) {
#pragma unroll
  for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
  if constexpr (EPI == kEpiLn || EPI == kEpiLnGelu) {
    // v = rstd (acc - mean c) + d
    const float4* cp = reinterpret_cast<const float4*>(cs);
    const float4* dp = reinterpret_cast<const float4*>(cb);
    const uint64_t NM = f2_pack(neg_mean, neg_mean), RS = f2_pack(rstd, rstd);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float4 c = cp[q], d = dp[q];
      f2_unpack(f2_fma(RS, f2_fma(NM, f2_pack(c.x, c.y), f2_pack(v[4 * q], v[4 * q + 1])),
                       f2_pack(d.x, d.y)),
                v[4 * q], v[4 * q + 1]);
      f2_unpack(f2_fma(RS, f2_fma(NM, f2_pack(c.z, c.w), f2_pack(v[4 * q + 2], v[4 * q + 3])),
                       f2_pack(d.z, d.w)),
                v[4 * q + 2], v[4 * q + 3]);
    }
  } else if (ep.bias != nullptr) {
    const uint4* bp = reinterpret_cast<const uint4*>(ep.bias + gcol);
#pragma unroll
    for (int q = 0; q < 4; ++q) add_bf16x8(v + 8 * q, __ldg(bp + q));
  }
  if constexpr (EPI == DORA_EPI_BIAS_GELU || EPI == kEpiLnGelu) {
#pragma unroll
    for (int e = 0; e < 32; e += 2) gelu_erf2(v[e], v[e + 1]);
  }
}

__device__ __forceinline__ void pack_row(const float (&v)[32], uint32_t (&o)[16]) {
#pragma unroll
  for (int e = 0; e < 16; ++e) o[e] = pack_bf16x2(v[2 * e], v[2 * e + 1]);
}

// Slice moments (mean, sum of squared deviations from it) of one 64-column
// slice of a rounded output row, from its two packed 32-column chunks.
__device__ __forceinline__ float2 slice_moments(const uint32_t (&lo)[16], const uint32_t (&hi)[16]) {
  float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    s4[e & 1] += bf16_lo(lo[e]) + bf16_hi(lo[e]);
    s4[2 + (e & 1)] += bf16_lo(hi[e]) + bf16_hi(hi[e]);
  }
  const float mean = ((s4[0] + s4[1]) + (s4[2] + s4[3])) * (1.0f / kSliceCols);
  float q4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 16; ++e) {
    const float a = bf16_lo(lo[e]) - mean, b = bf16_hi(lo[e]) - mean;
    const float c = bf16_lo(hi[e]) - mean, d = bf16_hi(hi[e]) - mean;
    q4[e & 1] += a * a + b * b;
    q4[2 + (e & 1)] += c * c + d * d;
  }
  return make_float2(mean, (q4[0] + q4[1]) + (q4[2] + q4[3]));
}

template <int BN, int EPI, bool PAIR>
__global__ void __launch_bounds__(Cfg<BN, EPI, PAIR>::kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ CUtensorMap tmY, const __grid_constant__ CUtensorMap tmR,
                uint16_t* __restrict__ Y, const LinearEpi ep, int m_cap,
                const int32_t* __restrict__ m_dev, int N, int K, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  pdl_trigger();
  if (smem_u32(smem_raw) & 1023u) {           // swizzled tiles need 1 KB alignment
    pdl_wait();
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem<BN, EPI, PAIR>& s = *reinterpret_cast<Smem<BN, EPI, PAIR>*>(smem_raw);
  using C = Cfg<BN, EPI, PAIR>;
  constexpr int kEpiWarps = C::kEpiWarps;
  constexpr int kBufs = C::kBufs;
  constexpr int kStages = C::kStages;
  constexpr bool kPair = C::kPair;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // Work is a list of tile pairs: pair p covers M-tiles 2*(p / n_tiles) and
  // 2*(p / n_tiles) + 1 of N-tile p % n_tiles (row pairs counted from the
  // last with ep.m_reverse); CTA `rank` of cluster c takes the M-tile
  // 2*(p / n_tiles) + rank of pairs c, c + clusters, ...
  // Both CTAs of a cluster walk the same pairs in lockstep.
  const int rank = static_cast<int>(cluster_ctarank());
  const int cid = blockIdx.x / kCluster;
  const int n_clusters = gridDim.x / kCluster;
  const int n_tiles = (N + BN - 1) / BN;
  const int kb_count = K / BK;
  constexpr uint32_t kTmemCols = 2 * BN;
  constexpr int kHalfB = BN / 2;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      // pair mode: the first CTA's MMAs release both CTAs' stages; otherwise
      // each CTA's own MMAs release its stage
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.acc_full[i], 1);
      // pair mode: the epilogues of both CTAs hand the accumulator back to the first
      mbar_init(&s.acc_empty[i], kPair ? 2 * kEpiWarps : kEpiWarps);
    }
    for (int w = 0; w < kEpiWarps; ++w) {
      for (int c = 0; c < (C::kResTma ? C::kBufs : 1); ++c) mbar_init(&s.res_full[w][c], 1);
      mbar_init(&s.cd_full[w], 1);
    }
    mbar_init(&s.drain, 1);
    s.abort_flag = 0;
    s.issued = 0;
    s.consumed = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmY);
    if (C::kResTma) tma_prefetch_desc(&tmR);
  }
  if (warp == 1) {
    if constexpr (kPair) tmem_alloc_pair(&s.tmem_base, kTmemCols);
    else tmem_alloc(&s.tmem_base, kTmemCols);
  }
  tc_fence_before();
  cluster_sync();              // peers' barriers are initialised before any remote signal
  tc_fence_after();
  // the set-up above overlaps the previous kernel; global memory waits for it
  pdl_wait();
  int M = m_cap;
  if (m_dev != nullptr) {
    const int v = *m_dev;
    M = v < 0 ? 0 : (v > m_cap ? m_cap : v);
  }
  const int m_pairs = (M + 2 * BM - 1) / (2 * BM);
  const int num_pairs = m_pairs * n_tiles;
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;
  // row pair of work item p; m_reverse walks them from the last, so that a
  // linear reading the output of one that walked forward starts on the rows
  // written last, still in L2
  auto mpair = [&](int p) {
    const int q0 = p / n_tiles;
    return ep.m_reverse ? m_pairs - 1 - q0 : q0;
  };

  if (warp == 0) {
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int pr = cid; ok && pr < num_pairs; pr += n_clusters) {
        const int mt = 2 * mpair(pr) + rank;
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
            if (rank == 0) mbar_arrive_expect_tx(&s.full[st], 2 * C::kStageBytes);
            tma_load_2d_pair(s.a[st], &tmA, &s.full[st], 0, kb * BK, mt * BM);
            tma_load_2d_pair(s.b[st], &tmB, &s.full[st], 0, kb * BK, nt * BN + rank * kHalfB);
          } else {
            // the X tile and both halves of the W tile (the map's box is BN/2 rows)
            mbar_arrive_expect_tx(&s.full[st], (BM + BN) * BK * 2);
            tma_load_2d(s.a[st], &tmA, &s.full[st], kb * BK, mt * BM);
            tma_load_2d(s.b[st], &tmB, &s.full[st], kb * BK, nt * BN);
            tma_load_2d(s.b[st] + kHalfB * BK, &tmB, &s.full[st], kb * BK, nt * BN + kHalfB);
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
          mma_commit(&s.empty[st]);                        // this CTA's stage free
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
    constexpr int kCols = C::kCols;                // columns per epilogue warp
    constexpr int kChunks = C::kChunks;
    constexpr int kBatch = C::kBatch;              // chunks per TMEM load
    const int ew = warp - 2;                      // epilogue warp index
    const int q = warp & 3;                       // TMEM lanes this warp may read
    const int slot = ew >> 2;                     // which column slice
    const uint32_t lane_sel = static_cast<uint32_t>(q * 32) << 16;
    int buf = 0;                                  // staging buffer to write next
    uint32_t res_pend = 0;                        // staging buffers with a residual load in flight
    uint32_t res_par = 0;                         // their next completion parity
    // Residual chunk `c` of the warp's 32 rows from row0, column col0 on, into
    // staging buffer c % kBufs (whose previous store must have read it).
    auto load_residual = [&](int c, int row0, int col0) {
      const int b = c % kBufs;
      if (lane == 0) {
        mbar_arrive_expect_tx(&s.res_full[ew][b], kStageChunk * 2);
        tma_load_2d(s.out[ew][b], &tmR, &s.res_full[ew][b], col0 + c * 32, row0);
      }
      res_pend |= 1u << b;
    };
    // Residual of the warp's whole 32-row chunks of tile pair `p` (the first
    // kBufs chunks), once the stores of the previous tile have read the buffers.
    auto prefetch_residual = [&](int p) {
      const int row0 = (2 * mpair(p) + rank) * BM + q * 32;
      if (row0 + 32 > M) return;
      const int col0 = (p % n_tiles) * BN + slot * kCols;
      if (lane == 0) bulk_wait_group_read0();
      __syncwarp();
#pragma unroll
      for (int c = 0; c < kBufs; ++c) {
        if (col0 + c * 32 >= N) break;
        load_residual(c, row0, col0);
      }
    };
    // Slice moments of the rounded output row: the first chunk of a 64-column
    // slice is kept packed until the second is done.
    uint32_t first_half[16];
    auto emit_moments = [&](const uint32_t(&o)[16], int row_, int gcol) {
      if ((gcol & 32) == 0) {
#pragma unroll
        for (int e = 0; e < 16; ++e) first_half[e] = o[e];
      } else {
        reinterpret_cast<float2*>(ep.stats_out)[static_cast<size_t>(gcol >> 6) * m_cap + row_] =
            slice_moments(first_half, o);
      }
    };
    // Folded LayerNorm: c and d of the warp's columns of tile pair `p`, one
    // bulk copy each into the warp's buffer, after the warp's reads of the
    // previous tile's values.
    bool cd_pend = false;
    uint32_t cd_par = 0;
    auto prefetch_cd = [&](int p) {
      const int col0 = (p % n_tiles) * BN + slot * kCols;
      const int cols = N - col0 < kCols ? N - col0 : kCols;
      if (cols <= 0) return;
      __syncwarp();                               // every lane's reads of the buffer are done
      if (lane == 0) {
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(&s.cd_full[ew], 2u * 4u * static_cast<uint32_t>(cols));
        bulk_load(s.cd[ew][0], ep.colsum + col0, 4u * cols, &s.cd_full[ew]);
        bulk_load(s.cd[ew][1], ep.colbias + col0, 4u * cols, &s.cd_full[ew]);
      }
      cd_pend = true;
    };
    // Folded LayerNorm: (mean, var) of this lane's row, loaded a tile ahead
    // (a warp's 32 rows are one 256-byte load).
    float2 mv = make_float2(0.f, 0.f);
    auto load_mv = [&](int p) {
      const int row_p = (2 * mpair(p) + rank) * BM + q * 32 + lane;
      if (row_p < M) mv = __ldg(reinterpret_cast<const float2*>(ep.stats_in) + row_p);
    };
    if constexpr (C::kLn)
      if (cid < num_pairs) {
        prefetch_cd(cid);
        load_mv(cid);
      }
    if constexpr (C::kResTma)
      if (cid < num_pairs) prefetch_residual(cid);
    int ti = 0;
    bool ok = true;
    for (int pr = cid; ok && pr < num_pairs; pr += n_clusters, ++ti) {
      const int acc = ti & 1;
      const uint32_t aph = (ti >> 1) & 1;
      const int mt = 2 * mpair(pr) + rank;
      const int nt = pr % n_tiles;
      const int row0 = mt * BM + q * 32;          // first row of this warp
      const int row = row0 + lane;
      const bool whole = row0 + 32 <= M;          // all 32 rows live: TMA store
      float neg_mean = 0.f, rstd = 0.f;           // folded LayerNorm of this row
      if constexpr (C::kLn) {
        neg_mean = -mv.x;
        rstd = rsqrtf(mv.y + ep.eps);
        if (pr + n_clusters < num_pairs) load_mv(pr + n_clusters);
      }
      if (!mbar_wait_warp(&s.acc_full[acc], aph, abort)) break;
      tc_fence_after();
      if constexpr (C::kLn) {
        if (cd_pend) {
          if (!mbar_wait_warp(&s.cd_full[ew], cd_par, abort)) break;
          cd_par ^= 1u;
          cd_pend = false;
        }
      }
#pragma unroll 1
      for (int cb = 0; cb < kChunks; cb += kBatch) {
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
          epilogue_math<EPI>(r[c], v, ep, gcol, neg_mean, rstd,
                             &s.cd[ew][0][((cb + c) * 32) % C::kCdCols],
                             &s.cd[ew][1][((cb + c) * 32) % C::kCdCols]);
          if (whole) {
            // row `lane` of the 32x32 chunk, 64-byte swizzle: 16-byte piece j
            // of row l sits at piece j ^ ((l >> 1) & 3).
            uint16_t* stage;
            if constexpr (C::kResTma) {
              const int rb = (cb + c) % kBufs;
              stage = s.out[ew][rb];
              if (!mbar_wait_warp(&s.res_full[ew][rb], (res_par >> rb) & 1u, abort)) {
                ok = false;
                break;
              }
              res_par ^= 1u << rb;
              res_pend &= ~(1u << rb);
            } else {
              // the store issued kBufs chunks ago from this buffer must have read it
              stage = s.out[ew][buf];
              if (lane == 0) {
                if constexpr (kBufs == 2) bulk_wait_group_read1();
                else bulk_wait_group_read0();
              }
              __syncwarp();
              buf = (buf + 1) % kBufs;
            }
            uint8_t* rowp = reinterpret_cast<uint8_t*>(stage) + lane * 64;
            if constexpr (C::kResTma) {
#pragma unroll
              for (int j = 0; j < 4; ++j)
                add_bf16x8(v + 8 * j,
                           *reinterpret_cast<const uint4*>(rowp + ((j ^ ((lane >> 1) & 3)) << 4)));
            }
            pack_row(v, o);
            if constexpr (C::kResTma)
              if (ep.stats_out != nullptr) emit_moments(o, row, gcol);
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
            if constexpr (C::kResTma && kBufs < kChunks) {
              // the chunk kBufs on goes into this buffer once the store has read it
              const int nc = cb + c + kBufs;
              const int col0 = nt * BN + slot * kCols;
              if (nc < kChunks && col0 + nc * 32 < N) {
                if (lane == 0) bulk_wait_group_read0();
                __syncwarp();
                load_residual(nc, row0, col0);
              }
            }
          } else if (row < M) {
            if constexpr (C::kResTma) {
              const uint4* rp =
                  reinterpret_cast<const uint4*>(ep.residual + static_cast<size_t>(row) * N + gcol);
#pragma unroll
              for (int j = 0; j < 4; ++j) add_bf16x8(v + 8 * j, __ldg(rp + j));
            }
            pack_row(v, o);
            if constexpr (C::kResTma)
              if (ep.stats_out != nullptr) emit_moments(o, row, gcol);
            uint4* yp = reinterpret_cast<uint4*>(Y + static_cast<size_t>(row) * N + gcol);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              yp[j] = make_uint4(o[4 * j], o[4 * j + 1], o[4 * j + 2], o[4 * j + 3]);
          }
        }
        if (!ok) break;
      }
      if constexpr (C::kResTma)
        if (ok && pr + n_clusters < num_pairs) prefetch_residual(pr + n_clusters);
      if constexpr (C::kLn)
        if (ok && pr + n_clusters < num_pairs) prefetch_cd(pr + n_clusters);
    }
    if (lane == 0) {
      bulk_wait_group0();                         // stores done before the CTA exits
      // after an abort: residual loads issued but never consumed land first
      for (int c = 0; c < kBufs; ++c)
        if (res_pend & (1u << c))
          mbar_wait_limited(&s.res_full[ew][c], (res_par >> c) & 1u, 100ull * 1000 * 1000);
      if (cd_pend) mbar_wait_limited(&s.cd_full[ew], cd_par, 100ull * 1000 * 1000);
    }
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
                                 const CUtensorMap& ty, const CUtensorMap& tr, uint16_t* y,
                                 const LinearEpi& ep, int m_cap, const int32_t* m_dev, int n,
                                 int k, int32_t* status, cudaStream_t stream) {
  static_assert(sizeof(Smem<BN, EPI, PAIR>) <= kSmemLimit, "shared memory");
  const size_t smem = sizeof(Smem<BN, EPI, PAIR>);
  auto kern = gemm_kernel<BN, EPI, PAIR>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.blockDim = dim3(Cfg<BN, EPI, PAIR>::kThreads);
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
  cfg.numAttrs = pdl_enabled() ? 2 : 1;          // dependent launch (the kernel waits)
  return cudaLaunchKernelEx(&cfg, kern, ta, tb, ty, tr, y, ep, m_cap, m_dev, n, k, status);
}

// BN = 256 tiles run in pair mode.
template <int BN>
static cudaError_t launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& ty,
                             const CUtensorMap& tr, uint16_t* y, const LinearEpi& ep, int epi,
                             int m_cap, const int32_t* m_dev, int n, int k, int32_t* status,
                             cudaStream_t stream) {
  constexpr bool kPair = BN == 256;
  switch (epi) {
    case DORA_EPI_BIAS_GELU:
      return launch_bn_epi<BN, DORA_EPI_BIAS_GELU, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev, n, k,
                                                          status, stream);
    case DORA_EPI_BIAS_RESIDUAL:
      return launch_bn_epi<BN, DORA_EPI_BIAS_RESIDUAL, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev,
                                                              n, k, status, stream);
    case kEpiResidualLongK:
      return launch_bn_epi<BN, kEpiResidualLongK, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev, n,
                                                         k, status, stream);
    case kEpiLn:
      return launch_bn_epi<BN, kEpiLn, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev, n, k, status,
                                              stream);
    case kEpiLnGelu:
      return launch_bn_epi<BN, kEpiLnGelu, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev, n, k, status,
                                                  stream);
    default:
      return launch_bn_epi<BN, DORA_EPI_BIAS, kPair>(ta, tb, ty, tr, y, ep, m_cap, m_dev, n, k,
                                                     status, stream);
  }
}

}  // namespace gemm

cudaError_t launch_linear(const uint16_t* x, int32_t m_cap, const int32_t* m_dev, int32_t k,
                          const uint16_t* w, int32_t n, int32_t epilogue, const LinearEpi& ep,
                          uint16_t* y, int32_t* status, cudaStream_t stream, int32_t lda) {
  if (m_cap == 0) return cudaSuccess;
  const int bn = (n % 256 == 0) ? 256 : 128;
  CUtensorMap ta, tb, ty, tr;
  if (lda != 0 && (lda < k || lda % 8 != 0)) return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&ta, x, static_cast<uint64_t>(k), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(lda != 0 ? lda : k) * 2, gemm::BK, gemm::BM) != 0)
    return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&tb, w, static_cast<uint64_t>(k), static_cast<uint64_t>(n),
                          static_cast<uint64_t>(k) * 2, gemm::BK, static_cast<uint32_t>(bn / 2)) != 0)
    return cudaErrorInvalidValue;
  if (encode_tmap_2d_bf16(&ty, y, static_cast<uint64_t>(n), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(n) * 2, 32, 32, 64) != 0)
    return cudaErrorInvalidValue;
  // the residual [m_cap, n] in the output's 32 x 32 chunks (unused otherwise)
  tr = ty;
  if (epilogue == DORA_EPI_BIAS_RESIDUAL &&
      encode_tmap_2d_bf16(&tr, ep.residual, static_cast<uint64_t>(n), static_cast<uint64_t>(m_cap),
                          static_cast<uint64_t>(n) * 2, 32, 32, 64) != 0)
    return cudaErrorInvalidValue;
  if (bn == 256) {
    const int epi = (epilogue == DORA_EPI_BIAS_RESIDUAL && k >= gemm::kLongK)
                        ? gemm::kEpiResidualLongK
                        : epilogue;
    return gemm::launch_bn<256>(ta, tb, ty, tr, y, ep, epi, m_cap, m_dev, n, k, status, stream);
  }
  return gemm::launch_bn<128>(ta, tb, ty, tr, y, ep, epilogue, m_cap, m_dev, n, k, status, stream);
}

}  // namespace dora
