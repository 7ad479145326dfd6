// Packed variable-length multi-head self-attention on tcgen05 tensor cores,
// the kernel for images longer than 256 tokens (launch_varlen_attn below picks
// it when max_seqlen > 256; shorter batches run attn_exchange_tcgen05.cu).
// For image i (rows [cu[i], cu[i+1]) of the packed buffer) and head h:
//     O = softmax(Q K^T * scale) V
// with no attention across images and no padding (Sec. 3.5 "Inference").
//
// Work unit = (image, head, 128-row query tile); a unit walks its keys in
// chunks of 128 ("steps").  One persistent CTA per SM owns a contiguous range
// of image-heads, split by estimated cost, and runs its steps through a
// pipeline in which no role waits on the softmax's own previous work:
//   warp 0       walks the CTA's units, loads Q and K/V chunks by TMA (the two
//                query tiles of an image of up to 256 tokens share the chunks),
//                and publishes a descriptor per step and per unit.  No other
//                role keeps unit bookkeeping.
//   warps 1-3    MMA issuers (one thread each): warp 1 issues S(j) = Q K^T
//                (M=128, N=keys rounded to 16, K=64) into S/P buffer j mod 2,
//                once both PVs of step j-2 are done with that buffer; warp
//                2 + h issues O_h (+)= P_h(j) V_h for key half h (keys
//                64h .. 64h+63 of the chunk).  A tcgen05.mma takes about 120
//                cycles to issue, so the two halves' PVs go out in parallel.
//   warps 4-11   softmax, two threads per query row (TMEM lane): warps 4-7
//                take key half 0 of every step, warps 8-11 half 1, 64 S
//                columns each, held in registers.  Each half keeps its own
//                running reference maximum, row sum and O accumulator for the
//                unit, so the two threads of a row never exchange anything.
//                A half's reference maximum is set on the unit's first chunk
//                and raised only when a later chunk exceeds it by more than
//                2^8 (then its O is rescaled in TMEM); otherwise P stays below
//                2^8 in the old frame, which bf16 and fp32 hold exactly.  A
//                half writes its P (bf16) over the first 32 of its own 64 S
//                columns, and zeroes the V rows of the chunk's last 16-key
//                group that lie past the image when they fall in its half.
//   warps 12-15  epilogue: once a unit's last PVs are done, the two halves'
//                partial results are merged, O = (a_0 O_0 + a_1 O_1) /
//                (a_0 l_0 + a_1 l_1) with a_h = 2^(m_h - max(m_0, m_1)), and
//                stored through shared memory four whole rows per store.
// TMEM (512 columns): S/P buffers 0-127 and 128-255; O_0 and O_1 of units of
// even parity in 256-319 and 320-383, of odd parity in 384-447 and 448-511,
// so a unit's PVs never wait for the previous unit's epilogue.  Rows past the image are computed but never stored;
// keys past it are masked, and V rows past it are zeroed so stale data cannot
// leak through 0 * NaN.
#include "attn_common.cuh"

namespace dora {
namespace attn {
namespace split {

constexpr int kSpBufs = 2;      // S/P buffers, used by steps in turn
__device__ __forceinline__ uint32_t tmem_sp(int b) { return 128u * static_cast<uint32_t>(b); }
// O of key half h for units of parity up (two units in flight)
__device__ __forceinline__ uint32_t tmem_o(int h, int up) {
  return 128u * kSpBufs + 128u * static_cast<uint32_t>(up) + 64u * static_cast<uint32_t>(h);
}
static_assert(128 * kSpBufs + 4 * 64 <= 512, "TMEM columns");

// Step descriptor (one 32-bit word).
constexpr uint32_t kDStage = 0x3u;        // K/V stage
constexpr uint32_t kDKvPar = 1u << 2;     // phase parity of that stage's load
constexpr uint32_t kDLast0 = 1u << 3;     // key half 0's last chunk of this unit
constexpr uint32_t kDLast1 = 1u << 4;     // key half 1's last chunk of this unit
constexpr uint32_t kDUPar = 1u << 5;      // unit parity: Q buffer
constexpr uint32_t kDQPar = 1u << 6;      // phase parity of the unit's Q load
constexpr uint32_t kDRelease = 1u << 7;   // the K/V stage is free after this step's PV
constexpr uint32_t kDUFirst = 1u << 8;    // first chunk of the unit (S waits for Q)
constexpr uint32_t kDULast = 1u << 25;    // last chunk of the unit (S frees Q)
constexpr uint32_t kDEnd = 1u << 31;      // no more steps
__device__ __forceinline__ int d_kc(uint32_t d) { return static_cast<int>((d >> 9) & 0xFFu); }
__device__ __forceinline__ int d_rows(uint32_t d) { return static_cast<int>((d >> 17) & 0xFFu); }
__device__ __forceinline__ int d_slot(uint32_t d) { return static_cast<int>((d >> 26) & 0x3u); }

struct Smem {
  uint16_t q[2][BQ * HD];       // 2 x 16 KB, by unit parity
  uint16_t k[kStages][KC * HD]; // 4 x 16 KB
  uint16_t v[kStages][KC * HD]; // 4 x 16 KB
  uint4 ostage[4][32 * 8];      // per epilogue warp: 32 output rows of 128 bytes
  float2 lm[kUnitRing][2][BQ];  // (row sum, reference maximum) of each half, by unit slot
  uint64_t q_full[2];
  uint64_t q_empty[2];
  uint64_t kv_full[kStages];
  uint64_t kv_empty[kStages];
  uint64_t s_full[kSpBufs];     // S of a step in S/P buffer b
  uint64_t p_full[kSpBufs][2];  // half h's P written over its S (one arrival per warp)
  uint64_t p_free[kSpBufs];     // both PVs of buffer b done
  uint64_t o_done[2][2];        // last PV of a unit into O_h (unit parity) done
  uint64_t o_free[2][2];        // O_h (unit parity) read out (one arrival per epilogue warp)
  uint64_t l_full[kUnitRing][2];  // a half's row sums of a unit published
  uint64_t sd_full[kDescRing];  // step descriptor published
  uint64_t sd_empty[kDescRing]; // ... read by the three issuers and the eight softmax warps
  uint64_t ud_full[kUnitRing];  // unit descriptor published
  uint64_t ud_empty[kUnitRing]; // ... and the unit finished by the four epilogue warps
  uint64_t drain[3];
  uint32_t sdesc[kDescRing];
  uint32_t urow[kUnitRing];     // first output row of the unit
  uint32_t uhead[kUnitRing];    // head | rows << 16 | key halves used << 24
  uint32_t tmem_base;
  int abort_flag;
  int ih_begin, ih_end;
  int q_issued, kv_issued;
};

__global__ void __launch_bounds__(kThreads, 1)
    varlen_attn_kernel(const __grid_constant__ QkvMaps mp, const int32_t* __restrict__ cu,
                       int batch, int max_seqlen, int t_cap, int heads, float scale_log2,
                       uint16_t* __restrict__ out, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  pdl_trigger();
  if (smem_u32(smem_raw) & 1023u) {
    pdl_wait();
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem& s = *reinterpret_cast<Smem*>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int dim = heads * HD;

  if (threadIdx.x == 64) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s.q_full[b], 1);
      mbar_init(&s.q_empty[b], 1);
      for (int h = 0; h < 2; ++h) {
        mbar_init(&s.o_done[h][b], 1);
        mbar_init(&s.o_free[h][b], 4);
      }
    }
    for (int b = 0; b < kSpBufs; ++b) {
      mbar_init(&s.s_full[b], 1);
      mbar_init(&s.p_full[b][0], 4);
      mbar_init(&s.p_full[b][1], 4);
      mbar_init(&s.p_free[b], 2);
    }
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&s.l_full[i][0], 4);
      mbar_init(&s.l_full[i][1], 4);
    }
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.kv_full[i], 1);
      mbar_init(&s.kv_empty[i], 2);                 // released by both PV issuers
    }
    for (int i = 0; i < kDescRing; ++i) {
      mbar_init(&s.sd_full[i], 1);
      mbar_init(&s.sd_empty[i], 11);
    }
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&s.ud_full[i], 1);
      mbar_init(&s.ud_empty[i], 4);
    }
    for (int i = 0; i < 3; ++i) mbar_init(&s.drain[i], 1);
    s.abort_flag = 0;
    s.q_issued = s.kv_issued = 0;
    fence_barrier_init();
    tma_prefetch_desc(&mp.m128);
    tma_prefetch_desc(&mp.m64);
    tma_prefetch_desc(&mp.m32);
    tma_prefetch_desc(&mp.m16);
  }
  if (warp == 1) tmem_alloc(&s.tmem_base, kTmemCols);
  // the set-up above overlaps the previous kernel; global memory waits for it
  pdl_wait();
  if (warp == 0) {
    long long b, e;
    find_range(cu, batch, heads, t_cap, max_seqlen, status, b, e);
    if (lane == 0) {
      s.ih_begin = static_cast<int>(b);
      s.ih_end = static_cast<int>(e);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;
  const int ih_b = s.ih_begin, ih_e = s.ih_end;

  if (warp == 0) {
    // ---------------- scheduler + TMA producer ----------------
    if (lane == 0) {
      Walker wk;
      wk.start(cu, heads, t_cap, ih_b, ih_e);
      int u = 0, loads = 0, dn = 0;
      int prev_stage[2] = {0, 0}, prev_par[2] = {0, 0};
      bool reuse_this = false;      // this unit reads the previous unit's K/V chunks
      bool ok = true;
      auto desc = [&](uint32_t d) -> bool {
        const int i = dn % kDescRing;
        if (!mbar_wait_sleep(&s.sd_empty[i], ((dn / kDescRing) & 1) ^ 1, abort, kSleepNs))
          return false;
        s.sdesc[i] = d;
        mbar_arrive(&s.sd_full[i]);
        ++dn;
        return true;
      };
      while (ok && !wk.done()) {
        const int n = wk.n, nch = (n + KC - 1) / KC;
        const int rows = min(BQ, n - wk.qt * BQ);
        Walker nx = wk;
        nx.next();
        // the next unit (the image-head's other query tile) reads the same chunks
        const bool reuse_next = !nx.done() && nx.ih == wk.ih && nch <= 2;
        // key half 1 has keys in a chunk of more than 64 keys: every chunk but
        // a short last one; none when the image has 64 tokens or fewer
        const int kc_last = n - (nch - 1) * KC;
        const int last1 = kc_last > 64 ? nch - 1 : nch - 2;
        const uint32_t gmask = n > 64 ? 3u : 1u;
        const int slot = u % kUnitRing;
        {
          // the slot is free once the epilogue has finished unit u - kUnitRing
          if (!mbar_wait_sleep(&s.ud_empty[slot], ((u / kUnitRing) & 1) ^ 1, abort, kSleepNs))
            break;
          s.urow[slot] = static_cast<uint32_t>(wk.lo + wk.qt * BQ);
          s.uhead[slot] = static_cast<uint32_t>(wk.head) | (static_cast<uint32_t>(rows) << 16) |
                          (gmask << 24);
          mbar_arrive(&s.ud_full[slot]);
        }
        const int qb = u & 1;
        if (!mbar_wait_sleep(&s.q_empty[qb], ((u >> 1) & 1) ^ 1, abort, kSleepNs)) break;
        const int rows16 = (rows + 15) & ~15;
        mbar_arrive_expect_tx(&s.q_full[qb], static_cast<uint32_t>(rows16 * HD * 2));
        load_rows(mp, s.q[qb], &s.q_full[qb], wk.head * HD, wk.lo + wk.qt * BQ, rows16);
        s.q_issued = u + 1;
        int cur_stage[2] = {0, 0}, cur_par[2] = {0, 0};
        for (int c = 0; ok && c < nch; ++c) {
          int stg, par;
          if (reuse_this) {
            stg = prev_stage[c];
            par = prev_par[c];
          } else {
            stg = loads % kStages;
            par = (loads / kStages) & 1;
            if (!mbar_wait_sleep(&s.kv_empty[stg], par ^ 1, abort, kSleepNs)) {
              ok = false;
              break;
            }
#ifdef DORA_TEST_WITHHOLD_KV_LOAD
            // timeout-path test library only: CTA 0 never issues its first K/V
            // load nor its expected bytes, so the S issuer's bounded wait on
            // that stage runs out with no copy in flight
            const bool withhold = blockIdx.x == 0 && loads == 0;
#else
            constexpr bool withhold = false;
#endif
            if (!withhold) {
              const int kc16 = (min(KC, n - c * KC) + 15) & ~15;
              mbar_arrive_expect_tx(&s.kv_full[stg], static_cast<uint32_t>(2 * kc16 * HD * 2));
              const int row = wk.lo + c * KC;
              load_rows(mp, s.k[stg], &s.kv_full[stg], dim + wk.head * HD, row, kc16);
              load_rows(mp, s.v[stg], &s.kv_full[stg], 2 * dim + wk.head * HD, row, kc16);
            }
            ++loads;
            s.kv_issued = loads;
          }
          if (c < 2) {
            cur_stage[c] = stg;
            cur_par[c] = par;
          }
          const uint32_t d =
              static_cast<uint32_t>(stg) | (par ? kDKvPar : 0u) | (c == nch - 1 ? kDLast0 : 0u) |
              (c == last1 ? kDLast1 : 0u) | ((u & 1) ? kDUPar : 0u) |
              (((u >> 1) & 1) ? kDQPar : 0u) | (reuse_next ? 0u : kDRelease) |
              (c == 0 ? kDUFirst : 0u) | (c == nch - 1 ? kDULast : 0u) |
              (static_cast<uint32_t>(min(KC, n - c * KC)) << 9) |
              (static_cast<uint32_t>(rows) << 17) | (static_cast<uint32_t>(slot) << 26);
          ok = desc(d);
        }
        prev_stage[0] = cur_stage[0];
        prev_stage[1] = cur_stage[1];
        prev_par[0] = cur_par[0];
        prev_par[1] = cur_par[1];
        reuse_this = reuse_next;
        ++u;
        wk = nx;
      }
      if (ok && desc(kDEnd)) {
        const int i = u % kUnitRing;      // no more units
        if (mbar_wait_sleep(&s.ud_empty[i], ((u / kUnitRing) & 1) ^ 1, abort, kSleepNs)) {
          s.uhead[i] = 0xFFFFFFFFu;
          mbar_arrive(&s.ud_full[i]);
        }
      }
    }
  } else if (warp >= 1 && warp <= 3) {
    // ---------------- MMA issuers: warp 1 issues S, warp 2 + h the PV of key half h ----------------
    // Each reads every step descriptor.  The only order between them is
    // explicit: S(j + kSpBufs) waits until both PVs of step j have read S/P
    // buffer j mod kSpBufs.
    if (lane == 0) {
      int uses[2] = {0, 0};        // units started in O_h, by unit parity (PV issuer of half h)
      for (int j = 0;; ++j) {
        const int i = j % kDescRing;
        if (!mbar_wait_sleep(&s.sd_full[i], (j / kDescRing) & 1, abort, kSleepNs)) break;
        const uint32_t d = s.sdesc[i];
        mbar_arrive(&s.sd_empty[i]);
        if (d & kDEnd) break;
        const int stg = static_cast<int>(d & kDStage);
        const int up = (d & kDUPar) ? 1 : 0;
        const int b = j % kSpBufs;
        const uint32_t bph = static_cast<uint32_t>(j / kSpBufs) & 1u;   // buffer use parity
        if (warp == 1) {
          // S(j) = Q K^T into S/P buffer b
          if ((d & kDUFirst) &&
              !mbar_wait_sleep(&s.q_full[up], (d & kDQPar) ? 1u : 0u, abort, kSleepNs))
            break;
          if (!mbar_wait_sleep(&s.kv_full[stg], (d & kDKvPar) ? 1u : 0u, abort, kSleepNs)) break;
          // the buffer's previous P has been read by its PV (step j - kSpBufs)
          if (j >= kSpBufs && !mbar_wait_sleep(&s.p_free[b], bph ^ 1u, abort, kSleepNs)) break;
          tc_fence_after();
          const uint64_t qd = sdesc_sw128(smem_u32(s.q[up]), 16, 1024);
          const uint64_t kd = sdesc_sw128(smem_u32(s.k[stg]), 16, 1024);
          const uint32_t id_s = idesc_bf16(BQ, (d_kc(d) + 15) & ~15, false);
          const uint32_t dt = tmem + tmem_sp(b);
          mma_bf16_ss(dt, qd, kd, id_s, 0u);
          mma_bf16_ss(dt, qd + 2, kd + 2, id_s, 1u);
          mma_bf16_ss(dt, qd + 4, kd + 4, id_s, 1u);
          mma_bf16_ss(dt, qd + 6, kd + 6, id_s, 1u);
          mma_commit(&s.s_full[b]);
          if (d & kDULast) mma_commit(&s.q_empty[up]);
        } else {
          // O_h (+)= P_h(j) V_h over the step's keys 64h .. 64h + 63
          constexpr uint32_t id_o = idesc_bf16(BQ, HD, true);
          const int h = warp - 2;
          const int kh = min(max(d_kc(d) - 64 * h, 0), 64);   // keys of this half
          const bool first = (d & kDUFirst) != 0 && kh > 0;
          // O_h held the half's part of an earlier unit until the epilogue read it
          if (first) {
            if (uses[up] > 0 &&
                !mbar_wait_sleep(&s.o_free[h][up], static_cast<uint32_t>(uses[up] - 1) & 1u,
                                 abort, kSleepNs))
              break;
            ++uses[up];
          }
          if (!mbar_wait_sleep(&s.p_full[b][h], bph, abort, kSleepNs)) break;
          tc_fence_after();
          if (kh > 0) {
            const int nk = (kh + 15) >> 4;
            // V rows 64h .. : 16 keys are 2048 bytes of the 128-byte-swizzled tile
            const uint64_t vd = sdesc_sw128(smem_u32(s.v[stg] + 64 * h * HD), 1024, 1024);
            const uint32_t dt = tmem + tmem_o(h, up), at = tmem + tmem_sp(b) + 64u * h;
            mma_bf16_ts(dt, at, vd, id_o, first ? 0u : 1u);
#pragma unroll
            for (int kk = 1; kk < 4; ++kk)       // 16 keys: 8 P columns
              if (kk < nk) mma_bf16_ts(dt, at + 8u * kk, vd + 128u * kk, id_o, 1u);
          }
          mma_commit(&s.p_free[b]);
          if (d & (h == 0 ? kDLast0 : kDLast1)) mma_commit(&s.o_done[h][up]);
          if (d & kDRelease) mma_commit(&s.kv_empty[stg]);
        }
      }
      mma_commit(&s.drain[warp - 1]);
      mbar_wait_limited(&s.drain[warp - 1], 0, kWaitLimitNs);
    }
  } else if (warp >= kSoftWarp0 && warp < kEpiWarp0) {
    // ---------------- softmax: key half h of every step, two threads per row ----------------
    const int h = (warp - kSoftWarp0) >> 2;
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;                   // query row of the tile (TMEM lane)
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    float m_ref = 0.f, l = 0.f;                          // the half's frame and row sum
    auto step = [&](int j, uint32_t d) -> bool {
      const int kc = d_kc(d), kc16 = (kc + 15) & ~15;
      const int kh = min(max(kc - 64 * h, 0), 64);       // keys in this half
      const bool live = quarter * 32 < d_rows(d) && kh > 0;   // warp-uniform
      const int b = j % kSpBufs;
      const uint32_t bph = static_cast<uint32_t>(j / kSpBufs) & 1u;   // buffer use parity
      const uint32_t tsp = tmem + lane_sel + tmem_sp(b) + 64u * h;   // this half's S columns
      if (!mbar_wait_warp_sleep(&s.s_full[b], bph, abort, kSleepNs)) return false;
      tc_fence_after();
      // S is done, so the K/V load landed: zero V rows [kc, kc16) (whole 128-byte
      // rows; they lie in one half, whose PV reads them)
      if (kc < kc16 && (kc >> 6) == h) {
        if (r < (kc16 - kc) * 8)
          reinterpret_cast<uint4*>(s.v[d & kDStage])[kc * 8 + r] = make_uint4(0u, 0u, 0u, 0u);
        fence_proxy_async_smem();
      }
      if (live) {
        uint32_t s0[32], s1[32];
        tmem_ld32(tsp, s0);
        tmem_ld32(tsp + 32u, s1);
        tmem_ld_wait();
        mask_tail(s0, kh);
        mask_tail(s1, kh - 32);
        const float mc = max32(s1, max32(s0, -INFINITY)) * scale_log2;
        // reference maximum: set on the unit's first chunk, raised past 2^8
        bool rescale = false;
        float alpha = 1.f;
        if (d & kDUFirst) {
          m_ref = mc;
          l = 0.f;
        } else {
          const bool need = mc > m_ref + kRescaleLog2;
          rescale = __any_sync(0xffffffffu, need) != 0;
          if (need) {
            alpha = ex2_approx(m_ref - mc);
            l *= alpha;
            m_ref = mc;
          }
        }
        // P over the first 32 of the half's own S columns, already read
        exp32_pack(s0, scale_log2, -m_ref, l);
        tmem_st16(tsp, lo16(s0));
        if (kh > 32) {
          exp32_pack(s1, scale_log2, -m_ref, l);
          tmem_st16(tsp + 16u, lo16(s1));
        }
        if (rescale) {
          // O_h holds the unit's earlier chunks once their PVs (step j - 1) are
          // done: bring the row to the raised reference before this chunk's PV
          const int pb = (j - 1) % kSpBufs;
          if (!mbar_wait_warp_sleep(&s.p_free[pb], static_cast<uint32_t>((j - 1) / kSpBufs) & 1u,
                                    abort, kSleepNs))
            return false;
          tc_fence_after();
#pragma unroll 1
          for (int q = 0; q < 2; ++q) {
            const uint32_t to = tmem + lane_sel + tmem_o(h, (d & kDUPar) ? 1 : 0) + 32u * q;
            uint32_t o[32];
            tmem_ld32(to, o);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st16(to, lo16(o));
            tmem_st16(to + 16u, *reinterpret_cast<const uint32_t(*)[16]>(&o[16]));
          }
        }
      }
      tmem_st_wait();
      if (d & (h == 0 ? kDLast0 : kDLast1)) {
        s.lm[d_slot(d)][h][r] = make_float2(l, m_ref);
        warp_arrive(&s.l_full[d_slot(d)][h]);
      }
      warp_arrive(&s.p_full[b][h]);
      return true;
    };
    for (int j = 0;; ++j) {
      const int i = j % kDescRing;
      if (!mbar_wait_warp_sleep(&s.sd_full[i], (j / kDescRing) & 1, abort, kSleepNs)) break;
      const uint32_t d = s.sdesc[i];
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.sd_empty[i]);
      if ((d & kDEnd) || !step(j, d)) break;
    }
  } else if (warp >= kEpiWarp0) {
    // ---------------- epilogue: merge the halves, O / row sum, four rows per store ----------------
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    uint4* const stage = s.ostage[warp - kEpiWarp0];
    uint32_t opar = 0u;            // o_done phase parity, bit 2 * h + unit parity
    uint32_t lpar = 0u;            // l_full phase parity, bit 2 * slot + h
    for (int u = 0;; ++u) {
      const int i = u % kUnitRing;
      // one descriptor per unit, then an end marker
      if (!mbar_wait_warp_sleep(&s.ud_full[i], (u / kUnitRing) & 1, abort, kSleepNs)) break;
      const uint32_t row0 = s.urow[i], hd = s.uhead[i];
      __syncwarp();
      if (hd == 0xFFFFFFFFu) break;
      const int rows = static_cast<int>((hd >> 16) & 0xFFu), head = static_cast<int>(hd & 0xFFFFu);
      const uint32_t gm = (hd >> 24) & 3u;
      bool ok = true;
      for (int g = 0; g < 2 && ok; ++g) {
        if (!(gm & (1u << g))) continue;
        ok = mbar_wait_warp_sleep(&s.o_done[g][u & 1], (opar >> (2 * g + (u & 1))) & 1u, abort,
                                  kSleepNs) &&
             mbar_wait_warp_sleep(&s.l_full[i][g], (lpar >> (2 * i + g)) & 1u, abort, kSleepNs);
        opar ^= 1u << (2 * g + (u & 1));
        lpar ^= 1u << (2 * i + g);
      }
      if (!ok) break;
      tc_fence_after();
      const bool live = quarter * 32 < rows;
      if (live) {
        // weights of the two partial results in a common frame
        // (only the halves the unit used are read: the other slot is stale)
        float a0 = 0.f, a1 = 0.f;
        if (gm == 3u) {
          const float2 lm0 = s.lm[i][0][r], lm1 = s.lm[i][1][r];
          const float mm = fmaxf(lm0.y, lm1.y);
          a0 = ex2_approx(lm0.y - mm);
          a1 = ex2_approx(lm1.y - mm);
          const float inv = 1.0f / (a0 * lm0.x + a1 * lm1.x);
          a0 *= inv;
          a1 *= inv;
        } else if (gm == 1u) {
          a0 = 1.0f / s.lm[i][0][r].x;
        } else {
          a1 = 1.0f / s.lm[i][1][r].x;
        }
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          uint32_t oa[32], ob[32];
          if (gm & 1u) tmem_ld32(tmem + lane_sel + tmem_o(0, u & 1) + 32u * h, oa);
          if (gm & 2u) tmem_ld32(tmem + lane_sel + tmem_o(1, u & 1) + 32u * h, ob);
          tmem_ld_wait();
          if (h == 1) {
            // all of O is in registers: the accumulators are free for the next unit
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
              if (gm & 1u) mbar_arrive(&s.o_free[0][u & 1]);
              if (gm & 2u) mbar_arrive(&s.o_free[1][u & 1]);
            }
          }
          float v[32];
          if (gm == 3u) {
#pragma unroll
            for (int e = 0; e < 32; ++e)
              v[e] = fmaf(__uint_as_float(oa[e]), a0, __uint_as_float(ob[e]) * a1);
          } else if (gm == 1u) {
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(oa[e]) * a0;
          } else {
#pragma unroll
            for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(ob[e]) * a1;
          }
#pragma unroll
          for (int c = 0; c < 4; ++c)
            stage[lane * 8 + ((4 * h + c) ^ (lane & 7))] =
                make_uint4(pack_bf16x2(v[c * 8 + 0], v[c * 8 + 1]),
                           pack_bf16x2(v[c * 8 + 2], v[c * 8 + 3]),
                           pack_bf16x2(v[c * 8 + 4], v[c * 8 + 5]),
                           pack_bf16x2(v[c * 8 + 6], v[c * 8 + 7]));
        }
      }
      // the unit's slot is free again (and O, if this warp's rows were dead)
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (!live) {
          if (gm & 1u) mbar_arrive(&s.o_free[0][u & 1]);
          if (gm & 2u) mbar_arrive(&s.o_free[1][u & 1]);
        }
        mbar_arrive(&s.ud_empty[i]);
      }
      if (live) {
        __syncwarp();
        const int c = lane & 7;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const int row = 4 * t + (lane >> 3);             // of this warp's 32
          if (quarter * 32 + row < rows)
            *reinterpret_cast<uint4*>(out + static_cast<size_t>(row0 + quarter * 32 + row) * dim +
                                      head * HD + c * 8) = stage[row * 8 + (c ^ (row & 7))];
        }
        __syncwarp();
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (*abort) {
    if (threadIdx.x == 0) {
      record_status(status, DORA_ERR_TIMEOUT);
      // let the last TMA load of every buffer land (earlier ones were consumed)
      for (int c = max(0, s.q_issued - 2); c < s.q_issued; ++c)
        mbar_wait_limited(&s.q_full[c & 1], (c >> 1) & 1, 100ull * 1000 * 1000);
      for (int c = max(0, s.kv_issued - kStages); c < s.kv_issued; ++c)
        mbar_wait_limited(&s.kv_full[c % kStages], (c / kStages) & 1, 100ull * 1000 * 1000);
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace split
}  // namespace attn

cudaError_t encode_qkv_maps(attn::QkvMaps* mp, const uint16_t* qkv, int32_t t_cap, int32_t heads) {
  const uint64_t row = static_cast<uint64_t>(3) * heads * attn::HD;
  CUtensorMap* maps[4] = {&mp->m128, &mp->m64, &mp->m32, &mp->m16};
  for (int i = 0; i < 4; ++i)
    if (encode_tmap_2d_bf16(maps[i], qkv, row, static_cast<uint64_t>(t_cap), row * 2, attn::HD,
                            static_cast<uint32_t>(attn::KC >> i)) != 0)
      return cudaErrorInvalidValue;
  return cudaSuccess;
}

// Images of up to 256 tokens have at most two key chunks, whose loads the
// two query tiles share: there one accumulator per query row (and three S/P
// buffers) measured faster; longer images run the per-key-half kernel above.
cudaError_t launch_varlen_attn(const uint16_t* qkv, const int32_t* cu, int32_t batch,
                               int32_t max_seqlen, int32_t t_cap, int32_t heads, float scale,
                               uint16_t* out, int32_t* status, cudaStream_t stream) {
  if (batch == 0 || t_cap == 0 || max_seqlen == 0) return cudaSuccess;
  attn::QkvMaps mp;
  cudaError_t e = encode_qkv_maps(&mp, qkv, t_cap, heads);
  if (e != cudaSuccess) return e;
  const long long ihs = static_cast<long long>(batch) * heads;
  if (ihs > 0x7fffffffLL) return cudaErrorInvalidValue;
  const float scale_log2 = scale * 1.4426950408889634f;
  if (max_seqlen <= 2 * attn::KC)
    return launch_varlen_attn_exchange(mp, cu, batch, max_seqlen, t_cap, heads, scale_log2, out,
                                       status, stream);
  const size_t smem = sizeof(attn::split::Smem);
  e = cudaFuncSetAttribute(attn::split::varlen_attn_kernel,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long cap = num_sms();
  const int grid = static_cast<int>(ihs < cap ? ihs : cap);
  return launch_pdl(attn::split::varlen_attn_kernel, dim3(grid), dim3(attn::kThreads), smem,
                    stream, mp, cu, batch, max_seqlen, t_cap, heads, scale_log2, out, status);
}

}  // namespace dora
