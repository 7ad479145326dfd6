// Packed variable-length multi-head self-attention on tcgen05 tensor cores,
// the kernel for images of up to 256 tokens (at most two key chunks, whose
// loads the image's two query tiles share); launch_varlen_attn in
// attn_tcgen05.cu picks it when max_seqlen <= 256.
// For image i (rows [cu[i], cu[i+1]) of the packed buffer) and head h:
//     O = softmax(Q K^T * scale) V
// with no attention across images and no padding (Sec. 3.5 "Inference").
//
// Work unit = (image, head, 128-row query tile); a unit walks its keys in
// chunks of 128 ("steps").  One persistent CTA per SM owns a contiguous range
// of image-heads, split by estimated cost, and runs its steps through a
// pipeline in which no role waits on the softmax's own previous work:
//   warp 0       walks the CTA's units, loads Q and K/V chunks by TMA in
//                128-row boxes (the two query tiles of an image of up to 256
//                tokens share the chunks), and publishes a descriptor per step
//                and per unit.  No other role keeps unit bookkeeping.  (Boxes
//                cut to the image's tail read fewer DRAM bytes but measured
//                slower on images of 35-134 tokens: the rows a 128-row box
//                reads past an image are the next image's, which it then finds
//                in L2.)
//   warps 1, 2   MMA issuers (one thread each): warp 1 issues S(j) = Q K^T
//                (M=128, N=keys rounded to 16, K=64) into S/P buffer j mod 3,
//                once PV(j-3) is done with that buffer; warp 2 issues O (+)= P(j) V
//                with P read from the same buffer, into O buffer (unit mod 2).
//                A single issuing thread could not keep up with 12 MMAs a step.
//   warps 4-11   softmax, two threads per query row (TMEM lane), 64 of a step's
//                128 S columns each, held in registers: the half maxima are
//                exchanged, then 2^x, partial row sum, and P (bf16) written over
//                the S columns just read.  Within a unit
//                the reference maximum is only raised when a later chunk exceeds
//                it by more than 2^8, and then O is rescaled in TMEM; otherwise
//                P stays below 2^8 in the old frame, which bf16 and fp32 hold
//                exactly as well.  The softmax also zeroes the V rows of a
//                chunk's last 16-key group that lie past the image.
//   warps 12-15  epilogue: when a unit's last PV is done, O / row sum, staged
//                through shared memory and stored four whole rows per store.
// TMEM (512 columns): S/P buffers 0-127, 128-255 and 256-383 (three, so
// that the loop softmax(j) -> PV(j) -> S(j+3) spans three steps), O buffers
// 384-447 and 448-511.  Rows past the image are computed but never stored; keys past it
// are masked, and V rows past it are zeroed so stale data cannot leak through
// 0 * NaN.
#include "attn_common.cuh"

namespace dora {
namespace attn {
namespace exch {

constexpr int kSpBufs = 3;      // S/P buffers, used by steps in turn
__device__ __forceinline__ uint32_t tmem_sp(int b) { return 128u * static_cast<uint32_t>(b); }
__device__ __forceinline__ uint32_t tmem_o(int b) {
  return 128u * kSpBufs + 64u * static_cast<uint32_t>(b);
}
static_assert(128 * kSpBufs + 2 * 64 <= 512, "TMEM columns");

// Step descriptor (one 32-bit word).
constexpr uint32_t kDStage = 0x3u;        // K/V stage
constexpr uint32_t kDKvPar = 1u << 2;     // phase parity of that stage's load
constexpr uint32_t kDFirst = 1u << 3;     // first key chunk of a unit
constexpr uint32_t kDLast = 1u << 4;      // last key chunk of a unit
constexpr uint32_t kDUPar = 1u << 5;      // unit parity: Q buffer and O buffer
constexpr uint32_t kDQPar = 1u << 6;      // phase parity of the unit's Q load
constexpr uint32_t kDRelease = 1u << 7;   // the K/V stage is free after this step's PV
constexpr uint32_t kDOWait = 1u << 8;     // the O buffer held an earlier unit
constexpr uint32_t kDOPar = 1u << 25;     // phase parity of that unit's O read-out
constexpr uint32_t kDEnd = 1u << 31;      // no more steps
__device__ __forceinline__ int d_kc(uint32_t d) { return static_cast<int>((d >> 9) & 0xFFu); }
__device__ __forceinline__ int d_rows(uint32_t d) { return static_cast<int>((d >> 17) & 0xFFu); }

struct Smem {
  uint16_t q[2][BQ * HD];       // 2 x 16 KB, by unit parity
  uint16_t k[kStages][KC * HD]; // 4 x 16 KB
  uint16_t v[kStages][KC * HD]; // 4 x 16 KB
  uint4 ostage[4][32 * 8];      // per epilogue warp: 32 output rows of 128 bytes
  float lsum[4][2][BQ];         // row sums of each column half, by unit mod 4
  float mx[kSpBufs][2][BQ];     // row maxima of each column half, by S/P buffer
  uint64_t q_full[2];
  uint64_t q_empty[2];
  uint64_t kv_full[kStages];
  uint64_t kv_empty[kStages];
  uint64_t s_full[kSpBufs];     // S of a step in S/P buffer b
  uint64_t p_full[kSpBufs];     // P written over it (one arrival per softmax warp)
  uint64_t xbar[kSpBufs][4];    // the two halves of a lane quarter exchanged their maxima
  uint64_t p_free[kSpBufs];     // PV of buffer b done
  uint64_t o_done[2];           // last PV of a unit in O buffer b done
  uint64_t o_free[2];           // O buffer b read out (one arrival per epilogue warp)
  uint64_t l_full[4];           // row sums of a unit (one arrival per softmax warp)
  uint64_t sd_full[kDescRing];  // step descriptor published
  uint64_t sd_empty[kDescRing]; // ... read by both issuers and the eight softmax warps
  uint64_t ud_full[kUnitRing];  // unit descriptor published
  uint64_t ud_empty[kUnitRing]; // ... read by the four epilogue warps
  uint64_t drain[2];
  uint32_t sdesc[kDescRing];
  uint32_t urow[kUnitRing];     // first output row of the unit
  uint32_t uhead[kUnitRing];    // head | rows << 16
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
      mbar_init(&s.o_done[b], 1);
      mbar_init(&s.o_free[b], 4);
    }
    for (int b = 0; b < kSpBufs; ++b) {
      mbar_init(&s.s_full[b], 1);
      mbar_init(&s.p_full[b], 8);
      for (int q = 0; q < 4; ++q) mbar_init(&s.xbar[b][q], 2);
      mbar_init(&s.p_free[b], 1);
    }
    for (int i = 0; i < 4; ++i) mbar_init(&s.l_full[i], 8);
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.kv_full[i], 1);
      mbar_init(&s.kv_empty[i], 1);
    }
    for (int i = 0; i < kDescRing; ++i) {
      mbar_init(&s.sd_full[i], 1);
      mbar_init(&s.sd_empty[i], 10);
    }
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&s.ud_full[i], 1);
      mbar_init(&s.ud_empty[i], 4);
    }
    mbar_init(&s.drain[0], 1);
    mbar_init(&s.drain[1], 1);
    s.abort_flag = 0;
    s.q_issued = s.kv_issued = 0;
    fence_barrier_init();
    tma_prefetch_desc(&mp.m128);
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
        {
          const int i = u % kUnitRing;
          if (!mbar_wait_sleep(&s.ud_empty[i], ((u / kUnitRing) & 1) ^ 1, abort, kSleepNs)) break;
          s.urow[i] = static_cast<uint32_t>(wk.lo + wk.qt * BQ);
          s.uhead[i] = static_cast<uint32_t>(wk.head) | (static_cast<uint32_t>(rows) << 16);
          mbar_arrive(&s.ud_full[i]);
        }
        const int qb = u & 1;
        if (!mbar_wait_sleep(&s.q_empty[qb], ((u >> 1) & 1) ^ 1, abort, kSleepNs)) break;
        mbar_arrive_expect_tx(&s.q_full[qb], BQ * HD * 2);
        tma_load_2d(s.q[qb], &mp.m128, &s.q_full[qb], wk.head * HD, wk.lo + wk.qt * BQ);
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
              mbar_arrive_expect_tx(&s.kv_full[stg], 2 * KC * HD * 2);
              const int row = wk.lo + c * KC;
              tma_load_2d(s.k[stg], &mp.m128, &s.kv_full[stg], dim + wk.head * HD, row);
              tma_load_2d(s.v[stg], &mp.m128, &s.kv_full[stg], 2 * dim + wk.head * HD, row);
            }
            ++loads;
            s.kv_issued = loads;
          }
          if (c < 2) {
            cur_stage[c] = stg;
            cur_par[c] = par;
          }
          const uint32_t d =
              static_cast<uint32_t>(stg) | (par ? kDKvPar : 0u) | (c == 0 ? kDFirst : 0u) |
              (c == nch - 1 ? kDLast : 0u) | ((u & 1) ? kDUPar : 0u) |
              (((u >> 1) & 1) ? kDQPar : 0u) | (reuse_next ? 0u : kDRelease) |
              (u >= 2 ? kDOWait : 0u) | ((((u >> 1) - 1) & 1) ? kDOPar : 0u) |
              (static_cast<uint32_t>(min(KC, n - c * KC)) << 9) |
              (static_cast<uint32_t>(rows) << 17);
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
  } else if (warp == 1 || warp == 2) {
    // ---------------- MMA issuers: warp 1 issues S, warp 2 issues PV (lane 0) ----------------
    // Each reads every step descriptor.  The only order between the two is
    // explicit: S(j + kSpBufs) waits until PV(j) has read S/P buffer j mod kSpBufs.
    if (lane == 0) {
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
          if ((d & kDFirst) &&
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
          if (d & kDLast) mma_commit(&s.q_empty[up]);
        } else {
          // O (+)= P(j) V into O buffer up
          constexpr uint32_t id_o = idesc_bf16(BQ, HD, true);
          const bool first = (d & kDFirst) != 0;
          if (first && (d & kDOWait) &&
              !mbar_wait_sleep(&s.o_free[up], (d & kDOPar) ? 1u : 0u, abort, kSleepNs))
            break;
          if (!mbar_wait_sleep(&s.p_full[b], bph, abort, kSleepNs)) break;
          tc_fence_after();
          const int nk = (d_kc(d) + 15) >> 4;
          const uint64_t vd = sdesc_sw128(smem_u32(s.v[stg]), 1024, 1024);
          const uint32_t dt = tmem + tmem_o(up), at = tmem + tmem_sp(b);
          mma_bf16_ts(dt, at, vd, id_o, first ? 0u : 1u);
#pragma unroll
          for (int kk = 1; kk < KC / 16; ++kk)   // 16 keys: 2048 bytes of V, 8 P columns
            if (kk < nk) mma_bf16_ts(dt, at + 8u * kk, vd + 128u * kk, id_o, 1u);
          mma_commit(&s.p_free[b]);
          if (d & kDLast) mma_commit(&s.o_done[up]);
          if (d & kDRelease) mma_commit(&s.kv_empty[stg]);
        }
      }
      mma_commit(&s.drain[warp - 1]);
      mbar_wait_limited(&s.drain[warp - 1], 0, kWaitLimitNs);
    }
  } else if (warp >= kSoftWarp0 && warp < kSoftWarp0 + 8) {
    // ---------------- softmax: two threads per query row, 64 columns each ----------------
    const int quarter = warp & 3;
    const int half = (warp - kSoftWarp0) >> 2;
    const int r = quarter * 32 + lane;                   // query row of the tile (TMEM lane)
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    float m_ref = 0.f, l = 0.f;                          // l: this half's partial row sum
    int u = 0;                                           // units finished
    auto step = [&](int j, uint32_t d) -> bool {
      const int kc = d_kc(d), kc16 = (kc + 15) & ~15;
      const int kh = min(max(kc - 64 * half, 0), 64);    // keys in this thread's half
      const bool live = quarter * 32 < d_rows(d);        // warp-uniform
      const int b = j % kSpBufs;
      const uint32_t bph = static_cast<uint32_t>(j / kSpBufs) & 1u;   // buffer use parity
      const uint32_t tsp = tmem + lane_sel + tmem_sp(b);
      if (!mbar_wait_warp_sleep(&s.s_full[b], bph, abort, kSleepNs)) return false;
      tc_fence_after();
      // S is done, so the K/V load landed: zero V rows [kc, kc16) (whole 128-byte rows)
      if (kc < kc16) {
        const int t = half * BQ + r;
        if (t < (kc16 - kc) * 8)
          reinterpret_cast<uint4*>(s.v[d & kDStage])[kc * 8 + t] = make_uint4(0u, 0u, 0u, 0u);
        fence_proxy_async_smem();
      }
      // this half's 64 S columns into registers (both blocks, always: arrays
      // filled only conditionally would stay live across iterations)
      uint32_t s0[32], s1[32];
      float mloc = -INFINITY;
      if (live) {
        tmem_ld32(tsp + static_cast<uint32_t>(64 * half), s0);
        tmem_ld32(tsp + static_cast<uint32_t>(64 * half + 32), s1);
        tmem_ld_wait();
        mask_tail(s0, kh);
        mask_tail(s1, kh - 32);
        mloc = max32(s1, max32(s0, -INFINITY));
      }
      // exchange the half maxima with the other thread of the row
      s.mx[b][half][r] = mloc;
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.xbar[b][quarter]);
      if (!mbar_wait_warp_sleep(&s.xbar[b][quarter], bph, abort, kSleepNs)) return false;
      const float mc = fmaxf(mloc, s.mx[b][half ^ 1][r]) * scale_log2;
      if (live) {
        // reference maximum: set on a unit's first chunk, raised past 2^8
        bool rescale = false;
        float alpha = 1.f;
        if (d & kDFirst) {
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
        // P over this half's S columns (16 columns per 32 keys)
        if (kh > 0) {
          exp32_pack(s0, scale_log2, -m_ref, l);
          tmem_st16(tsp + static_cast<uint32_t>(32 * half), lo16(s0));
        }
        if (kh > 32) {
          exp32_pack(s1, scale_log2, -m_ref, l);
          tmem_st16(tsp + static_cast<uint32_t>(32 * half + 16), lo16(s1));
        }
        if (rescale) {
          // O holds the chunks before this one once their PV is done: bring this
          // half's 32 columns to the raised reference before this chunk's PV
          const int pb = (j - 1) % kSpBufs;              // the previous step's buffer
          if (!mbar_wait_warp_sleep(&s.p_free[pb], static_cast<uint32_t>((j - 1) / kSpBufs) & 1u,
                                    abort, kSleepNs))
            return false;
          tc_fence_after();
          const uint32_t to = tmem + lane_sel + tmem_o((d & kDUPar) ? 1 : 0) +
                              static_cast<uint32_t>(32 * half);
          uint32_t o[32];
          tmem_ld32(to, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st16(to, lo16(o));
          tmem_st16(to + 16u, *reinterpret_cast<const uint32_t(*)[16]>(&o[16]));
        }
      }
      tmem_st_wait();
      if (d & kDLast) {
        s.lsum[u & 3][half][r] = l;
        warp_arrive(&s.l_full[u & 3]);
        ++u;
      }
      warp_arrive(&s.p_full[b]);
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
    // ---------------- epilogue: O / row sum, stored four rows per instruction ----------------
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    uint4* const stage = s.ostage[warp - kEpiWarp0];
    for (int u = 0;; ++u) {
      const int i = u % kUnitRing;
      // one descriptor per unit, then an end marker
      if (!mbar_wait_warp_sleep(&s.ud_full[i], (u / kUnitRing) & 1, abort, kSleepNs)) break;
      const uint32_t row0 = s.urow[i], hd = s.uhead[i];
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.ud_empty[i]);
      if (hd == 0xFFFFFFFFu) break;
      const int ob = u & 1;
      const int rows = static_cast<int>(hd >> 16), head = static_cast<int>(hd & 0xFFFFu);
      if (!mbar_wait_warp_sleep(&s.o_done[ob], (u >> 1) & 1, abort, kSleepNs)) break;
      if (!mbar_wait_warp_sleep(&s.l_full[u & 3], (u >> 2) & 1, abort, kSleepNs)) break;
      tc_fence_after();
      const bool live = quarter * 32 < rows;
      uint32_t oa[32], ob2[32];
      float inv = 1.f;
      if (live) {
        const uint32_t to = tmem + lane_sel + tmem_o(ob);
        tmem_ld32(to, oa);
        tmem_ld32(to + 32u, ob2);
        tmem_ld_wait();
        inv = 1.0f / (s.lsum[u & 3][0][r] + s.lsum[u & 3][1][r]);
      }
      warp_arrive(&s.o_free[ob]);
      if (live) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
          stage[lane * 8 + (c ^ (lane & 7))] = make_uint4(
              pack_bf16x2(__uint_as_float(oa[c * 8 + 0]) * inv, __uint_as_float(oa[c * 8 + 1]) * inv),
              pack_bf16x2(__uint_as_float(oa[c * 8 + 2]) * inv, __uint_as_float(oa[c * 8 + 3]) * inv),
              pack_bf16x2(__uint_as_float(oa[c * 8 + 4]) * inv, __uint_as_float(oa[c * 8 + 5]) * inv),
              pack_bf16x2(__uint_as_float(oa[c * 8 + 6]) * inv, __uint_as_float(oa[c * 8 + 7]) * inv));
#pragma unroll
        for (int c = 0; c < 4; ++c)
          stage[lane * 8 + ((c + 4) ^ (lane & 7))] = make_uint4(
              pack_bf16x2(__uint_as_float(ob2[c * 8 + 0]) * inv, __uint_as_float(ob2[c * 8 + 1]) * inv),
              pack_bf16x2(__uint_as_float(ob2[c * 8 + 2]) * inv, __uint_as_float(ob2[c * 8 + 3]) * inv),
              pack_bf16x2(__uint_as_float(ob2[c * 8 + 4]) * inv, __uint_as_float(ob2[c * 8 + 5]) * inv),
              pack_bf16x2(__uint_as_float(ob2[c * 8 + 6]) * inv, __uint_as_float(ob2[c * 8 + 7]) * inv));
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

}  // namespace exch
}  // namespace attn

cudaError_t launch_varlen_attn_exchange(const attn::QkvMaps& mp, const int32_t* cu,
                                        int32_t batch, int32_t max_seqlen, int32_t t_cap,
                                        int32_t heads, float scale_log2, uint16_t* out,
                                        int32_t* status, cudaStream_t stream) {
  const size_t smem = sizeof(attn::exch::Smem);
  cudaError_t e = cudaFuncSetAttribute(attn::exch::varlen_attn_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long ihs = static_cast<long long>(batch) * heads;
  const long long cap = num_sms();
  const int grid = static_cast<int>(ihs < cap ? ihs : cap);
  return launch_pdl(attn::exch::varlen_attn_kernel, dim3(grid), dim3(attn::kThreads), smem,
                    stream, mp, cu, batch, max_seqlen, t_cap, heads, scale_log2, out, status);
}

}  // namespace dora
