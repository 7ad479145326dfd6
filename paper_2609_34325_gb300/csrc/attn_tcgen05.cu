// Packed variable-length multi-head self-attention on tcgen05 tensor cores.
// For image i (rows [cu[i], cu[i+1]) of the packed buffer) and head h:
//     O = softmax(Q K^T * scale) V
// with no attention across images and no padding (Sec. 3.5 "Inference").
//
// Work unit = (image, head, 128-row query tile); a unit walks its keys in
// chunks of 128 ("steps").  One persistent CTA per SM owns a contiguous range
// of image-heads, split by estimated cost.  The CTA's units alternate between
// two warpgroups; each has its own MMA issuer, so the two run independently
// and one's exponentials overlap the other's tensor-core work:
//   warp 0       walks the CTA's steps two at a time (one per warpgroup), loads
//                Q and K/V chunks by TMA (a chunk both warpgroups need in the
//                same round is loaded once) and publishes a step descriptor per
//                warpgroup and a unit descriptor for the epilogue.  No other
//                role keeps unit bookkeeping.
//   warps 1, 14  MMA issuers of warpgroups 0 and 1 (one thread each):
//                S = Q K^T (M=128, N=keys rounded to 16, K=64) into the
//                warpgroup's S columns, then O (+)= P V with P read from TMEM.
//                A step's S is issued as soon as the previous S has been read,
//                ahead of the previous step's PV.
//   warps 2-9    softmax warpgroups, one thread per query row (TMEM lane):
//                row maximum, 2^x, row sum; P (bf16) to its own TMEM columns.
//                Within a unit the reference maximum is only raised when a
//                later chunk exceeds it by more than 2^8, and then O is rescaled
//                in TMEM; otherwise P stays below 2^8 in the old frame, which
//                bf16 and fp32 hold exactly as well.  They also zero the V rows
//                of a chunk's last 16-key group that lie past the image.
//   warps 10-13  epilogue: once a unit's last PV is done, O is read from TMEM,
//                divided by the row sum and stored; the O columns are handed
//                back for the warpgroup's next unit.
// TMEM (512 columns): warpgroup w owns [256w, 256w+256): S 0-127, P 128-191,
// O 192-255.  Rows past the image are computed but never stored; keys past it
// are masked, and V rows past it are zeroed so stale data cannot leak through
// 0 * NaN.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "dora_ptx.cuh"
#include "token_ops.cuh"

namespace dora {
namespace attn {

constexpr int BQ = 128;         // query rows per unit
constexpr int KC = 128;         // keys per step
constexpr int HD = 64;
constexpr int kStages = 4;      // K/V chunk ring
constexpr int kDescRing = 8;    // step descriptors in flight per warpgroup
constexpr int kUnitRing = 4;    // unit descriptors in flight per warpgroup
constexpr int kThreads = 480;   // 15 warps
constexpr int kIssuer0 = 1, kIssuer1 = 14;   // MMA issuer warps of warpgroups 0 and 1
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleLog2 = 8.f;    // raise the reference maximum past 2^8
constexpr uint32_t kSleepNs = 200000;  // waiting threads sleep instead of spinning
__device__ __forceinline__ uint32_t tmem_s(int w) { return 256u * static_cast<uint32_t>(w); }
__device__ __forceinline__ uint32_t tmem_p(int w) { return 256u * static_cast<uint32_t>(w) + 128u; }
__device__ __forceinline__ uint32_t tmem_o(int w) { return 256u * static_cast<uint32_t>(w) + 192u; }

// Step descriptor (one 32-bit word).
constexpr uint32_t kDStage = 0x3u;        // K/V stage
constexpr uint32_t kDKvPar = 1u << 2;     // phase parity of that stage's load
constexpr uint32_t kDFirst = 1u << 3;     // first key chunk of a unit
constexpr uint32_t kDLast = 1u << 4;      // last key chunk of a unit
constexpr uint32_t kDQbuf = 1u << 5;      // Q buffer of the unit
constexpr uint32_t kDQPar = 1u << 6;      // phase parity of that Q load
constexpr uint32_t kDPrevUnit = 1u << 7;  // the warpgroup had an earlier unit
constexpr uint32_t kDSolo = 1u << 8;      // the only step reading this K/V load
constexpr uint32_t kDEnd = 1u << 31;      // no more steps for this warpgroup
__device__ __forceinline__ int d_kc(uint32_t d) { return static_cast<int>((d >> 9) & 0xFFu); }
__device__ __forceinline__ int d_rows(uint32_t d) { return static_cast<int>((d >> 17) & 0xFFu); }
constexpr uint32_t kUEnd = 0xFFFFFFFFu;   // unit descriptor: no more units

struct Smem {
  uint16_t q[2][2][BQ * HD];    // [warpgroup][buffer], 4 x 16 KB
  uint16_t k[kStages][KC * HD]; // 4 x 16 KB
  uint16_t v[kStages][KC * HD]; // 4 x 16 KB
  float lsum[2][2][BQ];         // row sums [warpgroup][unit parity]
  uint64_t q_full[2][2];
  uint64_t q_empty[2][2];
  uint64_t kv_full[kStages];
  uint64_t kv_empty[kStages];   // two arrivals: both readers' PVs (a solo reader arrives twice)
  uint64_t s_full[2];           // S of warpgroup w computed
  uint64_t s_free[2];           // ... and read (one arrival per warp)
  uint64_t p_full[2];           // P written, O rescaled, V tail zeroed (one arrival per warp)
  uint64_t p_free[2];           // PV done: P buffer free, O current
  uint64_t o_done[2];           // last PV of a unit done
  uint64_t o_free[2];           // O read by the epilogue (one arrival per warp)
  uint64_t l_full[2][2];        // row sums of a unit written (one arrival per warp)
  uint64_t sd_full[2][kDescRing];   // step descriptor published
  uint64_t sd_empty[2][kDescRing];  // ... read by the issuer and the four softmax warps
  uint64_t ud_full[2][kUnitRing];   // unit descriptor published
  uint64_t ud_empty[2][kUnitRing];  // ... read by the four epilogue warps
  uint64_t drain[2];
  uint32_t sdesc[2][kDescRing];
  uint32_t urow[2][kUnitRing];      // first output row of the unit
  uint32_t uhead[2][kUnitRing];     // head | rows << 16, or kUEnd
  uint32_t tmem_base;
  int abort_flag;
  int ih_begin, ih_end;
  int q_issued[2], kv_issued;
};

// Rows of image `img`, clamped to the buffer (0 when its start lies outside).
__device__ __forceinline__ int image_rows(const int32_t* cu, int img, int t_cap, int& lo) {
  lo = cu[img];
  const int n = cu[img + 1] - lo;
  if (lo < 0 || lo > t_cap) {
    lo = 0;
    return 0;
  }
  return n < 0 ? 0 : (n > t_cap - lo ? t_cap - lo : n);
}

// Estimated cost of one image-head with n rows, in steps: every query tile
// walks every key chunk, plus one step of per-unit overhead.
__device__ __forceinline__ long long ih_cost(int n) {
  const long long q = (n + BQ - 1) / BQ;
  return q * (q + 1);
}

// Units (image, head, query tile) of the image-heads [ih, ih_end), in order.
// Image and head advance incrementally; an image's bounds are read once.
struct Walker {
  const int32_t* cu;
  int heads, t_cap;
  int ih, ih_end, img, head, lo, n, qt, nqt;
  __device__ __forceinline__ void load_image() {
    n = image_rows(cu, img, t_cap, lo);
    nqt = (n + BQ - 1) / BQ;
  }
  __device__ __forceinline__ void settle() {
    while (ih < ih_end && qt >= nqt) {
      ++ih;
      qt = 0;
      if (++head == heads) {
        head = 0;
        ++img;
        if (ih < ih_end) load_image();
      }
    }
  }
  __device__ __forceinline__ void start(const int32_t* c, int h, int tc, int b, int e) {
    cu = c;
    heads = h;
    t_cap = tc;
    ih = b;
    ih_end = e;
    img = b / h;
    head = b - img * h;
    lo = n = qt = nqt = 0;
    if (ih < ih_end) load_image();
    settle();
  }
  __device__ __forceinline__ bool done() const { return ih >= ih_end; }
  __device__ __forceinline__ void next() {
    if (ih < ih_end) {
      ++qt;
      settle();
    }
  }
};

// The steps (unit, key chunk) of one softmax warpgroup: the CTA's units of
// parity `wg`, each walked chunk by chunk.
struct Steps {
  Walker u;
  int c, nch, ju;
  bool has;
  __device__ __forceinline__ void refresh() {
    has = !u.done();
    nch = has ? (u.n + KC - 1) / KC : 0;
  }
  __device__ __forceinline__ void start(const int32_t* cu, int heads, int t_cap, int b, int e,
                                        int wg) {
    u.start(cu, heads, t_cap, b, e);
    if (wg) u.next();
    c = 0;
    ju = 0;
    refresh();
  }
  __device__ __forceinline__ void next_unit() {
    c = 0;
    ++ju;
    u.next();
    u.next();
    refresh();
  }
  __device__ __forceinline__ void advance() {
    if (++c < nch) return;
    next_unit();
  }
  __device__ __forceinline__ int kc() const { return min(KC, u.n - c * KC); }
  __device__ __forceinline__ int q_rows() const { return min(BQ, u.n - u.qt * BQ); }
  __device__ __forceinline__ bool last() const { return c == nch - 1; }
};

// Whole warp: the CTA's image-head range.  Image-head ih belongs to CTA
// floor(C(ih) * grid / total), C being the cost of the image-heads before it;
// CTA 0 also checks every image against the buffer and max_seqlen.
__device__ void find_range(const int32_t* cu, int batch, int heads, int t_cap, int max_seqlen,
                           int32_t* status, long long& ih_b, long long& ih_e) {
  const int lane = threadIdx.x & 31;
  long long total = 0;
  for (int i0 = 0; i0 < batch; i0 += 32) {
    const int i = i0 + lane;
    long long c = 0;
    if (i < batch) {
      int lo;
      c = ih_cost(image_rows(cu, i, t_cap, lo));
      if (blockIdx.x == 0) {
        const int l0 = cu[i], n = cu[i + 1] - l0;
        if (l0 < 0 || l0 > t_cap || n > t_cap - l0 || n > max_seqlen)
          record_status(status, DORA_ERR_DEVICE_SEQLEN);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    total += c;
  }
  const long long nih = static_cast<long long>(batch) * heads;
  const long long G = gridDim.x, b = blockIdx.x;
  ih_b = nih;
  ih_e = nih;
  if (total == 0) {
    ih_b = ih_e = 0;
    return;
  }
  total *= heads;
  const long long xb = b * total, xe = (b + 1) * total;
  bool fb = false, fe = (b == G - 1);
  long long pre = 0;                 // cost of one head of the images before i0
  for (int i0 = 0; i0 < batch && !(fb && fe); i0 += 32) {
    const int i = i0 + lane;
    long long c = 0;
    if (i < batch) {
      int lo;
      c = ih_cost(image_rows(cu, i, t_cap, lo));
    }
    long long incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long t = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += t;
    }
    const long long base = static_cast<long long>(heads) * (pre + incl - c) * G;   // C(i, 0) * G
    // first image-head of image i whose C * G reaches x, or -1
    auto first_at = [&](long long x) -> long long {
      if (i >= batch) return -1;
      if (base >= x) return static_cast<long long>(i) * heads;
      if (c > 0) {
        const long long h = (x - base + c * G - 1) / (c * G);
        if (h < heads) return static_cast<long long>(i) * heads + h;
      }
      return -1;
    };
    if (!fb) {
      const long long r = first_at(xb);
      const unsigned m = __ballot_sync(0xffffffffu, r >= 0);
      if (m) {
        ih_b = __shfl_sync(0xffffffffu, r, __ffs(m) - 1);
        fb = true;
      }
    }
    if (!fe) {
      const long long r = first_at(xe);
      const unsigned m = __ballot_sync(0xffffffffu, r >= 0);
      if (m) {
        ih_e = __shfl_sync(0xffffffffu, r, __ffs(m) - 1);
        fe = true;
      }
    }
    pre += __shfl_sync(0xffffffffu, incl, 31);
  }
}

__device__ __forceinline__ void mask_tail(uint32_t (&a)[32], int live) {
  if (live < 32) {
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (e >= live) a[e] = __float_as_uint(-INFINITY);
  }
}

__device__ __forceinline__ float max32(const uint32_t (&a)[32], float m) {
  float m0 = m, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY;
#pragma unroll
  for (int e = 0; e < 32; e += 8) {
    m0 = max3f(m0, __uint_as_float(a[e]), __uint_as_float(a[e + 1]));
    m1 = max3f(m1, __uint_as_float(a[e + 2]), __uint_as_float(a[e + 3]));
    m2 = max3f(m2, __uint_as_float(a[e + 4]), __uint_as_float(a[e + 5]));
    m3 = max3f(m3, __uint_as_float(a[e + 6]), __uint_as_float(a[e + 7]));
  }
  return max3f(m0, m1, fmaxf(m2, m3));
}

// p = 2^(s * scale_log2 - m) for 32 keys: packed to bf16, summed into l.
__device__ __forceinline__ void exp32(const uint32_t (&a)[32], float scale_log2, float neg_m,
                                      uint32_t (&pk)[16], float& l) {
  float l0 = 0.f, l1 = 0.f, l2 = 0.f, l3 = 0.f;
#pragma unroll
  for (int e = 0; e < 32; e += 4) {
    const float p0 = ex2_approx(fmaf(__uint_as_float(a[e]), scale_log2, neg_m));
    const float p1 = ex2_approx(fmaf(__uint_as_float(a[e + 1]), scale_log2, neg_m));
    const float p2 = ex2_approx(fmaf(__uint_as_float(a[e + 2]), scale_log2, neg_m));
    const float p3 = ex2_approx(fmaf(__uint_as_float(a[e + 3]), scale_log2, neg_m));
    l0 += p0;
    l1 += p1;
    l2 += p2;
    l3 += p3;
    pk[e >> 1] = pack_bf16x2(p0, p1);
    pk[(e >> 1) + 1] = pack_bf16x2(p2, p3);
  }
  l += (l0 + l1) + (l2 + l3);
}

// One arrival for the whole warp, after every lane's prior tcgen05 accesses.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  tc_fence_before();
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

__global__ void __launch_bounds__(kThreads, 1)
    varlen_attn_kernel(const __grid_constant__ CUtensorMap tm, const int32_t* __restrict__ cu,
                       int batch, int max_seqlen, int t_cap, int heads, float scale_log2,
                       uint16_t* __restrict__ out, int32_t* status) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_u32(smem_raw) & 1023u) {
    if (threadIdx.x == 0) record_status(status, DORA_ERR_UNSUPPORTED);
    return;
  }
  Smem& s = *reinterpret_cast<Smem*>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int dim = heads * HD;

  if (warp == 0) {
    long long b, e;
    find_range(cu, batch, heads, t_cap, max_seqlen, status, b, e);
    if (lane == 0) {
      s.ih_begin = static_cast<int>(b);
      s.ih_end = static_cast<int>(e);
    }
  } else if (threadIdx.x == 64) {
    for (int w = 0; w < 2; ++w) {
      for (int b = 0; b < 2; ++b) {
        mbar_init(&s.q_full[w][b], 1);
        mbar_init(&s.q_empty[w][b], 1);
        mbar_init(&s.l_full[w][b], 4);
      }
      mbar_init(&s.s_full[w], 1);
      mbar_init(&s.s_free[w], 4);
      mbar_init(&s.p_full[w], 4);
      mbar_init(&s.p_free[w], 1);
      mbar_init(&s.o_done[w], 1);
      mbar_init(&s.o_free[w], 4);
      for (int i = 0; i < kDescRing; ++i) {
        mbar_init(&s.sd_full[w][i], 1);
        mbar_init(&s.sd_empty[w][i], 5);
      }
      for (int i = 0; i < kUnitRing; ++i) {
        mbar_init(&s.ud_full[w][i], 1);
        mbar_init(&s.ud_empty[w][i], 4);
      }
      mbar_init(&s.drain[w], 1);
    }
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.kv_full[i], 1);
      mbar_init(&s.kv_empty[i], 2);
    }
    s.abort_flag = 0;
    s.q_issued[0] = s.q_issued[1] = s.kv_issued = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tm);
  }
  if (warp == 1) tmem_alloc(&s.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_base;
  volatile int* abort = &s.abort_flag;
  const int ih_b = s.ih_begin, ih_e = s.ih_end;

  if (warp == 0) {
    // ---------------- scheduler + TMA producer ----------------
    if (lane == 0) {
      Steps st[2];
      st[0].start(cu, heads, t_cap, ih_b, ih_e, 0);
      st[1].start(cu, heads, t_cap, ih_b, ih_e, 1);
      int loads = 0, qn[2] = {0, 0}, dn[2] = {0, 0}, un[2] = {0, 0};
      bool ended[2] = {false, false};
      bool ok = true;
      auto desc = [&](int w, uint32_t d) -> bool {
        const int i = dn[w] % kDescRing;
        if (!mbar_wait_sleep(&s.sd_empty[w][i], ((dn[w] / kDescRing) & 1) ^ 1, abort, kSleepNs))
          return false;
        s.sdesc[w][i] = d;
        mbar_arrive(&s.sd_full[w][i]);
        ++dn[w];
        return true;
      };
      auto unit = [&](int w, uint32_t row, uint32_t hd) -> bool {
        const int i = un[w] % kUnitRing;
        if (!mbar_wait_sleep(&s.ud_empty[w][i], ((un[w] / kUnitRing) & 1) ^ 1, abort, kSleepNs))
          return false;
        s.urow[w][i] = row;
        s.uhead[w][i] = hd;
        mbar_arrive(&s.ud_full[w][i]);
        ++un[w];
        return true;
      };
      while (ok && !(ended[0] && ended[1])) {
        // this round: the next step of each warpgroup; one load when they share a chunk
        const bool shared = !ended[0] && !ended[1] && st[0].has && st[1].has &&
                            st[0].u.ih == st[1].u.ih && st[0].c == st[1].c;
        int load0 = 0;
        for (int w = 0; w < 2 && ok; ++w) {
          if (ended[w]) continue;
          Steps& x = st[w];
          if (!x.has) {
            ok = desc(w, kDEnd) && unit(w, 0u, kUEnd);
            ended[w] = true;
            continue;
          }
          const int rows = x.q_rows();
          if (x.c == 0) {
            if (!unit(w, static_cast<uint32_t>(x.u.lo + x.u.qt * BQ),
                      static_cast<uint32_t>(x.u.head) | (static_cast<uint32_t>(rows) << 16))) {
              ok = false;
              break;
            }
            const int qb = qn[w] & 1;
            if (!mbar_wait_sleep(&s.q_empty[w][qb], ((qn[w] >> 1) & 1) ^ 1, abort, kSleepNs)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&s.q_full[w][qb], BQ * HD * 2);
            tma_load_2d(s.q[w][qb], &tm, &s.q_full[w][qb], x.u.head * HD, x.u.lo + x.u.qt * BQ);
            ++qn[w];
          }
          int ld = load0;
          if (!(w == 1 && shared)) {
            ld = loads;
            const int stg = ld % kStages;
            if (!mbar_wait_sleep(&s.kv_empty[stg], ((ld / kStages) & 1) ^ 1, abort, kSleepNs)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&s.kv_full[stg], 2 * KC * HD * 2);
            const int row = x.u.lo + x.c * KC;
            tma_load_2d(s.k[stg], &tm, &s.kv_full[stg], dim + x.u.head * HD, row);
            tma_load_2d(s.v[stg], &tm, &s.kv_full[stg], 2 * dim + x.u.head * HD, row);
            ++loads;
            load0 = ld;
          }
          const int qi = qn[w] - 1;                       // this unit's Q load
          const uint32_t d =
              static_cast<uint32_t>(ld % kStages) | (((ld / kStages) & 1) ? kDKvPar : 0u) |
              (x.c == 0 ? kDFirst : 0u) | (x.last() ? kDLast : 0u) | ((qi & 1) ? kDQbuf : 0u) |
              (((qi >> 1) & 1) ? kDQPar : 0u) | (x.ju > 0 ? kDPrevUnit : 0u) |
              (shared ? 0u : kDSolo) | (static_cast<uint32_t>(x.kc()) << 9) |
              (static_cast<uint32_t>(rows) << 17);
          if (!desc(w, d)) {
            ok = false;
            break;
          }
          x.advance();
        }
      }
      s.q_issued[0] = qn[0];
      s.q_issued[1] = qn[1];
      s.kv_issued = loads;
    }
  } else if (warp == kIssuer0 || warp == kIssuer1) {
    // ---------------- MMA issuer of warpgroup w (lane 0) ----------------
    const int w = warp == kIssuer0 ? 0 : 1;
    if (lane == 0) {
      constexpr uint32_t id_o = idesc_bf16(BQ, HD, true);
      const uint32_t ts = tmem + tmem_s(w), tp = tmem + tmem_p(w), to = tmem + tmem_o(w);
      int j = 0, ju = 0;
      bool ok = true;
      auto next_desc = [&](uint32_t& d) -> bool {
        const int i = j % kDescRing;
        if (!mbar_wait_sleep(&s.sd_full[w][i], (j / kDescRing) & 1, abort, kSleepNs)) return false;
        d = s.sdesc[w][i];
        mbar_arrive(&s.sd_empty[w][i]);
        return true;
      };
      // S = Q K^T of step j
      auto issue_s = [&](uint32_t d) -> bool {
        const int stg = static_cast<int>(d & kDStage);
        const uint32_t qb = (d & kDQbuf) ? 1u : 0u;
        if ((d & kDFirst) &&
            !mbar_wait_sleep(&s.q_full[w][qb], (d & kDQPar) ? 1u : 0u, abort, kSleepNs))
          return false;
        if (!mbar_wait_sleep(&s.kv_full[stg], (d & kDKvPar) ? 1u : 0u, abort, kSleepNs))
          return false;
        if (j > 0 && !mbar_wait_sleep(&s.s_free[w], (j - 1) & 1, abort, kSleepNs)) return false;
        tc_fence_after();
        const uint64_t qd = sdesc_sw128(smem_u32(s.q[w][qb]), 16, 1024);
        const uint64_t kd = sdesc_sw128(smem_u32(s.k[stg]), 16, 1024);
        const uint32_t id_s = idesc_bf16(BQ, (d_kc(d) + 15) & ~15, false);
        mma_bf16_ss(ts, qd, kd, id_s, 0u);
        mma_bf16_ss(ts, qd + 2, kd + 2, id_s, 1u);
        mma_bf16_ss(ts, qd + 4, kd + 4, id_s, 1u);
        mma_bf16_ss(ts, qd + 6, kd + 6, id_s, 1u);
        mma_commit(&s.s_full[w]);
        if (d & kDLast) mma_commit(&s.q_empty[w][qb]);
        ++j;
        return true;
      };
      // O (+)= P V of step jp
      auto issue_pv = [&](uint32_t d, int jp) -> bool {
        const bool first = (d & kDFirst) != 0;
        if (first && (d & kDPrevUnit) &&
            !mbar_wait_sleep(&s.o_free[w], (ju - 1) & 1, abort, kSleepNs))
          return false;
        if (!mbar_wait_sleep(&s.p_full[w], jp & 1, abort, kSleepNs)) return false;
        tc_fence_after();
        const int nk = (d_kc(d) + 15) >> 4;
        const uint64_t vd = sdesc_sw128(smem_u32(s.v[d & kDStage]), 1024, 1024);
        mma_bf16_ts(to, tp, vd, id_o, first ? 0u : 1u);
#pragma unroll
        for (int kk = 1; kk < KC / 16; ++kk)   // 16 keys: 2048 bytes of V, 8 P columns
          if (kk < nk) mma_bf16_ts(to, tp + 8u * kk, vd + 128u * kk, id_o, 1u);
        mma_commit(&s.p_free[w]);
        if (d & kDLast) {
          mma_commit(&s.o_done[w]);
          ++ju;
        }
        mma_commit(&s.kv_empty[d & kDStage]);
        if (d & kDSolo) mma_commit(&s.kv_empty[d & kDStage]);
        return true;
      };
      uint32_t dcur;
      ok = next_desc(dcur);
      if (ok && !(dcur & kDEnd)) {
        ok = issue_s(dcur);
        while (ok) {
          uint32_t dn;
          if (!next_desc(dn)) break;
          const bool end = (dn & kDEnd) != 0;
          if (!end && !issue_s(dn)) break;
          if (!issue_pv(dcur, j - (end ? 1 : 2))) break;
          if (end) break;
          dcur = dn;
        }
      }
      mma_commit(&s.drain[w]);
      mbar_wait_limited(&s.drain[w], 0, kWaitLimitNs);
    }
  } else if (warp < 10) {
    // ---------------- softmax: warpgroup w, one thread per query row ----------------
    const int w = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;                   // query row of the tile (TMEM lane)
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t ts = tmem + lane_sel + tmem_s(w);
    const uint32_t tp = tmem + lane_sel + tmem_p(w);
    const uint32_t to = tmem + lane_sel + tmem_o(w);
    float m_ref = 0.f, l = 0.f;
    int ju = 0;
    auto step = [&](int j, uint32_t d) -> bool {
      const int kc = d_kc(d), kc16 = (kc + 15) & ~15;
      const int nb = (kc + 31) >> 5;
      const bool live = quarter * 32 < d_rows(d);        // warp-uniform
      if (!mbar_wait_warp_sleep(&s.s_full[w], j & 1, abort, kSleepNs)) return false;
      tc_fence_after();
      // S is done, so the K/V load landed: zero V rows [kc, kc16) (whole 128-byte rows)
      if (kc < kc16) {
        const int t = r;                                  // 0..127 over the warpgroup
        if (t < (kc16 - kc) * 8)
          reinterpret_cast<uint4*>(s.v[d & kDStage])[kc * 8 + t] = make_uint4(0u, 0u, 0u, 0u);
        fence_proxy_async_smem();
      }
      bool p_ok = j == 0;                                // P buffer known to be free
      if (live) {
        float mloc = -INFINITY;
        for (int b = 0; b < nb; ++b) {
          uint32_t a[32];
          tmem_ld32(ts + static_cast<uint32_t>(32 * b), a);
          tmem_ld_wait();
          mask_tail(a, kc - 32 * b);
          mloc = max32(a, mloc);
        }
        const float mc = mloc * scale_log2;
        if (d & kDFirst) {
          m_ref = mc;
          l = 0.f;
        } else {
          const bool need = mc > m_ref + kRescaleLog2;
          if (__any_sync(0xffffffffu, need)) {
            // raise the reference: O (complete up to the previous chunk) and l
            if (!mbar_wait_warp_sleep(&s.p_free[w], (j - 1) & 1, abort, kSleepNs)) return false;
            p_ok = true;
            tc_fence_after();
            const float m_new = need ? mc : m_ref;
            const float alpha = ex2_approx(m_ref - m_new);
#pragma unroll 1
            for (int h = 0; h < 2; ++h) {
              uint32_t o[32], o2[16];
              tmem_ld32(to + static_cast<uint32_t>(32 * h), o);
              tmem_ld_wait();
#pragma unroll
              for (int e = 0; e < 16; ++e) o2[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
              tmem_st16(to + static_cast<uint32_t>(32 * h), o2);
#pragma unroll
              for (int e = 0; e < 16; ++e) o2[e] = __float_as_uint(__uint_as_float(o[e + 16]) * alpha);
              tmem_st16(to + static_cast<uint32_t>(32 * h + 16), o2);
            }
            l *= alpha;
            m_ref = m_new;
          }
        }
        if (!p_ok) {
          if (!mbar_wait_warp_sleep(&s.p_free[w], (j - 1) & 1, abort, kSleepNs)) return false;
          tc_fence_after();
        }
        for (int b = 0; b < nb; ++b) {
          uint32_t a[32], pk[16];
          tmem_ld32(ts + static_cast<uint32_t>(32 * b), a);
          tmem_ld_wait();
          if (b == nb - 1) warp_arrive(&s.s_free[w]);
          mask_tail(a, kc - 32 * b);
          exp32(a, scale_log2, -m_ref, pk, l);
          tmem_st16(tp + static_cast<uint32_t>(16 * b), pk);
        }
        tmem_st_wait();
      } else {
        warp_arrive(&s.s_free[w]);
        // arrive on p_full only after the previous PV: keeps phases apart
        if (!p_ok && !mbar_wait_warp_sleep(&s.p_free[w], (j - 1) & 1, abort, kSleepNs)) return false;
      }
      if (d & kDLast) {
        s.lsum[w][ju & 1][r] = l;
        warp_arrive(&s.l_full[w][ju & 1]);
        ++ju;
      }
      warp_arrive(&s.p_full[w]);
      return true;
    };
    for (int j = 0;; ++j) {
      const int i = j % kDescRing;
      if (!mbar_wait_warp_sleep(&s.sd_full[w][i], (j / kDescRing) & 1, abort, kSleepNs)) break;
      const uint32_t d = s.sdesc[w][i];
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.sd_empty[w][i]);
      if ((d & kDEnd) || !step(j, d)) break;
    }
  } else {
    // ---------------- epilogue: normalise and store O ----------------
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    int ue[2] = {0, 0};
    bool have[2] = {false, false}, done[2] = {false, false};
    uint32_t urow[2] = {0u, 0u}, uhd[2] = {0u, 0u};
    uint64_t t0 = 0;
    uint32_t spins = 0;
    bool ok = true;
    // Units finish out of order between the warpgroups: serve whichever is done.
    while (ok && !(done[0] && done[1])) {
      bool did = false;
      for (int w = 0; w < 2 && ok; ++w) {
        if (done[w]) continue;
        const uint32_t hint = done[w ^ 1] ? 4096u : 256u;
        if (!have[w]) {
          const int i = ue[w] % kUnitRing;
          if (!__all_sync(0xffffffffu,
                          mbar_try_wait_hint(&s.ud_full[w][i], (ue[w] / kUnitRing) & 1, hint)))
            continue;
          urow[w] = s.urow[w][i];
          uhd[w] = s.uhead[w][i];
          __syncwarp();
          if (lane == 0) mbar_arrive(&s.ud_empty[w][i]);
          did = true;
          if (uhd[w] == kUEnd) {
            done[w] = true;
            continue;
          }
          have[w] = true;
        }
        if (!__all_sync(0xffffffffu, mbar_try_wait_hint(&s.o_done[w], ue[w] & 1, hint))) continue;
        const int ub = ue[w] & 1;
        if (!mbar_wait_warp_sleep(&s.l_full[w][ub], (ue[w] >> 1) & 1, abort, kSleepNs)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int q_rows = static_cast<int>(uhd[w] >> 16);
        const int head = static_cast<int>(uhd[w] & 0xFFFFu);
        const bool live = quarter * 32 < q_rows;
        uint32_t oa[32], ob[32];
        float lr = 1.f;
        if (live) {
          const uint32_t to = tmem + lane_sel + tmem_o(w);
          tmem_ld32(to, oa);
          tmem_ld32(to + 32u, ob);
          tmem_ld_wait();
          lr = s.lsum[w][ub][r];
        }
        warp_arrive(&s.o_free[w]);
        if (live && r < q_rows) {
          const float inv = 1.0f / lr;
          uint4* dst = reinterpret_cast<uint4*>(
              out + static_cast<size_t>(urow[w] + r) * dim + head * HD);
#pragma unroll
          for (int qd = 0; qd < 4; ++qd)
            dst[qd] = make_uint4(
                pack_bf16x2(__uint_as_float(oa[qd * 8 + 0]) * inv, __uint_as_float(oa[qd * 8 + 1]) * inv),
                pack_bf16x2(__uint_as_float(oa[qd * 8 + 2]) * inv, __uint_as_float(oa[qd * 8 + 3]) * inv),
                pack_bf16x2(__uint_as_float(oa[qd * 8 + 4]) * inv, __uint_as_float(oa[qd * 8 + 5]) * inv),
                pack_bf16x2(__uint_as_float(oa[qd * 8 + 6]) * inv, __uint_as_float(oa[qd * 8 + 7]) * inv));
#pragma unroll
          for (int qd = 0; qd < 4; ++qd)
            dst[4 + qd] = make_uint4(
                pack_bf16x2(__uint_as_float(ob[qd * 8 + 0]) * inv, __uint_as_float(ob[qd * 8 + 1]) * inv),
                pack_bf16x2(__uint_as_float(ob[qd * 8 + 2]) * inv, __uint_as_float(ob[qd * 8 + 3]) * inv),
                pack_bf16x2(__uint_as_float(ob[qd * 8 + 4]) * inv, __uint_as_float(ob[qd * 8 + 5]) * inv),
                pack_bf16x2(__uint_as_float(ob[qd * 8 + 6]) * inv, __uint_as_float(ob[qd * 8 + 7]) * inv));
        }
        have[w] = false;
        ++ue[w];
        did = true;
      }
      if (did) {
        t0 = 0;
        spins = 0;
      } else if ((++spins & 15u) == 0u) {
        // bounded idle time, decided by lane 0 for the whole warp
        int quit = 0;
        if (lane == 0) {
          const uint64_t now = globaltimer_ns();
          if (t0 == 0) t0 = now;
          if (*abort) {
            quit = 1;
          } else if (now - t0 > kWaitLimitNs) {
            *abort = 1;
            quit = 1;
          }
        }
        if (__shfl_sync(0xffffffffu, quit, 0)) ok = false;
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
      for (int w = 0; w < 2; ++w)
        for (int c = max(0, s.q_issued[w] - 2); c < s.q_issued[w]; ++c)
          mbar_wait_limited(&s.q_full[w][c & 1], (c >> 1) & 1, 100ull * 1000 * 1000);
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

}  // namespace attn

cudaError_t launch_varlen_attn(const uint16_t* qkv, const int32_t* cu, int32_t batch,
                               int32_t max_seqlen, int32_t t_cap, int32_t heads, float scale,
                               uint16_t* out, int32_t* status, cudaStream_t stream) {
  if (batch == 0 || t_cap == 0 || max_seqlen == 0) return cudaSuccess;
  CUtensorMap tm;
  const uint64_t row = static_cast<uint64_t>(3) * heads * attn::HD;
  if (encode_tmap_2d_bf16(&tm, qkv, row, static_cast<uint64_t>(t_cap), row * 2, attn::HD,
                          attn::KC) != 0)
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(attn::Smem);
  cudaError_t e = cudaFuncSetAttribute(attn::varlen_attn_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long ihs = static_cast<long long>(batch) * heads;
  if (ihs > 0x7fffffffLL) return cudaErrorInvalidValue;
  const long long cap = num_sms();
  const int grid = static_cast<int>(ihs < cap ? ihs : cap);
  const float scale_log2 = scale * 1.4426950408889634f;
  attn::varlen_attn_kernel<<<grid, attn::kThreads, smem, stream>>>(
      tm, cu, batch, max_seqlen, t_cap, heads, scale_log2, out, status);
  return cudaGetLastError();
}

}  // namespace dora
