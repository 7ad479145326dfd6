// Packed variable-length multi-head self-attention on tcgen05 tensor cores.
// For image i (rows [cu[i], cu[i+1]) of the packed buffer) and head h:
//     O = softmax(Q K^T * scale) V
// with no attention across images and no padding (Sec. 3.5 "Inference").
//
// Work unit = (image, head, 128-row query tile).  One persistent CTA per SM
// owns a contiguous range of units; consecutive query tiles of one image-head
// reuse the key/value tile already in shared memory, and the next image-head's
// tile is prefetched into the second stage.  Units alternate between two slots,
// each with its own softmax warpgroup and its own 256-column TMEM region, so
// one slot's softmax overlaps the other slot's MMAs and loads.
//   warp 0     TMA: Q tile per slot, K and V tiles of up to 256 keys (2 stages).
//   warp 1     MMA: S = Q K^T (M=128, N=keys rounded to 16, K=64) into the
//              slot's region; O = P V (M=128, N=64) with P read from TMEM, into
//              region + [128, 192).  S of a step is issued before the PV of the
//              previous step.
//   warps 2-9  two softmax warpgroups, one thread per query row (TMEM lane):
//              row max, exp2, row sum; P packed to bf16 and written back over
//              the S columns already consumed (tcgen05.st); O of every key
//              tile folded into fp32 registers with the online-softmax rescale.
// Images up to 256 tokens take one key tile; longer ones take several, with
// the online rescale.  Rows past the image skip the exponentials; keys past it
// are masked, and V rows past it are zeroed in shared memory so stale data
// cannot leak through 0 * NaN.
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
constexpr int KVT = 256;        // keys per key tile
constexpr int BOX = 128;        // rows per TMA box
constexpr int HD = 64;
constexpr int kSlots = 2;       // units in flight: one per softmax warpgroup
constexpr int kThreads = 64 + kSlots * 128;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kRegion = 256;   // TMEM columns per slot: S, then P over [0,128)
constexpr uint32_t kTmemO = 128;    // O of a slot at region + 128

struct Smem {
  uint16_t q[kSlots][BQ * HD];  // 2 x 16 KB, one per slot
  uint16_t k[2][KVT * HD];      // 2 x 32 KB key tiles
  uint16_t v[2][KVT * HD];      // 2 x 32 KB value tiles
  uint64_t q_full[kSlots];
  uint64_t q_empty[kSlots];
  uint64_t kv_full[2];
  uint64_t kv_empty[2];
  uint64_t s_full[kSlots];
  uint64_t p_full[kSlots];
  uint64_t o_full[kSlots];
  uint64_t r_free[kSlots];      // a slot's TMEM region read out by its warpgroup
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int q_issued[kSlots];
  int q_used[kSlots];
  int kv_issued;
  int kv_used;
};

// Decoded work unit: image, head, query tile, first row and token count.
struct Unit {
  int img, head, qt, lo, n;
};

struct Units {
  const int32_t* cu;
  int heads, qtiles, t_cap;
  __device__ __forceinline__ Unit get(long u) const {
    Unit r;
    const long per_img = static_cast<long>(heads) * qtiles;
    r.img = static_cast<int>(u / per_img);
    const int rem = static_cast<int>(u - static_cast<long>(r.img) * per_img);
    r.head = rem / qtiles;
    r.qt = rem - r.head * qtiles;
    r.lo = cu[r.img];
    int n = cu[r.img + 1] - r.lo;
    if (r.lo < 0 || r.lo > t_cap || n > t_cap - r.lo)
      n = (r.lo < 0 || r.lo > t_cap) ? 0 : t_cap - r.lo;   // clamp to the buffer
    r.n = n;
    return r;
  }
  __device__ __forceinline__ static bool valid(const Unit& x) { return x.qt * BQ < x.n; }
  __device__ __forceinline__ static int kv_tiles(const Unit& x) { return (x.n + KVT - 1) / KVT; }
};

// Key/value tile bookkeeping every role replays identically: a unit reuses the
// tile of the previous valid unit of the CTA when both are the same image and
// head and the image fits one tile; otherwise each of its key tiles is a new
// load into stage (load count & 1).
struct KvTrack {
  int img = -1, head = -1, nkv = 0, loads = 0;
  __device__ __forceinline__ bool reuse(const Unit& x, int nkv_x) {
    const bool r = nkv_x == 1 && nkv == 1 && x.img == img && x.head == head;
    img = x.img;
    head = x.head;
    nkv = nkv_x;
    return r;
  }
};

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
  const int qtiles = (max_seqlen + BQ - 1) / BQ;
  const Units U{cu, heads, qtiles, t_cap};
  const long total = static_cast<long>(batch) * heads * qtiles;
  const long u_begin = total * blockIdx.x / gridDim.x;
  const long u_end = total * (blockIdx.x + 1) / gridDim.x;

  if (threadIdx.x == 0) {
    // device-side check of the boundaries, images spread over the CTAs
    for (int i = blockIdx.x; i < batch; i += gridDim.x) {
      const int lo = cu[i], n = cu[i + 1] - lo;
      if (lo < 0 || lo > t_cap || n > t_cap - lo || n > max_seqlen)
        record_status(status, DORA_ERR_DEVICE_SEQLEN);
    }
    for (int i = 0; i < kSlots; ++i) {
      mbar_init(&s.q_full[i], 1);
      mbar_init(&s.q_empty[i], 1);
      mbar_init(&s.s_full[i], 1);
      mbar_init(&s.p_full[i], 128);
      mbar_init(&s.o_full[i], 1);
      mbar_init(&s.r_free[i], 128);
      s.q_issued[i] = s.q_used[i] = 0;
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.kv_full[i], 1);
      mbar_init(&s.kv_empty[i], 1);
    }
    mbar_init(&s.drain, 1);
    s.abort_flag = 0;
    s.kv_issued = s.kv_used = 0;
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
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int qn[kSlots] = {0, 0};
      int k = 0;                 // valid-unit index in this CTA; slot = k & 1
      KvTrack kv;
      bool ok = true;
      for (long u = u_begin; ok && u < u_end; ++u) {
        const Unit x = U.get(u);
        if (!Units::valid(x)) continue;
        const int slot = k++ & 1;
        const int nkv = Units::kv_tiles(x);
        const bool reuse = kv.reuse(x, nkv);
        if (!mbar_wait(&s.q_empty[slot], (qn[slot] & 1) ^ 1, abort)) break;
        mbar_arrive_expect_tx(&s.q_full[slot], BQ * HD * 2);
        tma_load_2d(s.q[slot], &tm, &s.q_full[slot], x.head * HD, x.lo + x.qt * BQ);
        ++qn[slot];
        if (reuse) continue;
        for (int j = 0; j < nkv; ++j) {
          const int st = kv.loads & 1;
          const int valid = min(KVT, x.n - j * KVT);
          const int boxes = (valid + BOX - 1) / BOX;
          if (!mbar_wait(&s.kv_empty[st], ((kv.loads >> 1) & 1) ^ 1, abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&s.kv_full[st], boxes * 2 * BOX * HD * 2);
          for (int b = 0; b < boxes; ++b) {
            const int row = x.lo + j * KVT + b * BOX;
            tma_load_2d(s.k[st] + b * BOX * HD, &tm, &s.kv_full[st], dim + x.head * HD, row);
            tma_load_2d(s.v[st] + b * BOX * HD, &tm, &s.kv_full[st], 2 * dim + x.head * HD, row);
          }
          ++kv.loads;
        }
      }
      s.q_issued[0] = qn[0];
      s.q_issued[1] = qn[1];
      s.kv_issued = kv.loads;
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    // Per step (unit, key tile): S into the slot's region, then the PV of the
    // previous step, so one warpgroup's softmax overlaps the other's MMAs.
    if (lane == 0) {
      constexpr uint32_t id_o = idesc_bf16(BQ, HD, true);
      int qn[kSlots] = {0, 0};
      int steps[kSlots] = {0, 0};     // S issued per slot
      int pvs[kSlots] = {0, 0};       // PV issued per slot
      int kfull = 0;                  // key-tile loads waited for
      int k = 0;
      KvTrack kv;
      bool ok = true;
      // the step whose PV is still to be issued
      bool pend = false;
      int p_slot = 0, p_nm = 0, p_st = 0;
      bool p_release = false;
      auto issue_pv = [&]() -> bool {
        if (!mbar_wait(&s.p_full[p_slot], pvs[p_slot] & 1, abort)) return false;
        tc_fence_after();
        const uint32_t region = tmem + static_cast<uint32_t>(p_slot) * kRegion;
        const uint32_t vbase = smem_u32(s.v[p_st]);
        for (int kk = 0; kk < p_nm / 16; ++kk) {
          const uint64_t vd = sdesc_sw128(vbase + static_cast<uint32_t>(kk * 16 * 128), 1024, 1024);
          mma_bf16_ts(region + kTmemO, region + static_cast<uint32_t>(8 * kk), vd, id_o,
                      kk > 0 ? 1u : 0u);
        }
        mma_commit(&s.o_full[p_slot]);
        if (p_release) mma_commit(&s.kv_empty[p_st]);
        ++pvs[p_slot];
        pend = false;
        return true;
      };
      for (long u = u_begin; ok && u < u_end; ++u) {
        const Unit x = U.get(u);
        if (!Units::valid(x)) continue;
        const int slot = k++ & 1;
        const int nkv = Units::kv_tiles(x);
        const bool reuse = kv.reuse(x, nkv);
        bool last_use = true;       // does no later unit of the CTA reuse this tile?
        if (nkv == 1) {
          for (long w = u + 1; w < u_end; ++w) {
            const Unit y = U.get(w);
            if (!Units::valid(y)) continue;
            last_use = !(y.img == x.img && y.head == x.head);
            break;
          }
        }
        if (!mbar_wait(&s.q_full[slot], qn[slot] & 1, abort)) break;
        const uint64_t qd = sdesc_sw128(smem_u32(s.q[slot]), 16, 1024);
        for (int j = 0; j < nkv; ++j) {
          const int valid = min(KVT, x.n - j * KVT);
          const int nm = (valid + 15) & ~15;
          const int st = (reuse ? kv.loads - 1 : kv.loads) & 1;
          if (!reuse) {
            if (!mbar_wait(&s.kv_full[st], (kv.loads >> 1) & 1, abort)) {
              ok = false;
              break;
            }
            ++kv.loads;
            ++kfull;
          }
          if (pend && p_slot == slot && !issue_pv()) {   // same region: PV first
            ok = false;
            break;
          }
          if (steps[slot] > 0 && !mbar_wait(&s.r_free[slot], (steps[slot] - 1) & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t region = tmem + static_cast<uint32_t>(slot) * kRegion;
          const uint64_t kd = sdesc_sw128(smem_u32(s.k[st]), 16, 1024);
          const uint32_t id_s = idesc_bf16(BQ, nm, false);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            mma_bf16_ss(region, qd + 2 * kk, kd + 2 * kk, id_s, kk > 0 ? 1u : 0u);
          mma_commit(&s.s_full[slot]);
          if (j == nkv - 1) mma_commit(&s.q_empty[slot]);
          ++steps[slot];
          if (pend && !issue_pv()) {                      // other slot's PV
            ok = false;
            break;
          }
          pend = true;
          p_slot = slot;
          p_nm = nm;
          p_st = st;
          p_release = nkv > 1 || last_use;
        }
        ++qn[slot];
      }
      if (ok && pend) issue_pv();
      s.q_used[0] = qn[0];
      s.q_used[1] = qn[1];
      s.kv_used = kfull;
      mma_commit(&s.drain);
      mbar_wait_limited(&s.drain, 0, kWaitLimitNs);
    }
  } else {
    // ---------------- softmax warpgroups: thread <-> query row r ----------------
    const int wg = (warp - 2) >> 2;                 // slot served by this warpgroup
    const int quarter = warp & 3;
    const int r = quarter * 32 + lane;
    const uint32_t region = tmem + static_cast<uint32_t>(wg) * kRegion;
    const uint32_t lane_sel = static_cast<uint32_t>(quarter * 32) << 16;
    int g = 0, k = 0;
    KvTrack kv;
    bool ok = true;
    for (long u = u_begin; ok && u < u_end; ++u) {
      const Unit x = U.get(u);
      if (!Units::valid(x)) continue;
      const int slot = k++ & 1;
      const int nkv = Units::kv_tiles(x);
      const bool reuse = kv.reuse(x, nkv);
      if (slot != wg) {
        if (!reuse) kv.loads += nkv;                 // keep the load count in step
        continue;
      }
      const int q_rows = min(BQ, x.n - x.qt * BQ);
      const bool row_live = r < q_rows;
      const bool warp_live = quarter * 32 < q_rows;      // warp-uniform
      (void)row_live;
      float o[HD];
#pragma unroll
      for (int d = 0; d < HD; ++d) o[d] = 0.f;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < nkv; ++j, ++g) {
        const int valid = min(KVT, x.n - j * KVT);
        const int nm = (valid + 15) & ~15;
        const int nc = (valid + 31) & ~31;
        const int st = (reuse ? kv.loads - 1 : kv.loads) & 1;
        const int load_idx = reuse ? -1 : kv.loads;
        if (!reuse) ++kv.loads;
        if (!mbar_wait_warp(&s.s_full[wg], g & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float alpha = 1.f;
        uint32_t pk[16];
        if (warp_live) {
          // Keys [valid, nc) of the last chunk are masked to -inf; rows past the
          // image are computed like the others (they only feed O rows that are
          // never stored), which keeps the inner loops free of predicates.
          const int nch = nc >> 5;
          const int rem = valid & 31;                  // live keys of a partial last chunk
          float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          for (int ch = 0; ch < nch; ++ch) {
            uint32_t a[32];
            tmem_ld32(region + lane_sel + static_cast<uint32_t>(ch * 32), a);
            tmem_ld_wait();
            if (rem != 0 && ch + 1 == nch) {
#pragma unroll
              for (int e = 0; e < 32; ++e)
                if (e >= rem) a[e] = __float_as_uint(-INFINITY);
            }
#pragma unroll
            for (int e = 0; e < 32; ++e) m4[e & 3] = fmaxf(m4[e & 3], __uint_as_float(a[e]));
          }
          const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
          const float m_new = fmaxf(m_run, mx * scale_log2);
          const float neg_m = -m_new;
          alpha = ex2_approx(m_run - m_new);
          float l4[4] = {0.f, 0.f, 0.f, 0.f};
          for (int ch = 0; ch < nch; ++ch) {
            uint32_t a[32];
            tmem_ld32(region + lane_sel + static_cast<uint32_t>(ch * 32), a);
            tmem_ld_wait();
            if (rem != 0 && ch + 1 == nch) {
#pragma unroll
              for (int e = 0; e < 32; ++e)
                if (e >= rem) a[e] = __float_as_uint(-INFINITY);
            }
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              const float p0 = ex2_approx(fmaf(__uint_as_float(a[e]), scale_log2, neg_m));
              const float p1 = ex2_approx(fmaf(__uint_as_float(a[e + 1]), scale_log2, neg_m));
              l4[e & 3] += p0;
              l4[(e + 1) & 3] += p1;
              pk[e >> 1] = pack_bf16x2(p0, p1);
            }
            // P columns [16 ch, 16 ch + 16) lie in S columns this thread already read
            tmem_st16(region + lane_sel + static_cast<uint32_t>(ch * 16), pk);
          }
          l_run = l_run * alpha + ((l4[0] + l4[1]) + (l4[2] + l4[3]));
          m_run = m_new;
        } else {
          // the whole warp is past the image: zero P rows keep O finite
#pragma unroll
          for (int e = 0; e < 16; ++e) pk[e] = 0u;
          for (int c = 0; c < nc; c += 32)
            tmem_st16(region + lane_sel + static_cast<uint32_t>(c >> 1), pk);
        }
        tmem_st_wait();
        // Zero V rows [valid, nm) of a key tile this unit loaded: the PV product
        // reads them against zero P columns.  Wait for the load first so that
        // it cannot overwrite the zeros; later users of the tile issue their
        // PV after this one.
        if (load_idx >= 0 && valid < nm) {
          const bool kv_ok = mbar_wait(&s.kv_full[st], (load_idx >> 1) & 1, abort);
          if (!__all_sync(0xffffffffu, kv_ok)) {
            ok = false;
            break;
          }
          for (int vr = r; vr < nm; vr += BQ) {
            if (vr < valid) continue;
            uint4* vrow = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(s.v[st]) + vr * 128);
#pragma unroll
            for (int qd = 0; qd < 8; ++qd) vrow[qd] = make_uint4(0u, 0u, 0u, 0u);
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&s.p_full[wg]);
        if (!mbar_wait_warp(&s.o_full[wg], g & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < HD; c += 32) {
          uint32_t orr[32];
          tmem_ld32(region + lane_sel + kTmemO + static_cast<uint32_t>(c), orr);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[c + e] = o[c + e] * alpha + __uint_as_float(orr[e]);
        }
        tc_fence_before();
        mbar_arrive(&s.r_free[wg]);
      }
      if (!ok) break;
      if (row_live) {
        const float inv = 1.0f / l_run;
        uint4* dst = reinterpret_cast<uint4*>(
            out + static_cast<size_t>(x.lo + x.qt * BQ + r) * dim + x.head * HD);
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
      // let every TMA load that was issued but never consumed land first
      for (int sl = 0; sl < kSlots; ++sl)
        for (int c = s.q_used[sl]; c < s.q_issued[sl]; ++c)
          mbar_wait_limited(&s.q_full[sl], c & 1, 100ull * 1000 * 1000);
      for (int c = s.kv_used; c < s.kv_issued; ++c)
        mbar_wait_limited(&s.kv_full[c & 1], (c >> 1) & 1, 100ull * 1000 * 1000);
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
                          attn::BOX) != 0)
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(attn::Smem);
  cudaError_t e = cudaFuncSetAttribute(attn::varlen_attn_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long units = static_cast<long>(batch) * heads * ((max_seqlen + attn::BQ - 1) / attn::BQ);
  const long cap = num_sms();
  const int grid = static_cast<int>(units < cap ? units : cap);
  const float scale_log2 = scale * 1.4426950408889634f;
  attn::varlen_attn_kernel<<<grid, attn::kThreads, smem, stream>>>(
      tm, cu, batch, max_seqlen, t_cap, heads, scale_log2, out, status);
  return cudaGetLastError();
}

}  // namespace dora
