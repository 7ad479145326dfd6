// Shared pieces of the two packed variable-length attention kernels
// (attn_tcgen05.cu: per-key-half accumulators, for images longer than 256
// tokens; attn_exchange_tcgen05.cu: one accumulator per query row, for images
// of up to 256 tokens): tile sizes, the walk over (image, head, query tile)
// units, the split of image-heads over the persistent CTAs, the tail-sized
// TMA loads and the softmax arithmetic on 32 keys.
#pragma once

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
constexpr int kDescRing = 8;    // step descriptors in flight
constexpr int kUnitRing = 4;    // unit descriptors in flight
constexpr int kThreads = 512;   // 16 warps: 128 registers a thread
constexpr int kSoftWarp0 = 4;   // softmax warps 4-11
constexpr int kEpiWarp0 = 12;   // epilogue warps 12-15
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleLog2 = 8.f;    // raise the reference maximum past 2^8
constexpr uint32_t kSleepNs = 200000;  // waiting threads sleep instead of spinning

// The four tensor maps of the packed qkv buffer: tiles of 128 rows, and
// 64-, 32- and 16-row boxes for the image tails.
struct QkvMaps {
  CUtensorMap m128, m64, m32, m16;
};

// Rows r16 (a multiple of 16, at most 128) of column block x from row y into
// dst: one 128-row box, or 64-, 32- and 16-row boxes stacked, so an image's
// tail is read rounded up to 16 rows instead of 128.  Every offset is a whole
// number of 8-row swizzle atoms, so the stacked boxes land exactly as one
// 128-row box would.
__device__ __forceinline__ void load_rows(const QkvMaps& mp, uint16_t* dst, uint64_t* bar, int x,
                                          int y, int r16) {
  if (r16 >= 128) {
    tma_load_2d(dst, &mp.m128, bar, x, y);
    return;
  }
  int off = 0;
  if (r16 & 64) {
    tma_load_2d(dst, &mp.m64, bar, x, y);
    off = 64;
  }
  if (r16 & 32) {
    tma_load_2d(dst + off * HD, &mp.m32, bar, x, y + off);
    off += 32;
  }
  if (r16 & 16) tma_load_2d(dst + off * HD, &mp.m16, bar, x, y + off);
}

// Rows of the image with bounds [b0, b1), clamped to the buffer (0 when its
// start lies outside); lo receives its first row.
__device__ __forceinline__ int clamp_rows(int b0, int b1, int t_cap, int& lo) {
  lo = b0;
  const int n = b1 - b0;
  if (lo < 0 || lo > t_cap) {
    lo = 0;
    return 0;
  }
  return n < 0 ? 0 : (n > t_cap - lo ? t_cap - lo : n);
}

// Rows of image `img`, clamped to the buffer (0 when its start lies outside).
__device__ __forceinline__ int image_rows(const int32_t* cu, int img, int t_cap, int& lo) {
  return clamp_rows(cu[img], cu[img + 1], t_cap, lo);
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

// Whole warp: the CTA's image-head range.  Image-head ih belongs to CTA
// floor(C(ih) * grid / total), C being the cost of the image-heads before it
// (image-major, head-minor order); CTA 0 also checks every image against the
// buffer and max_seqlen.  Each lane owns a contiguous block of images whose
// bounds it reads as one batch of independent loads, so the whole search
// costs about two memory round trips for any batch (a walk over the batch
// 32 images at a time, each chunk's loads waiting for the previous chunk's
// shuffles, took 4-9 us at 256 images).
__device__ inline void find_range(const int32_t* cu, int batch, int heads, int t_cap, int max_seqlen,
                                  int32_t* status, long long& ih_b, long long& ih_e) {
  const int lane = threadIdx.x & 31;
  const int per = (batch + 31) / 32;
  const int i0 = min(batch, lane * per), i1 = min(batch, i0 + per);
  long long mine = 0, c_last = 0;       // this lane's cost sum and its last image's cost
  for (int k0 = i0; k0 < i1; k0 += 8) {
    int bnd[9];
#pragma unroll
    for (int t = 0; t < 9; ++t) bnd[t] = (k0 + t <= i1) ? __ldg(cu + k0 + t) : 0;
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      if (k0 + t < i1) {
        int lo;
        c_last = ih_cost(clamp_rows(bnd[t], bnd[t + 1], t_cap, lo));
        mine += c_last;
        if (blockIdx.x == 0) {
          const int l0 = bnd[t], n = bnd[t + 1] - l0;
          if (l0 < 0 || l0 > t_cap || n > t_cap - l0 || n > max_seqlen)
            record_status(status, DORA_ERR_DEVICE_SEQLEN);
        }
      }
    }
  }
  long long incl = mine;                // one head's cost of the images up to this lane's last
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  const long long one_head = __shfl_sync(0xffffffffu, incl, 31);
  const long long nih = static_cast<long long>(batch) * heads;
  if (one_head == 0) {
    ih_b = ih_e = 0;
    return;
  }
  const long long total = one_head * heads, G = gridDim.x, bx = blockIdx.x;
  // first image-head with C * G >= x (nih if none): C grows along the order,
  // so it lies in the first lane whose last image-head reaches x, found by
  // that lane walking its own images (their bounds are in L1 by now)
  auto locate = [&](long long x) -> long long {
    const bool has = i0 < i1 && (heads * (incl - c_last) + (heads - 1) * c_last) * G >= x;
    const unsigned m = __ballot_sync(0xffffffffu, has);
    if (m == 0u) return nih;
    const int owner = __ffs(m) - 1;
    long long r = nih;
    if (lane == owner) {
      long long pre = incl - mine;      // one head's cost of the images before i0
      for (int i = i0; i < i1; ++i) {
        int lo;
        const long long c = ih_cost(image_rows(cu, i, t_cap, lo));
        const long long base = heads * pre * G;
        if (base >= x) {
          r = static_cast<long long>(i) * heads;
          break;
        }
        if (base + (heads - 1) * c * G >= x) {   // one of this image's heads (c > 0)
          r = static_cast<long long>(i) * heads + (x - base + c * G - 1) / (c * G);
          break;
        }
        pre += c;
      }
    }
    return __shfl_sync(0xffffffffu, r, owner);
  };
  ih_b = locate(bx * total);
  ih_e = (bx == G - 1) ? nih : locate((bx + 1) * total);
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

// p = 2^(s * scale_log2 - m) for 32 keys, summed into l and packed to bf16 in
// place: pair (2k, 2k+1) lands in a[k], whose S value is already consumed.
__device__ __forceinline__ void exp32_pack(uint32_t (&a)[32], float scale_log2, float neg_m,
                                           float& l) {
  const uint64_t sc = f2_pack(scale_log2, scale_log2), nm = f2_pack(neg_m, neg_m);
  uint64_t acc = f2_pack(0.f, 0.f);
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    float x0, x1;
    f2_unpack(f2_fma(f2_pack(__uint_as_float(a[e]), __uint_as_float(a[e + 1])), sc, nm), x0, x1);
    const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
    acc = f2_add(acc, f2_pack(p0, p1));
    a[e >> 1] = pack_bf16x2(p0, p1);
  }
  float l0, l1;
  f2_unpack(acc, l0, l1);
  l += l0 + l1;
}

// The packed half of a block, as the 16-column store operand.
__device__ __forceinline__ const uint32_t (&lo16(const uint32_t (&a)[32]))[16] {
  return *reinterpret_cast<const uint32_t(*)[16]>(&a[0]);
}

// One arrival for the whole warp, after every lane's prior tcgen05 accesses.
__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  tc_fence_before();
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(bar);
}

}  // namespace attn

// Encodes the four maps of a [t_cap, 3 * heads * 64] qkv buffer.
cudaError_t encode_qkv_maps(attn::QkvMaps* mp, const uint16_t* qkv, int32_t t_cap, int32_t heads);

// The kernel for images of up to 256 tokens (attn_exchange_tcgen05.cu).
cudaError_t launch_varlen_attn_exchange(const attn::QkvMaps& mp, const int32_t* cu,
                                        int32_t batch, int32_t max_seqlen, int32_t t_cap,
                                        int32_t heads, float scale_log2, uint16_t* out,
                                        int32_t* status, cudaStream_t stream);

}  // namespace dora
