// elementwise.cu -- the element-wise parts of AQD's integer inference path:
//   * requant (Eq. 6 bias + Eq. 2 fixed-point rescale and clip) of an int32 tensor,
//   * the integer skip add of Eq. 7 with Eq. 8's dyadic factor (optionally reading the
//     skip through a nearest 2x upsample, the FPN top-down add),
//   * max-pooling directly on codes (Sec. 3.2.4),
//   * code packing / unpacking and the one-time weight preparation.
// An int32 input on contiguous rows takes the staged kernel (bulk async copies of whole
// pixel rows into shared memory, consumer warps with per-lane channel constants); other int32
// inputs the lane kernel (kV channels per lane, direct loads); packed-code inputs the group
// kernels (one thread per pixel's 32-channel group: whole packed groups per load and store).
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace aqd {
namespace elt {

constexpr int kThreads = 256;
constexpr int kLanePix = 6;  // pixels per warp step of the element-wise lane kernel (table form)

__device__ __forceinline__ void load_vals(const uint8_t* row, int bits, int c, int ch0, bool is_signed,
                                          int32_t v[32]) {
  if (bits == 32 && (c % 32) == 0) {
    const int4* p = reinterpret_cast<const int4*>(row + 4 * (int64_t)ch0);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int4 x = p[q];
      v[4 * q] = x.x; v[4 * q + 1] = x.y; v[4 * q + 2] = x.z; v[4 * q + 3] = x.w;
    }
  } else if (bits != 32 && (bits != 8 || (c % 32) == 0)) {
    unpack_group_vals(row + (ch0 >> 5) * group_bytes(bits), bits, is_signed, v);
  } else {
#pragma unroll 4
    for (int i = 0; i < 32; ++i) v[i] = (ch0 + i < c) ? read_code(row, ch0 + i, bits, is_signed) : 0;
  }
}

__device__ __forceinline__ void store_vals(uint8_t* row, int bits, int c, int ch0, const int32_t v[32]) {
  if (bits == 32) {
    int32_t* p = reinterpret_cast<int32_t*>(row) + ch0;
    if ((c % 32) == 0) {
#pragma unroll
      for (int q = 0; q < 8; ++q)
        reinterpret_cast<int4*>(p)[q] = make_int4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    } else {
      for (int i = 0; i < 32; ++i)
        if (ch0 + i < c) p[i] = v[i];
    }
  } else if (bits == 8 && (c % 32) != 0) {
    for (int i = 0; i < 32; ++i)
      if (ch0 + i < c) row[ch0 + i] = (uint8_t)v[i];
  } else {
    uint32_t g[8];
    pack_group_vals(v, bits, g);
    store_group(row + (ch0 >> 5) * group_bytes(bits), g, bits);
  }
}

template <bool kHasSkip>
__global__ void __launch_bounds__(kThreads) eltwise_kernel(const EltArgs a) {
  const int groups = (a.c + 31) / 32;
  const int64_t total = (int64_t)a.n * a.h * a.w * groups;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= total) return;
  const int64_t pix = t / groups;
  const int ch0 = (int)(t - pix * groups) * 32;
  int32_t av[32];
  load_vals(a.a + pix * a.a_row_bytes, a.a_bits, a.c, ch0, a.a_bits == 32, av);
  int32_t sv[32];
  if (kHasSkip) {
    const int64_t hw = (int64_t)a.h * a.w;
    const int64_t img = pix / hw;
    const int64_t rem = pix - img * hw;
    const int hh = (int)(rem / a.w), ww = (int)(rem - (rem / a.w) * a.w);
    const int64_t sp = (img * a.b_h + hh / a.upsample) * a.b_w + ww / a.upsample;
    load_vals(a.b + sp * a.b_row_bytes, a.b_bits, a.c, ch0, a.b_bits == 32, sv);
  }
  int32_t out[32];
#pragma unroll 4
  for (int i = 0; i < 32; ++i) {
    const int ch = ch0 + i;
    EpiChan ec{};
    if (ch < a.c) {
      const int64_t idx = (int64_t)a.level * a.c + ch;
      ec.bias = a.bias ? a.bias[idx] : 0;
      if (a.y_bits != 32) { ec.m0 = a.m0[idx]; ec.r = (int8_t)(31 + a.shift[idx]); }
      if (kHasSkip) { ec.c = a.skip_c[idx]; ec.d = a.skip_d[idx]; }
    }
    out[i] = epilogue<kHasSkip>(av[i], kHasSkip ? sv[i] : 0, ec, a.scale_main, a.y_bits);
  }
  store_vals(a.y + pix * a.y_row_bytes, a.y_bits, a.c, ch0, out);
}

// The same operation for whole 32-channel groups (c % 32 == 0), with coalesced traffic and
// broadcast table reads. A block takes spans of 256 consecutive (pixel, group) units; since
// c % 32 == 0, unit u's input bytes sit at u * (group bytes) and its output bytes likewise,
// so a span is one contiguous range of each. All threads copy the span's input into shared
// memory with consecutive 16-byte loads, each thread works on one unit, and the results
// leave the same way. When the group count G divides 256, the threads of a warp take units
// of one channel group (pixel = lane), so the per-channel constants are read as broadcasts.
// When there is no skip, the output is codes and every channel has R = 31 + shift >= 33,
// Eq. 6 -> Eq. 2 runs in 32-bit form: u = sat32(a + bias) by a saturating add, and
// rhu(u * M0, R) = (mulhi(u, M0) + 2^(R-33)) >> (R-32) (the low product word cannot carry
// into the rounded result); the clip is one min.relu. Otherwise each element takes the
// int64 epilogue as written.
constexpr int kTabChannels = 512;  // channels whose constants fit the static shared table

__device__ __forceinline__ int32_t sat_add32(int32_t a, int32_t b) {
  int32_t r;
  asm("add.sat.s32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Bytes of one (pixel, 32-channel group) unit at `bits` (4 * bits, or 128 for int32).
__device__ __forceinline__ int unit_bytes(int bits) { return bits == 32 ? 128 : group_bytes(bits); }

// 16-byte slot q of int32 unit u in the staging buffer, rotated by the unit's key so that
// eight lanes touching eight units, or eight slots of one unit, use eight different bank
// groups
__device__ __forceinline__ int stage_slot(int u, int q, int key) { return u * 8 + (q ^ key); }

template <bool kHasSkip>
__global__ void __launch_bounds__(kThreads, 3) eltwise_group_kernel(const EltArgs a) {
  __shared__ int4 stage[kThreads * 8];   // 32 KB: one span of int32 units (or of smaller ones)
  __shared__ EpiChan tab[kTabChannels];  // 8 KB
  int fast = (!kHasSkip && a.y_bits != 32) ? 1 : 0;
  for (int ch = threadIdx.x; ch < a.c; ch += kThreads) {
    const int64_t idx = (int64_t)a.level * a.c + ch;
    EpiChan ec{};
    ec.bias = a.bias ? a.bias[idx] : 0;
    if (a.y_bits != 32) {
      ec.m0 = a.m0[idx];
      ec.r = (int8_t)(31 + a.shift[idx]);
      if (ec.r < 33) fast = 0;
    }
    if (kHasSkip) { ec.c = a.skip_c[idx]; ec.d = a.skip_d[idx]; }
    tab[ch] = ec;
  }
  fast = __syncthreads_and(fast);  // also publishes the table
  const int qmax = (1 << (a.y_bits & 15)) - 1;
  const int G = a.c / 32;
  const int64_t total = (int64_t)a.n * a.h * a.w * G;
  const int tid = threadIdx.x;
  // this thread's unit within a span, and the staging key of a unit: (unit / G) & 7 when a
  // warp's lanes take consecutive pixels of one group, else unit & 7
  const bool by_group = (kThreads % G) == 0;  // G is then a power of two
  const int lg = by_group ? __ffs(G) - 1 : 0;
  const int per_group = kThreads / G;
  const int j = by_group ? (tid % per_group) * G + tid / per_group : tid;
  auto key = [&](int u) { return by_group ? (u >> lg) & 7 : u & 7; };
  const int gin = unit_bytes(a.a_bits), gout = unit_bytes(a.y_bits);
  uint8_t* sbytes = reinterpret_cast<uint8_t*>(stage);
  for (int64_t base = (int64_t)blockIdx.x * kThreads; base < total; base += (int64_t)gridDim.x * kThreads) {
    const int nu = (int)(total - base < kThreads ? total - base : kThreads);
    const bool mine = j < nu;
    const int64_t t = base + j;
    // pixels number below 2^31 (checked on the host), units usually too: 32-bit division then
    const int pix = total <= 0x7FFFFFFF ? (int)t / G : (int)(t / G);
    const int ch0 = (int)(t - (int64_t)pix * G) * 32;
    int32_t v[32];
    if (a.a_bits == 32) {
      const int4* src = reinterpret_cast<const int4*>(a.a) + base * 8;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int k = tid + i * kThreads;
        if (k < nu * 8) stage[stage_slot(k >> 3, k & 7, key(k >> 3))] = __ldg(src + k);
      }
      __syncthreads();
      if (mine) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int4 x = stage[stage_slot(j, q, key(j))];
          v[4 * q] = x.x; v[4 * q + 1] = x.y; v[4 * q + 2] = x.z; v[4 * q + 3] = x.w;
        }
      }
    } else {
      // packed codes: the span's bytes as 16-byte chunks (a multiple of 4 bytes when partial)
      const int nbytes = nu * gin;
      const uint8_t* src = a.a + base * gin;
      for (int k = tid; k * 16 < nbytes; k += kThreads) {
        if (k * 16 + 16 <= nbytes) {
          stage[k] = __ldg(reinterpret_cast<const int4*>(src) + k);
        } else {
          for (int b = k * 16; b < nbytes; b += 4)
            reinterpret_cast<uint32_t*>(sbytes)[b / 4] = __ldg(reinterpret_cast<const uint32_t*>(src) + b / 4);
        }
      }
      __syncthreads();
      if (mine) unpack_group_vals(sbytes + j * gin, a.a_bits, false, v);
    }
    if (mine) {
      if (!kHasSkip && fast) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const EpiChan ec = tab[ch0 + i];
          const int32_t u = sat_add32(v[i], ec.bias);
          v[i] = __vimin_s32_relu((__mulhi(u, ec.m0) + (1 << (ec.r - 33))) >> (ec.r - 32), qmax);
        }
      } else {
        int32_t sv[32];
        if (kHasSkip) {
          const int hw = a.h * a.w;
          const int img = pix / hw;
          const int rem = pix - img * hw;
          const int hh = rem / a.w, ww = rem - (rem / a.w) * a.w;
          const int64_t sp = ((int64_t)img * a.b_h + hh / a.upsample) * a.b_w + ww / a.upsample;
          load_vals(a.b + sp * a.b_row_bytes, a.b_bits, a.c, ch0, a.b_bits == 32, sv);
        }
#pragma unroll 4
        for (int i = 0; i < 32; ++i)
          v[i] = epilogue<kHasSkip>(v[i], kHasSkip ? sv[i] : 0, tab[ch0 + i], a.scale_main, a.y_bits);
      }
    }
    __syncthreads();  // every thread has read its unit from the staging buffer
    if (a.y_bits == 32) {
      if (mine) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          stage[stage_slot(j, q, key(j))] = make_int4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      }
      __syncthreads();
      int4* dst = reinterpret_cast<int4*>(a.y) + base * 8;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int k = tid + i * kThreads;
        if (k < nu * 8) dst[k] = stage[stage_slot(k >> 3, k & 7, key(k >> 3))];
      }
    } else {
      if (mine) {
        uint32_t g[8];
        pack_group_vals(v, a.y_bits, g);
        uint32_t* d = reinterpret_cast<uint32_t*>(sbytes + (int64_t)j * gout);
        for (int w = 0; w < gout / 4; ++w) d[w] = g[w];
      }
      __syncthreads();
      const int nbytes = nu * gout;
      uint8_t* dst = a.y + base * gout;
      for (int k = tid; k * 16 < nbytes; k += kThreads) {
        if (k * 16 + 16 <= nbytes) {
          reinterpret_cast<int4*>(dst)[k] = stage[k];
        } else {
          for (int b = k * 16; b < nbytes; b += 4)
            reinterpret_cast<uint32_t*>(dst)[b / 4] = reinterpret_cast<const uint32_t*>(sbytes)[b / 4];
        }
      }
    }
    __syncthreads();  // the staging buffer is free for the next span
  }
}

// Requant (Eq. 6 + Eq. 2) and the integer skip add (Eq. 7/8, then Eq. 2) of an int32 tensor
// with kV consecutive channels per lane (c % (32 kV) == 0): lane l of a warp owns channels
// 32 kV g + kV l .. + kV - 1 of one block g of 32 kV channels for the whole launch, so their
// constants stay in registers, and the warp's load of one pixel's block is 128 kV contiguous
// bytes (one 4 kV-byte load per lane). A packed skip code tensor gives each lane one 32-bit
// word per pixel (its kV channels lie in one word). The packed output is assembled across
// lanes: output word w of a 32-channel group holds its channels [w q, (w + 1) q), q = 32 / bits,
// channel i at bit 8 (i % 4) + bits ((i % q) / 4); a lane's channels land in one word, so an OR
// over the lanes of a word builds it and one of them stores it. Warps of one block take every
// warps_per_block-th pixel, kPix per step with their loads issued first.
//
// Each block picks one of two exact forms of the epilogue once, from the constants of all c
// channels:
//  - table: every rescale has R = 31 + shift >= 33, where rhu(u M0, R) equals
//    (mulhi(u, M0) + 2^(R-33)) >> (R-32); and, with a skip, the main path is not rescaled
//    (Eq. 7 with the skip rescaled), the skip codes are at most 8 bits wide and the block's
//    shared-memory table T[s][ch] = bias + rhu(s c, d) (built in int64 for every code s) fits
//    int32. Then Eq. 6 + Eq. 7 is sat32(a + T[s][ch]), one saturating 32-bit add; without a
//    skip it is sat32(a + bias). Table column of channel ch: ch + ch / 32, so the lanes of a
//    warp, whose channels step by kV, read 32 distinct banks whatever their codes.
//  - general: Eq. 6 -> Eq. 7 -> Eq. 2 in int64 exactly as defined (the shared epilogue).
template <int kV>
struct LaneVec;
template <> struct LaneVec<1> { typedef int32_t T; };
template <> struct LaneVec<2> { typedef int2 T; };
template <> struct LaneVec<4> { typedef int4 T; };
template <int kV>
__device__ __forceinline__ void ld_lane(const void* p, int32_t (&v)[kV]) {
  const typename LaneVec<kV>::T x = __ldg(reinterpret_cast<const typename LaneVec<kV>::T*>(p));
  if constexpr (kV == 1) { v[0] = x; }
  else if constexpr (kV == 2) { v[0] = x.x; v[1] = x.y; }
  else { v[0] = x.x; v[1] = x.y; v[2] = x.z; v[3] = x.w; }
}
template <int kV>
__device__ __forceinline__ void st_lane(void* p, const int32_t (&v)[kV]) {
  if constexpr (kV == 1) *reinterpret_cast<int32_t*>(p) = v[0];
  else if constexpr (kV == 2) *reinterpret_cast<int2*>(p) = make_int2(v[0], v[1]);
  else *reinterpret_cast<int4*>(p) = make_int4(v[0], v[1], v[2], v[3]);
}
// sat32(x + y) of two int32 values
__device__ __forceinline__ int32_t add_sat_s32(int32_t x, int32_t y) {
  int32_t r;
  asm("add.sat.s32 %0, %1, %2;" : "=r"(r) : "r"(x), "r"(y));
  return r;
}

// Per-lane geometry shared by both forms.
struct LaneGeo {
  int64_t first, npix, stride;  // first pixel, pixel count, pixel stride of a step
  int wpb, ch0, lane;
  bool same_grid;
};

template <bool kSkip, int kSkipBits>
__device__ __forceinline__ int64_t skip_pixel(const EltArgs& a, const LaneGeo& g, int64_t pix) {
  if (g.same_grid) return pix;
  const int64_t hw = (int64_t)a.h * a.w;
  const int64_t img = pix / hw, rem = pix - img * hw;
  const int hh = (int)(rem / a.w), ww = (int)(rem - (rem / a.w) * a.w);
  return (img * a.b_h + hh / a.upsample) * a.b_w + ww / a.upsample;
}

// OR this lane's word contribution with the other lanes of its output word and store it
template <int kOut, int kV>
__device__ __forceinline__ void store_codes(const EltArgs& a, const LaneGeo& g, int64_t pix, uint32_t v) {
  constexpr int q = 32 / kOut;
  constexpr int span = (q / 4 * 4 + kV - 1) / kV;  // lanes per output word
#pragma unroll
  for (int off = 1; off < span; off <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, off);
  const int i0 = g.ch0 & 31;
  if (pix < g.npix && g.lane % span == 0)
    reinterpret_cast<uint32_t*>(a.y + pix * a.y_row_bytes + (g.ch0 >> 5) * group_bytes(kOut))[i0 / q] = v;
}

// bit position of channel i (of a 32-channel group) in its packed word
template <int kBits>
__device__ __forceinline__ int code_pos(int i) {
  constexpr int q = 32 / kBits;
  return 8 * (i & 3) + kBits * ((i % q) >> 2);
}

template <bool kSkip, int kOut, int kSkipBits, int kV>
__device__ __forceinline__ void lane_fast(const EltArgs& a, const LaneGeo& g, const int32_t (&b)[kV],
                                          const int32_t (&m0)[kV], const int32_t (&rnd)[kV],
                                          const int32_t (&sh)[kV], const int32_t* tab, int tstride) {
  constexpr int kPix = kLanePix;
  const int i0 = g.ch0 & 31;
  // channel i0 + k of a packed word sits at bit base + 8 k (kV divides 4 and i0): shift the
  // word once per pixel instead of once per channel
  const int sbase = kSkip && kSkipBits <= 8 ? code_pos<kSkip && kSkipBits <= 8 ? kSkipBits : 8>(i0) : 0;
  const int obase = kOut != 32 ? code_pos<kOut != 32 ? kOut : 8>(i0) : 0;
  for (int64_t p0 = g.first; p0 < g.npix; p0 += g.stride) {
    int32_t av[kPix][kV];
    uint32_t sw[kPix];
#pragma unroll
    for (int u = 0; u < kPix; ++u) {
      const int64_t pix = p0 + (int64_t)u * g.wpb;
#pragma unroll
      for (int k = 0; k < kV; ++k) av[u][k] = 0;
      sw[u] = 0;
      if (pix >= g.npix) continue;
      ld_lane<kV>(reinterpret_cast<const int32_t*>(a.a) + pix * a.c + g.ch0, av[u]);
      if constexpr (kSkip && kSkipBits <= 8) {
        const uint8_t* srow = a.b + skip_pixel<kSkip, kSkipBits>(a, g, pix) * a.b_row_bytes;
        sw[u] = __ldg(reinterpret_cast<const uint32_t*>(srow + (g.ch0 >> 5) * group_bytes(kSkipBits)) +
                      i0 / (32 / kSkipBits)) >> sbase;
      }
    }
#pragma unroll
    for (int u = 0; u < kPix; ++u) {
      const int64_t pix = p0 + (int64_t)u * g.wpb;
      int32_t y[kV];
      uint32_t v = 0;
#pragma unroll
      for (int k = 0; k < kV; ++k) {
        int32_t bk = b[k];
        if constexpr (kSkip && kSkipBits <= 8) {
          const int s = (int)((sw[u] >> (8 * k)) & ((1u << kSkipBits) - 1u));
          bk = tab[s * tstride + b[k]];  // b[k]: this channel's table column
        }
        const int32_t uu = add_sat_s32(av[u][k], bk);
        if constexpr (kOut == 32) {
          y[k] = uu;
        } else {
          y[k] = __vimin_s32_relu((__mulhi(uu, m0[k]) + rnd[k]) >> sh[k], (1 << kOut) - 1);
          v |= (uint32_t)y[k] << (8 * k);
        }
      }
      if constexpr (kOut == 32) {
        if (pix < g.npix) st_lane<kV>(reinterpret_cast<int32_t*>(a.y + pix * a.y_row_bytes) + g.ch0, y);
      } else {
        store_codes<kOut, kV>(a, g, pix, v << obase);
      }
    }
  }
}

// (not inlined: its int64 arithmetic would otherwise set the register budget of the table form)
template <bool kSkip, int kOut, int kSkipBits, int kV>
__device__ __noinline__ void lane_general(const EltArgs& a, const LaneGeo& g, const EpiChan (&ec)[kV]) {
  constexpr int kPix = 2;
  const int i0 = g.ch0 & 31;
  for (int64_t p0 = g.first; p0 < g.npix; p0 += g.stride) {
    int32_t av[kPix][kV], sv[kPix][kV];
#pragma unroll
    for (int u = 0; u < kPix; ++u) {
      const int64_t pix = p0 + (int64_t)u * g.wpb;
#pragma unroll
      for (int k = 0; k < kV; ++k) { av[u][k] = 0; sv[u][k] = 0; }
      if (pix >= g.npix) continue;
      ld_lane<kV>(reinterpret_cast<const int32_t*>(a.a) + pix * a.c + g.ch0, av[u]);
      if constexpr (kSkip) {
        const uint8_t* srow = a.b + skip_pixel<kSkip, kSkipBits>(a, g, pix) * a.b_row_bytes;
        if constexpr (kSkipBits == 32) {
          ld_lane<kV>(reinterpret_cast<const int32_t*>(srow) + g.ch0, sv[u]);
        } else {
          const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(srow + (g.ch0 >> 5) * group_bytes(kSkipBits)) +
                                   i0 / (32 / kSkipBits));
#pragma unroll
          for (int k = 0; k < kV; ++k)
            sv[u][k] = (int32_t)((w >> code_pos<kSkipBits>(i0 + k)) & ((1u << kSkipBits) - 1u));
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kPix; ++u) {
      const int64_t pix = p0 + (int64_t)u * g.wpb;
      int32_t y[kV];
      uint32_t v = 0;
#pragma unroll
      for (int k = 0; k < kV; ++k) {
        y[k] = epilogue<kSkip>(av[u][k], sv[u][k], ec[k], a.scale_main, kOut);
        if constexpr (kOut != 32) v |= (uint32_t)y[k] << code_pos<kOut>(i0 + k);
      }
      if constexpr (kOut == 32) {
        if (pix < g.npix) st_lane<kV>(reinterpret_cast<int32_t*>(a.y + pix * a.y_row_bytes) + g.ch0, y);
      } else {
        store_codes<kOut, kV>(a, g, pix, v);
      }
    }
  }
}

template <bool kSkip, int kOut, int kSkipBits, int kV>
__global__ void __launch_bounds__(kThreads, 3)
    eltwise_lane_kernel(const EltArgs a, int64_t npix, int warps_per_block, int tstride) {
  extern __shared__ int32_t tab[];  // kSkip, tstride > 0: [2^kSkipBits][tstride] bias + rhu(s c, d)
  LaneGeo g;
  g.lane = threadIdx.x & 31;
  const int blocks = a.c / (32 * kV);
  const int wg = blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5);
  g.first = wg / blocks;
  g.ch0 = 32 * kV * (wg % blocks) + kV * g.lane;
  g.npix = npix;
  g.wpb = warps_per_block;
  g.same_grid = a.upsample == 1 && a.b_h == a.h && a.b_w == a.w;
  const int64_t lv = (int64_t)a.level * a.c;
  bool ok = true;
  if constexpr (kOut != 32)
    for (int ch = threadIdx.x; ch < a.c; ch += kThreads) ok = ok && __ldg(a.shift + lv + ch) >= 2;  // R >= 33
  if constexpr (kSkip) {
    if constexpr (kSkipBits <= 8) {
      if (tstride > 0 && a.scale_main == 0) {
        // one channel per thread: its constants once, then its 2^kSkipBits entries
        for (int ch = threadIdx.x; ch < a.c; ch += kThreads) {
          const int d = __ldg(a.skip_d + lv + ch);
          const int64_t bias = a.bias ? __ldg(a.bias + lv + ch) : 0, cc = __ldg(a.skip_c + lv + ch);
          ok = ok && d >= 0 && d <= 62;
          const int dd = d >= 0 && d <= 62 ? d : 0;
          for (int sc = 0; sc < (1 << kSkipBits); ++sc) {
            const int64_t t = bias + rhu(sc * cc, dd);
            ok = ok && t >= INT32_MIN && t <= INT32_MAX;
            tab[sc * tstride + ch + (ch >> 5)] = (int32_t)t;
          }
        }
      } else {
        ok = false;
      }
    } else {
      ok = false;
    }
  }
  ok = __syncthreads_and(ok);
  EpiChan ec[kV];
#pragma unroll
  for (int k = 0; k < kV; ++k) {
    const int64_t idx = lv + g.ch0 + k;
    ec[k].bias = a.bias ? __ldg(a.bias + idx) : 0;
    ec[k].m0 = kOut != 32 ? __ldg(a.m0 + idx) : 0;
    ec[k].r = kOut != 32 ? (int8_t)(31 + __ldg(a.shift + idx)) : 0;
    ec[k].c = kSkip ? __ldg(a.skip_c + idx) : 0;
    ec[k].d = kSkip ? __ldg(a.skip_d + idx) : 0;
  }
  if (ok) {
    g.stride = (int64_t)kLanePix * g.wpb;
    int32_t b[kV], m0[kV], rnd[kV], sh[kV];
#pragma unroll
    for (int k = 0; k < kV; ++k) {
      const int ch = g.ch0 + k;
      b[k] = kSkip ? ch + (ch >> 5) : ec[k].bias;
      m0[k] = ec[k].m0;
      sh[k] = kOut != 32 ? ec[k].r - 32 : 1;
      rnd[k] = kOut != 32 ? 1 << (ec[k].r - 33) : 0;
    }
    lane_fast<kSkip, kOut, kSkipBits, kV>(a, g, b, m0, rnd, sh, tab, tstride);
  } else {
    g.stride = (int64_t)2 * g.wpb;
    lane_general<kSkip, kOut, kSkipBits, kV>(a, g, ec);
  }
}

// The same requant / skip add with its inputs staged through shared memory by the bulk-copy
// engine: rows of consecutive pixels are contiguous in HBM (the int32 tensor, and the skip
// tensor on the same grid), so one 1D bulk copy per operand fills a stage of P pixels (about
// 32 KB of int32 rows, StageGeo). A producer warp (one thread) keeps `stages` stages in flight
// per block, so the bytes in
// flight no longer depend on registers; 8 consumer warps take the filled stages in turn.
// Warp w owns channel block w % cblocks (kV channels per lane, constants in registers) and
// every (8 / cblocks)-th pixel of a stage. The epilogue is the table form above (exact when
// the block's check passes) or, if not, the int64 general form on each pixel's lane group.
// Every wait is bounded: a wait that runs out sets the status word to a timeout, raises the
// block's abort flag and leaves; the producer then waits (bounded) for its copies in flight.
struct StageGeo {
  int P;                 // pixels per stage
  int stages;
  int64_t nchunks;       // ceil(npix / P)
  uint32_t a_bytes;      // bytes of one stage's int32 rows (P * c * 4)
  uint32_t s_bytes;      // bytes of one stage's skip rows (P * b_row_bytes, 0 without a skip)
  uint32_t stage_bytes;  // a_bytes + s_bytes rounded to 128
  uint32_t tab_bytes;    // skip table bytes rounded to 128
};

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar), "l"(policy) : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// one pixel of one lane group in the int64 general form (rare: constants the table cannot hold)
template <bool kSkip, int kOut, int kSkipBits, int kV>
__device__ __noinline__ void staged_general(const EltArgs& a, const int32_t* arow, const uint8_t* srow,
                                            int ch0, int lane, int64_t pix) {
  const int64_t lv = (int64_t)a.level * a.c;
  const int i0 = ch0 & 31;
  uint32_t v = 0;
  int32_t y[kV];
#pragma unroll
  for (int k = 0; k < kV; ++k) {
    EpiChan ec;
    const int64_t idx = lv + ch0 + k;
    ec.bias = a.bias ? __ldg(a.bias + idx) : 0;
    ec.m0 = kOut != 32 ? __ldg(a.m0 + idx) : 0;
    ec.r = kOut != 32 ? (int8_t)(31 + __ldg(a.shift + idx)) : 0;
    ec.c = kSkip ? __ldg(a.skip_c + idx) : 0;
    ec.d = kSkip ? __ldg(a.skip_d + idx) : 0;
    int32_t sv = 0;
    if constexpr (kSkip) {
      const int i = i0 + k;
      const uint32_t w = reinterpret_cast<const uint32_t*>(srow + (ch0 >> 5) * group_bytes(kSkipBits))[i / (32 / kSkipBits)];
      sv = (int32_t)((w >> code_pos<kSkipBits>(i)) & ((1u << kSkipBits) - 1u));
    }
    y[k] = epilogue<kSkip>(arow[ch0 + k], sv, ec, a.scale_main, kOut);
    if constexpr (kOut != 32) v |= (uint32_t)y[k] << code_pos<kOut>(i0 + k);
  }
  if constexpr (kOut == 32) {
    st_lane<kV>(reinterpret_cast<int32_t*>(a.y + pix * a.y_row_bytes) + ch0, y);
  } else {
    constexpr int q = 32 / kOut;
    constexpr int span = (q / 4 * 4 + kV - 1) / kV;
#pragma unroll
    for (int off = 1; off < span; off <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, off);
    if (lane % span == 0)
      reinterpret_cast<uint32_t*>(a.y + pix * a.y_row_bytes + (ch0 >> 5) * group_bytes(kOut))[i0 / q] = v;
  }
}

template <bool kSkip, int kOut, int kSkipBits, int kV>
__global__ void __launch_bounds__(kThreads + 32, kSkip ? 2 : 3)  // the skip form: its table limits it to 2
    eltwise_staged_kernel(const EltArgs a, int64_t npix, const StageGeo sg, int tstride) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ uint64_t bars[2 * 8];  // full[s], empty[s], s < 8
  __shared__ int abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int32_t* tab = reinterpret_cast<int32_t*>(smem);
  uint8_t* stage0 = smem + sg.tab_bytes;
  const uint32_t full0 = tc::smem_u32(&bars[0]), empty0 = tc::smem_u32(&bars[8]);
  if (tid == 0) {
    abort_flag = 0;
    for (int s = 0; s < sg.stages; ++s) {
      tc::mbar_init(full0 + 8 * s, 1);
      tc::mbar_init(empty0 + 8 * s, kThreads / 32);
    }
    tc::fence_barrier_init();
  }
  // the block's form (table fits / every R >= 33) and its skip table, as in the lane kernel
  const int64_t lv = (int64_t)a.level * a.c;
  bool ok = true, small = true;  // small: every table entry within [-2^30, 2^30]
  if (tid < kThreads) {
    if constexpr (kOut != 32)
      for (int ch = tid; ch < a.c; ch += kThreads) ok = ok && __ldg(a.shift + lv + ch) >= 2;
    if constexpr (kSkip) {
      if (tstride > 0 && a.scale_main == 0) {
        for (int ch = tid; ch < a.c; ch += kThreads) {
          const int d = __ldg(a.skip_d + lv + ch);
          const int64_t bias = a.bias ? __ldg(a.bias + lv + ch) : 0, cc = __ldg(a.skip_c + lv + ch);
          ok = ok && d >= 0 && d <= 62;
          const int dd = d >= 0 && d <= 62 ? d : 0;
          for (int sc = 0; sc < (1 << kSkipBits); ++sc) {
            const int64_t t = bias + rhu(sc * cc, dd);
            ok = ok && t >= INT32_MIN && t <= INT32_MAX;
            small = small && t >= -(1LL << 30) && t <= (1LL << 30);
            tab[sc * tstride + ch + (ch >> 5)] = (int32_t)t;
          }
        }
      } else {
        ok = false;
      }
    }
  }
  ok = __syncthreads_and(ok);
  small = __syncthreads_and(small);

  if (warp == kThreads / 32) {
    // producer: thread 0 of the last warp issues the stage copies
    if (lane != 0) return;
    const uint64_t pol = policy_evict_first();
    int it = 0;
    bool live = true;
    for (int64_t j = blockIdx.x; j < sg.nchunks && live; j += gridDim.x, ++it) {
      const int s = it % sg.stages;
      if (it >= sg.stages && !tc::mbar_wait(empty0 + 8 * s, ((it / sg.stages) - 1) & 1, &abort_flag)) {
        tc::fail(&abort_flag, a.status);
        live = false;
        break;
      }
      const int64_t p0 = j * sg.P;
      const int np = (int)(npix - p0 < sg.P ? npix - p0 : sg.P);
      const uint32_t ab = (uint32_t)np * (uint32_t)a.c * 4u;
      const uint32_t sb = kSkip ? (uint32_t)np * (uint32_t)a.b_row_bytes : 0u;
      const uint32_t dst = tc::smem_u32(stage0 + (size_t)s * sg.stage_bytes);
      tc::mbar_arrive_expect_tx(full0 + 8 * s, ab + sb);
      bulk_g2s(dst, a.a + p0 * a.c * 4, ab, full0 + 8 * s, pol);
      if constexpr (kSkip) bulk_g2s(dst + sg.a_bytes, a.b + p0 * a.b_row_bytes, sb, full0 + 8 * s, pol);
    }
    // before leaving, the copies still in flight (the last `stages` chunks) land: bounded
    const int issued = it;
    for (int k = issued - sg.stages > 0 ? issued - sg.stages : 0; k < issued; ++k) {
      const int s = k % sg.stages;
      if (!tc::mbar_wait(full0 + 8 * s, (k / sg.stages) & 1, &abort_flag)) break;
    }
    return;
  }

  // consumers
  const int cblocks = a.c / (32 * kV);
  const int cb = warp % cblocks, pg = warp / cblocks, pgs = (kThreads / 32) / cblocks;
  const int ch0 = 32 * kV * cb + kV * lane;
  const int i0 = ch0 & 31;
  // b: the bias (no skip) or the channel's table column (skip)
  int32_t b[kV], m0[kV], rnd[kV], sh[kV];
#pragma unroll
  for (int k = 0; k < kV; ++k) {
    const int ch = ch0 + k;
    const int64_t idx = lv + ch;
    const int r = kOut != 32 ? 31 + __ldg(a.shift + idx) : 33;
    b[k] = kSkip ? ch + (ch >> 5) : (a.bias ? __ldg(a.bias + idx) : 0);
    m0[k] = kOut != 32 ? __ldg(a.m0 + idx) : 0;
    sh[k] = r - 32;
    rnd[k] = r >= 33 ? 1 << (r - 33) : 0;
  }
  const int sbase = kSkip ? code_pos<kSkip ? kSkipBits : 8>(i0) : 0;
  const int obase = kOut != 32 ? code_pos<kOut != 32 ? kOut : 8>(i0) : 0;
  int it = 0;
  for (int64_t j = blockIdx.x; j < sg.nchunks; j += gridDim.x, ++it) {
    const int s = it % sg.stages;
    if (!tc::mbar_wait(full0 + 8 * s, (it / sg.stages) & 1, &abort_flag)) {
      tc::fail(&abort_flag, a.status);
      return;
    }
    const int64_t p0 = j * sg.P;
    const int np = (int)(npix - p0 < sg.P ? npix - p0 : sg.P);
    const uint8_t* st = stage0 + (size_t)s * sg.stage_bytes;
    if (!ok) {
      for (int p = pg; p < np; p += pgs)
        staged_general<kSkip, kOut, kSkipBits, kV>(a, reinterpret_cast<const int32_t*>(st) + (size_t)p * a.c,
                                                   st + sg.a_bytes + (size_t)p * a.b_row_bytes, ch0, lane, p0 + p);
    } else {
      // two pixels per step (the second clamped to the last one and its store predicated off)
      // so their chains interleave
      for (int p = pg; p < np; p += 2 * pgs) {
        const int pp[2] = {p, p + pgs < np ? p + pgs : np - 1};
        int32_t av[2][kV];
        uint32_t sw[2] = {0, 0};
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const int32_t* arow = reinterpret_cast<const int32_t*>(st) + pp[u] * a.c;
          if constexpr (kV == 4) {
            const int4 x = *reinterpret_cast<const int4*>(arow + ch0);
            av[u][0] = x.x; av[u][1] = x.y; av[u][2] = x.z; av[u][3] = x.w;
          } else if constexpr (kV == 2) {
            const int2 x = *reinterpret_cast<const int2*>(arow + ch0);
            av[u][0] = x.x; av[u][1] = x.y;
          } else {
            av[u][0] = arow[ch0];
          }
          if constexpr (kSkip)
            sw[u] = reinterpret_cast<const uint32_t*>(st + sg.a_bytes + pp[u] * (int)a.b_row_bytes +
                                                      (ch0 >> 5) * group_bytes(kSkipBits))[i0 / (32 / kSkipBits)] >> sbase;
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          const bool live = u == 0 || p + pgs < np;
          uint8_t* yrow = a.y + (p0 + pp[u]) * a.y_row_bytes;
          int32_t y[kV];
          uint32_t v = 0;
          int32_t us[kV];
          if constexpr (kSkip) {
            // codes: masked once, then byte k of the word is channel k's code
            const uint32_t swm = sw[u] & (((1u << kSkipBits) - 1u) * 0x01010101u);
            int32_t t[kV];
            int32_t f = 0;  // sign bit set iff some a is outside [-2^30, 2^30)
#pragma unroll
            for (int k = 0; k < kV; ++k) {
              const uint32_t code = k == 0 ? (swm & 0xffu) : (k == 3 ? swm >> 24 : __byte_perm(swm, 0u, 0x4440u + k));
              t[k] = tab[(int)code * tstride + b[k]];
              f |= av[u][k] + (1 << 30);
            }
            if (small && f >= 0) {
              // |a| <= 2^30 and |t| <= 2^30: the sum cannot leave int32
#pragma unroll
              for (int k = 0; k < kV; ++k) us[k] = av[u][k] + t[k];
            } else {
              // sat32(a + t): the wrapped sum, replaced by the bound of a's sign where a and t
              // have one sign and the sum the other
#pragma unroll
              for (int k = 0; k < kV; ++k) {
                const int32_t w = (int32_t)((uint32_t)av[u][k] + (uint32_t)t[k]);
                us[k] = ((w ^ av[u][k]) & (w ^ t[k])) < 0 ? (av[u][k] >> 31) ^ INT32_MAX : w;
              }
            }
          } else {
#pragma unroll
            for (int k = 0; k < kV; ++k) us[k] = add_sat_s32(av[u][k], b[k]);
          }
#pragma unroll
          for (int k = 0; k < kV; ++k) {
            const int32_t uu = us[k];
            if constexpr (kOut == 32) {
              y[k] = uu;
            } else {
              y[k] = __vimin_s32_relu((__mulhi(uu, m0[k]) + rnd[k]) >> sh[k], (1 << kOut) - 1);
              v += (uint32_t)y[k] << (8 * k);
            }
          }
          if constexpr (kOut == 32) {
            if (live) st_lane<kV>(reinterpret_cast<int32_t*>(yrow) + ch0, y);
          } else {
            constexpr int q = 32 / kOut;
            constexpr int span = (q / 4 * 4 + kV - 1) / kV;
            v <<= obase;
#pragma unroll
            for (int off = 1; off < span; off <<= 1) v |= __shfl_xor_sync(0xffffffffu, v, off);
            if (live && lane % span == 0)
              reinterpret_cast<uint32_t*>(yrow + (ch0 >> 5) * group_bytes(kOut))[i0 / q] = v;
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) tc::mbar_arrive(empty0 + 8 * s);
  }
}

__global__ void __launch_bounds__(kThreads) maxpool_kernel(const PoolArgs a) {
  const int groups = (a.c + 31) / 32;
  const int64_t total = (int64_t)a.n * a.ho * a.wo * groups;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= total) return;
  const int64_t pix = t / groups;
  const int ch0 = (int)(t - pix * groups) * 32;
  const int64_t hw = (int64_t)a.ho * a.wo;
  const int64_t img = pix / hw;
  const int64_t rem = pix - img * hw;
  const int oh = (int)(rem / a.wo), ow = (int)(rem - (rem / a.wo) * a.wo);
  int32_t best[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) best[i] = 0;  // codes are >= 0; every window holds a tap
  for (int r = 0; r < a.k; ++r) {
    const int hi = oh * a.stride - a.pad + r;
    if (hi < 0 || hi >= a.h) continue;
    for (int s = 0; s < a.k; ++s) {
      const int wi = ow * a.stride - a.pad + s;
      if (wi < 0 || wi >= a.w) continue;
      int32_t v[32];
      load_vals(a.x + ((img * a.h + hi) * a.w + wi) * a.row_bytes, a.bits, a.c, ch0, false, v);
#pragma unroll
      for (int i = 0; i < 32; ++i) best[i] = max(best[i], v[i]);
    }
  }
  store_vals(a.y + pix * a.row_bytes, a.bits, a.c, ch0, best);
}

// Max-pool on packed codes of 2, 4 or 8 bits (Sec. 3.2.4: max-pooling commutes with the
// monotone quantizer, so it runs on the codes), word by word with PoolAcc's packed 16-bit
// maxima. One thread owns kVec words of one output pixel's row. A window tap outside the input
// is replaced by the nearest row / column inside it: the padding is smaller than the window,
// so that tap lies in the same window, and a maximum taken twice is the same maximum. With
// kK = 3 (the network's 3x3 pools) the 9 taps are unrolled and their loads issued together;
// kK = 0 loops over a.k.
// Grid: z = image, y = output row, x = the row's (output pixel, unit) pairs, unit fastest
// (ushift = log2 of the units per pixel when that is a power of two, else -1).
template <int kBits, int kVec, int kK>
__global__ void __launch_bounds__(kThreads) maxpool_packed_kernel(const PoolArgs a, int ushift) {
  const int units = (int)(a.row_bytes / (4 * kVec));
  const int x = blockIdx.x * kThreads + threadIdx.x;
  const int ow = ushift >= 0 ? x >> ushift : x / units;
  const int u = x - ow * units;
  if (ow >= a.wo) return;
  const int oh = blockIdx.y, img = blockIdx.z;
  const int64_t pix = ((int64_t)img * a.ho + oh) * a.wo + ow;
  PoolAcc<kBits> acc[kVec];
#pragma unroll
  for (int v = 0; v < kVec; ++v) acc[v].init();
  const int k = kK > 0 ? kK : a.k;
  // the window's taps in row-major order, two per maximum (an odd last one alone)
  auto tap = [&](int t, uint32_t (&w)[kVec]) {
    const int r = t / k, s = t - r * k;
    const int hi = min(max(oh * a.stride - a.pad + r, 0), a.h - 1);
    const int wi = min(max(ow * a.stride - a.pad + s, 0), a.w - 1);
    const uint32_t* src = reinterpret_cast<const uint32_t*>(
        a.x + (((int64_t)img * a.h + hi) * a.w + wi) * a.row_bytes) + u * kVec;
    if constexpr (kVec == 4) {
      const uint4 q = __ldg(reinterpret_cast<const uint4*>(src));
      w[0] = q.x; w[1] = q.y; w[2] = q.z; w[3] = q.w;
    } else {
#pragma unroll
      for (int v = 0; v < kVec; ++v) w[v] = __ldg(src + v);
    }
  };
  const int taps = k * k;
#pragma unroll
  for (int t = 0; t + 1 < (kK > 0 ? kK * kK : taps); t += 2) {
    uint32_t w0[kVec], w1[kVec];
    tap(t, w0);
    tap(t + 1, w1);
#pragma unroll
    for (int v = 0; v < kVec; ++v) acc[v].add2(w0[v], w1[v]);
  }
  if (taps & 1) {
    uint32_t w0[kVec];
    tap(taps - 1, w0);
#pragma unroll
    for (int v = 0; v < kVec; ++v) acc[v].add(w0[v]);
  }
  uint32_t o[kVec];
#pragma unroll
  for (int v = 0; v < kVec; ++v) o[v] = acc[v].word();
  uint32_t* dst = reinterpret_cast<uint32_t*>(a.y + pix * a.row_bytes) + u * kVec;
  if constexpr (kVec == 4) {
    *reinterpret_cast<uint4*>(dst) = make_uint4(o[0], o[1], o[2], o[3]);
  } else {
#pragma unroll
    for (int v = 0; v < kVec; ++v) dst[v] = o[v];
  }
}

// The 3x3 stride-2 max-pool (the stem's) on packed codes, two horizontally adjacent outputs
// per thread: their windows share the middle column, so 5 columns x 3 rows of taps serve both.
// Per column the three rows' maximum first (one three-input maximum per plane), then each
// output's three columns. Taps outside the input are clamped inside, as above. Thread x of
// grid row (img, oh) takes output pair x >> ushift (x / units when the units per pixel are not
// a power of two), unit x - pair * units; false past the row's end.
template <int kBits, int kVec>
__device__ __forceinline__ bool pool3s2_pair(const PoolArgs& a, int ushift, int img, int oh, int x, int& ow, int& u,
                                             uint32_t (&oa)[kVec], uint32_t (&ob)[kVec]) {
  const int units = (int)(a.row_bytes / (4 * kVec));
  const int op = ushift >= 0 ? x >> ushift : x / units;  // output pair: columns 2 op, 2 op + 1
  u = x - op * units;
  ow = 2 * op;
  if (ow >= a.wo) return false;
  const uint8_t* rows[3];
#pragma unroll
  for (int r = 0; r < 3; ++r)
    rows[r] = a.x + ((int64_t)img * a.h + min(max(2 * oh - a.pad + r, 0), a.h - 1)) * a.w * a.row_bytes +
              (int64_t)u * kVec * 4;
  auto column = [&](int c, PoolAcc<kBits> (&m)[kVec]) {
    const int64_t off = (int64_t)min(max(2 * ow - a.pad + c, 0), a.w - 1) * a.row_bytes;
    uint32_t w[3][kVec];
#pragma unroll
    for (int r = 0; r < 3; ++r) {
      const uint32_t* src = reinterpret_cast<const uint32_t*>(rows[r] + off);
      if constexpr (kVec == 4) {
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(src));
        w[r][0] = q.x; w[r][1] = q.y; w[r][2] = q.z; w[r][3] = q.w;
      } else {
#pragma unroll
        for (int v = 0; v < kVec; ++v) w[r][v] = __ldg(src + v);
      }
    }
#pragma unroll
    for (int v = 0; v < kVec; ++v) m[v].set3(w[0][v], w[1][v], w[2][v]);
  };
  PoolAcc<kBits> A[kVec], B[kVec], c1[kVec], c3[kVec];
  column(0, A);
  column(1, c1);
  column(2, B);
#pragma unroll
  for (int v = 0; v < kVec; ++v) A[v].max3(c1[v], B[v]);  // A = max(col 0, col 1, col 2); B = col 2
  column(3, c3);
  column(4, c1);
#pragma unroll
  for (int v = 0; v < kVec; ++v) B[v].max3(c3[v], c1[v]);  // B = max(col 2, col 3, col 4)
#pragma unroll
  for (int v = 0; v < kVec; ++v) { oa[v] = A[v].word(); ob[v] = B[v].word(); }
  return true;
}

template <int kVec>
__device__ __forceinline__ void store_words(uint8_t* p, const uint32_t (&o)[kVec]) {
  if constexpr (kVec == 4) {
    *reinterpret_cast<uint4*>(p) = make_uint4(o[0], o[1], o[2], o[3]);
  } else {
#pragma unroll
    for (int v = 0; v < kVec; ++v) reinterpret_cast<uint32_t*>(p)[v] = o[v];
  }
}

// Grid: z = image, y = output row, x = the row's (output pair, unit) pairs, unit fastest.
// (3 blocks per SM: measured faster than the unconstrained register count, and than 4)
template <int kBits, int kVec>
__global__ void __launch_bounds__(kThreads, kBits == 2 ? 2 : 3) maxpool3s2_pair_kernel(const PoolArgs a, int ushift) {
  int ow, u;
  uint32_t oa[kVec], ob[kVec];
  const int img = blockIdx.z, oh = blockIdx.y;
  if (!pool3s2_pair<kBits, kVec>(a, ushift, img, oh, blockIdx.x * kThreads + threadIdx.x, ow, u, oa, ob)) return;
  uint8_t* dst = a.y + (((int64_t)img * a.ho + oh) * a.wo + ow) * a.row_bytes + (int64_t)u * kVec * 4;
  store_words<kVec>(dst, oa);
  if (ow + 1 < a.wo) store_words<kVec>(dst + a.row_bytes, ob);
}

// The byte image of one packed unit (kVec words of 2- or 4-bit codes): one byte per code, in
// channel order (channel i of a word at bit 8 (i % 4) + bits ((i % q) / 4), q = 32 / bits, so
// the word's bit planes (w >> bits j) & 0x0303.. / 0x0F0F.. hold channels 4 j .. 4 j + 3).
template <int kBits, int kVec>
__device__ __forceinline__ void store_code_bytes(uint8_t* p, const uint32_t (&o)[kVec]) {
  constexpr int kPl = 8 / kBits;                     // byte planes per word
  constexpr uint32_t kB = kBits == 2 ? 0x03030303u : 0x0F0F0F0Fu;
#pragma unroll
  for (int v = 0; v < kVec; ++v) {
    uint32_t b[kPl];
#pragma unroll
    for (int j = 0; j < kPl; ++j) b[j] = (o[v] >> (kBits * j)) & kB;
    if constexpr (kPl == 4) *reinterpret_cast<uint4*>(p + 16 * v) = make_uint4(b[0], b[1], b[2], b[3]);
    else *reinterpret_cast<uint2*>(p + 8 * v) = make_uint2(b[0], b[1]);
  }
}

// Max-pool (3x3, stride 2) fused with the expansion of its output for a convolution with
// padding cpad: writes the pooled codes to a.y and their zero-padded byte image (rows of c
// bytes; image row (img (ho + 2 cpad) + oh + cpad) (wo + 2 cpad) + ow + cpad) to ws. Grid row
// y = ho of each image writes the image's border pixels (zeros), spread over its x threads.
template <int kBits, int kVec>
__global__ void __launch_bounds__(kThreads, kBits == 2 ? 2 : 3)
    maxpool3s2_expand_kernel(const PoolArgs a, int ushift, uint8_t* ws, int cpad) {
  const int img = blockIdx.z, oh = blockIdx.y;
  const int hp = a.ho + 2 * cpad, wp = a.wo + 2 * cpad;
  const int64_t ibase = (int64_t)img * hp * wp;
  constexpr int kUnitBytes = kVec * 4 * 8 / kBits;  // byte-image bytes of one packed unit
  if (oh == a.ho) {
    // border: cpad rows on top and bottom (wp pixels each), cpad columns left and right
    const int units = (int)(a.row_bytes / (4 * kVec));
    const int nb = 2 * cpad * wp + 2 * cpad * a.ho;
    const int64_t items = (int64_t)nb * units;
    for (int64_t e = (int64_t)blockIdx.x * kThreads + threadIdx.x; e < items; e += (int64_t)gridDim.x * kThreads) {
      const int b = (int)(e / units), uu = (int)(e - (int64_t)b * units);
      int r, cidx;
      if (b < 2 * cpad * wp) {
        const int t = b / wp;
        r = t < cpad ? t : a.ho + t;  // rows 0 .. cpad - 1, then ho + cpad .. ho + 2 cpad - 1
        cidx = b - t * wp;
      } else {
        const int b2 = b - 2 * cpad * wp, t = b2 / (2 * cpad), s2 = b2 - t * 2 * cpad;
        r = cpad + t;
        cidx = s2 < cpad ? s2 : a.wo + s2;
      }
      uint8_t* p = ws + ((ibase + (int64_t)r * wp + cidx) * a.c) + (int64_t)uu * kUnitBytes;
#pragma unroll
      for (int k = 0; k < kUnitBytes; k += 16) *reinterpret_cast<uint4*>(p + k) = make_uint4(0u, 0u, 0u, 0u);
    }
    return;
  }
  int ow, u;
  uint32_t oa[kVec], ob[kVec];
  if (!pool3s2_pair<kBits, kVec>(a, ushift, img, oh, blockIdx.x * kThreads + threadIdx.x, ow, u, oa, ob)) return;
  uint8_t* dst = a.y + (((int64_t)img * a.ho + oh) * a.wo + ow) * a.row_bytes + (int64_t)u * kVec * 4;
  uint8_t* img_row = ws + ((ibase + (int64_t)(oh + cpad) * wp + ow + cpad) * a.c) + (int64_t)u * kUnitBytes;
  store_words<kVec>(dst, oa);
  store_code_bytes<kBits, kVec>(img_row, oa);
  if (ow + 1 < a.wo) {
    store_words<kVec>(dst + a.row_bytes, ob);
    store_code_bytes<kBits, kVec>(img_row + a.c, ob);
  }
}

__global__ void __launch_bounds__(kThreads)
pack_kernel(const int32_t* codes, int64_t rows, int c, int bits, int64_t row_bytes, uint8_t* out) {
  const int groups = (c + 31) / 32;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= rows * groups) return;
  const int64_t r = t / groups;
  const int ch0 = (int)(t - r * groups) * 32;
  int32_t v[32];
#pragma unroll 4
  for (int i = 0; i < 32; ++i) v[i] = (ch0 + i < c) ? codes[r * c + ch0 + i] : 0;
  if (bits == 8) {
    for (int i = 0; i < 32; ++i)
      if (ch0 + i < c) out[r * row_bytes + ch0 + i] = (uint8_t)(v[i] & 0xFF);
    return;
  }
  uint32_t g[8];
  pack_group_vals(v, bits, g);
  store_group(out + r * row_bytes + (ch0 >> 5) * group_bytes(bits), g, bits);
}

__global__ void __launch_bounds__(kThreads)
unpack_kernel(const uint8_t* packed, int64_t rows, int c, int bits, int64_t row_bytes, int is_signed,
              int32_t* out) {
  const int groups = (c + 31) / 32;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= rows * groups) return;
  const int64_t r = t / groups;
  const int ch0 = (int)(t - r * groups) * 32;
  int32_t v[32];
  load_vals(packed + r * row_bytes, bits, c, ch0, is_signed != 0, v);
  for (int i = 0; i < 32; ++i)
    if (ch0 + i < c) out[r * c + ch0 + i] = v[i];
}

// Prepared weights: E4M3 sign-magnitude bytes [cout_pad][k_pad] (zero padded; only when
// every |w| <= 15) followed by int16 [cout][k_total].
__global__ void __launch_bounds__(kThreads)
prepare_weights_kernel(const uint8_t* wp, int w_bits, int w_format, WeightGeom g, int64_t w_row_bytes,
                       int make_e4m3, uint8_t* out) {
  // make_e4m3: 0 none (weights too wide for the tensor cores), 1 the plain layout, 2 the
  // split layout of 8-bit two's-complement weights (per 128 channels: w_lo rows, w_hi rows)
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  const int64_t e4_rows = make_e4m3 == 2 ? g.split_rows : g.cout_pad;
  const int64_t n_e4 = e4_rows * g.k_pad;
  const int64_t n_i16 = (int64_t)g.cout * g.k_total;
  if (t >= n_e4 + n_i16) return;
  int64_t co, k;
  int part = 0;  // split layout: 0 = w_lo, 1 = w_hi
  if (t < n_e4) {
    int64_t rr = t / g.k_pad;
    k = t - rr * g.k_pad;
    if (make_e4m3 == 2) {
      const int64_t blk = rr / 256, within = rr - blk * 256;
      part = (int)(within >> 7);
      co = blk * 128 + (within & 127);
    } else {
      co = rr;
    }
  } else {
    co = (t - n_e4) / g.k_total; k = (t - n_e4) - co * g.k_total;
  }
  int32_t w = 0;
  if (co < g.cout && k < g.k_total) {
    const int64_t tap = k / g.cin;
    const int ch = (int)(k - tap * g.cin);
    const uint8_t* row = wp + (co * g.kh * g.kw + tap) * w_row_bytes;
    if (w_format == 0) {
      w = read_code(row, ch, w_bits, true);
    } else {  // Eq. 3 odd grid: eta -> 2 eta - (2^k - 1)
      w = 2 * read_code(row, ch, w_bits, false) - ((1 << w_bits) - 1);
    }
  }
  if (t < n_e4) {
    if (make_e4m3 == 2) w = part == 0 ? (w & 15) : (w >> 4);  // w = 16 w_hi + w_lo, w_lo in [0, 15]
    if (make_e4m3) {
      const uint32_t mag = (uint32_t)(w < 0 ? -w : w);
      out[t] = (uint8_t)((w < 0 ? 0x80u : 0u) | (mag & 0x0Fu));
    } else {
      out[t] = 0;
    }
  } else {
    reinterpret_cast<int16_t*>(out + g.i16_offset)[t - n_e4] = (int16_t)w;
  }
}

// The E2M1 block of the prepared weights: byte b of row co holds weights k = 2b (low nibble)
// and 2b + 1 (high nibble) as the E2M1 values w / 2: sign bit 3, magnitude code |w| for
// |w| <= 4 (0, 0.5, 1, 1.5, 2). Padding rows and columns are 0.
__global__ void __launch_bounds__(kThreads)
prepare_fp4_kernel(const uint8_t* wp, int w_bits, int w_format, WeightGeom g, int64_t w_row_bytes, uint8_t* out) {
  const int64_t row_bytes = g.k_pad / 2;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= (int64_t)g.cout_pad * row_bytes) return;
  const int64_t co = t / row_bytes, kb = t - co * row_bytes;
  uint32_t byte = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int64_t k = 2 * kb + h;
    int32_t w = 0;
    if (co < g.cout && k < g.k_total) {
      const int64_t tap = k / g.cin;
      const int ch = (int)(k - tap * g.cin);
      const uint8_t* row = wp + (co * g.kh * g.kw + tap) * w_row_bytes;
      w = w_format == 0 ? read_code(row, ch, w_bits, true) : 2 * read_code(row, ch, w_bits, false) - ((1 << w_bits) - 1);
    }
    const uint32_t nib = (w < 0 ? 8u : 0u) | (uint32_t)(w < 0 ? -w : w);
    byte |= nib << (4 * h);
  }
  out[g.fp4_offset + t] = (uint8_t)byte;
}

inline unsigned blocks_for(int64_t n) { return (unsigned)((n + kThreads - 1) / kThreads); }

}  // namespace elt

static int check_launch(const char* what, std::string* err) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { *err = std::string(what) + ": " + cudaGetErrorString(e); return 3; }
  return 0;
}

// kV channels per lane: int32 input, c % (32 kV) == 0, 2/4/8/32-bit output, 2/4/8/32-bit skip.
// One wave of blocks (the resident count per SM for this kernel and table size, times the SMs),
// each building its table once; the warp count a multiple of the channel-block count (warps of
// one channel block take every warps_per_block-th pixel).
template <bool kSkip, int kOut, int kSkipBits, int kV>
static void launch_lane_k(const EltArgs& a, int ts, int sms, cudaStream_t stream) {
  auto kern = elt::eltwise_lane_kernel<kSkip, kOut, kSkipBits, kV>;
  const size_t smem = ts > 0 ? ((size_t)ts << kSkipBits) * sizeof(int32_t) : 0;
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, elt::kThreads, smem) != cudaSuccess || occ < 1) occ = 1;
  const int cblocks = a.c / (32 * kV);
  const int64_t npix = (int64_t)a.n * a.h * a.w;
  int g = cblocks, w = elt::kThreads / 32;  // blocks must be a multiple of cblocks / gcd(cblocks, 8)
  while (w) { const int t = g % w; g = w; w = t; }
  const int64_t unit = cblocks / g;
  int64_t blocks = (int64_t)sms * occ;
  const int64_t need = (npix * cblocks + 7) / 8;  // one pixel per warp at most
  if (blocks > need) blocks = need;
  blocks = blocks / unit * unit;
  if (blocks < unit) blocks = unit;
  const int wpb = (int)(blocks * (elt::kThreads / 32) / cblocks);
  kern<<<(unsigned)blocks, elt::kThreads, smem, stream>>>(a, npix, wpb, ts);
}
template <bool kSkip, int kSkipBits, int kV>
static bool launch_lane_v(const EltArgs& a, int ts, int sms, cudaStream_t stream) {
  switch (a.y_bits) {
    case 2: launch_lane_k<kSkip, 2, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 4: launch_lane_k<kSkip, 4, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 8: launch_lane_k<kSkip, 8, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 32: launch_lane_k<kSkip, 32, kSkipBits, kV>(a, ts, sms, stream); return true;
    default: return false;
  }
}
template <bool kSkip, int kSkipBits>
static bool launch_lane(const EltArgs& a, int sms, cudaStream_t stream) {
  // the skip table's row stride: c columns plus one per 32 channels, rounded to 32 banks; none
  // when the main path is rescaled, the skip is int32 or the table would pass 48 KB
  int ts = 0;
  if (kSkip && kSkipBits <= 8 && a.scale_main == 0) {
    ts = (a.c + a.c / 32 + 31) / 32 * 32;
    if (((size_t)ts << kSkipBits) * sizeof(int32_t) > 48 * 1024) ts = 0;
  }
  const int v = a.c % 128 == 0 ? 4 : (a.c % 64 == 0 ? 2 : 1);  // channels per lane
  if (v == 4) return launch_lane_v<kSkip, kSkipBits, 4>(a, ts, sms, stream);
  if (v == 2) return launch_lane_v<kSkip, kSkipBits, 2>(a, ts, sms, stream);
  return launch_lane_v<kSkip, kSkipBits, 1>(a, ts, sms, stream);
}

// The staged kernel: one wave of blocks, 2 stages of about 32 KB of int32 rows each.
template <bool kSkip, int kOut, int kSkipBits, int kV>
static void launch_staged_k(const EltArgs& a, int ts, int sms, cudaStream_t stream) {
  auto kern = elt::eltwise_staged_kernel<kSkip, kOut, kSkipBits, kV>;
  const int64_t npix = (int64_t)a.n * a.h * a.w;
  const int row = a.c * 4;
  elt::StageGeo g{};
  g.P = 32768 / row > 0 ? 32768 / row : 1;  // measured: fewer, larger stages beat more, smaller ones
  g.stages = 2;
  g.nchunks = (npix + g.P - 1) / g.P;
  g.a_bytes = (uint32_t)g.P * (uint32_t)row;
  g.s_bytes = kSkip ? (uint32_t)g.P * (uint32_t)a.b_row_bytes : 0u;
  g.stage_bytes = (g.a_bytes + g.s_bytes + 127u) / 128u * 128u;
  g.tab_bytes = ts > 0 ? (uint32_t)((((size_t)ts << kSkipBits) * sizeof(int32_t) + 127) / 128 * 128) : 0u;
  const size_t smem = g.tab_bytes + (size_t)g.stages * g.stage_bytes;
  // the dynamic limit goes to the device maximum (less the kernel's static barriers), never to
  // this call's size: a graph node captured earlier with a larger table must stay launchable
  // after a smaller call
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  cudaFuncAttributes fa{};
  cudaFuncGetAttributes(&fa, kern);
  const int maxdyn = optin - (int)fa.sharedSizeBytes;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, maxdyn > (int)smem ? maxdyn : (int)smem);
  int occ = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kern, elt::kThreads + 32, smem) != cudaSuccess || occ < 1)
    occ = 1;
  int64_t blocks = (int64_t)sms * occ;
  if (blocks > g.nchunks) blocks = g.nchunks;
  kern<<<(unsigned)blocks, elt::kThreads + 32, smem, stream>>>(a, npix, g, ts);
}
template <bool kSkip, int kSkipBits, int kV>
static bool launch_staged_v(const EltArgs& a, int ts, int sms, cudaStream_t stream) {
  switch (a.y_bits) {
    case 2: launch_staged_k<kSkip, 2, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 4: launch_staged_k<kSkip, 4, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 8: launch_staged_k<kSkip, 8, kSkipBits, kV>(a, ts, sms, stream); return true;
    case 32: launch_staged_k<kSkip, 32, kSkipBits, kV>(a, ts, sms, stream); return true;
    default: return false;
  }
}
// Whether the staged kernel takes these arguments: contiguous int32 rows (and skip rows on the
// same grid, 2/4/8-bit, whole 16-byte rows) at 16-byte aligned addresses, and a channel-block
// count that divides the 8 consumer warps.
static bool staged_applies(const EltArgs& a) {
  if (a.a_bits != 32 || a.c % 32 != 0 || a.a_row_bytes != (int64_t)a.c * 4 || a.y_bits == 3) return false;
  if ((uintptr_t)a.a % 16 != 0) return false;
  const int v = a.c % 128 == 0 ? 4 : (a.c % 64 == 0 ? 2 : 1);
  const int cblocks = a.c / (32 * v);
  if (cblocks != 1 && cblocks != 2 && cblocks != 4 && cblocks != 8) return false;
  if (a.has_skip) {
    if (a.b_bits != 2 && a.b_bits != 4 && a.b_bits != 8) return false;
    if (!(a.upsample == 1 && a.b_h == a.h && a.b_w == a.w)) return false;
    if (a.b_row_bytes % 16 != 0 || (uintptr_t)a.b % 16 != 0) return false;
  }
  return true;
}
template <bool kSkip, int kSkipBits>
static bool launch_staged(const EltArgs& a, int sms, cudaStream_t stream) {
  int ts = 0;
  if (kSkip && a.scale_main == 0) {
    ts = (a.c + a.c / 32 + 31) / 32 * 32;
    if (((size_t)ts << kSkipBits) * sizeof(int32_t) > 48 * 1024) ts = 0;
  }
  const int v = a.c % 128 == 0 ? 4 : (a.c % 64 == 0 ? 2 : 1);
  if (v == 4) return launch_staged_v<kSkip, kSkipBits, 4>(a, ts, sms, stream);
  if (v == 2) return launch_staged_v<kSkip, kSkipBits, 2>(a, ts, sms, stream);
  return launch_staged_v<kSkip, kSkipBits, 1>(a, ts, sms, stream);
}

int launch_elementwise(const EltArgs& a, cudaStream_t stream, std::string* err) {
  const int64_t total = (int64_t)a.n * a.h * a.w * ((a.c + 31) / 32);
  if (total == 0) return 0;
  const bool lane_ok = a.a_bits == 32 && a.c % 32 == 0 && a.y_bits != 3 &&
                       (!a.has_skip || a.b_bits == 2 || a.b_bits == 4 || a.b_bits == 8 || a.b_bits == 32);
  if (lane_ok) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 152;
    bool ok = false;
    if (staged_applies(a)) {
      if (!a.has_skip) ok = launch_staged<false, 0>(a, sms, stream);
      else if (a.b_bits == 2) ok = launch_staged<true, 2>(a, sms, stream);
      else if (a.b_bits == 4) ok = launch_staged<true, 4>(a, sms, stream);
      else ok = launch_staged<true, 8>(a, sms, stream);
      if (ok) return check_launch("eltwise launch", err);
    }
    if (!a.has_skip) ok = launch_lane<false, 0>(a, sms, stream);
    else if (a.b_bits == 2) ok = launch_lane<true, 2>(a, sms, stream);
    else if (a.b_bits == 4) ok = launch_lane<true, 4>(a, sms, stream);
    else if (a.b_bits == 8) ok = launch_lane<true, 8>(a, sms, stream);
    else ok = launch_lane<true, 32>(a, sms, stream);
    if (ok) return check_launch("eltwise launch", err);
  }
  if (a.c <= elt::kTabChannels && a.c % 32 == 0) {
    // enough blocks for every SM several times over; each block stages the constants once
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const unsigned cap = (unsigned)(sms > 0 ? sms : 152) * 6u;
    const unsigned blocks = elt::blocks_for(total) < cap ? elt::blocks_for(total) : cap;
    if (a.has_skip) elt::eltwise_group_kernel<true><<<blocks, elt::kThreads, 0, stream>>>(a);
    else elt::eltwise_group_kernel<false><<<blocks, elt::kThreads, 0, stream>>>(a);
  } else if (a.has_skip) {
    elt::eltwise_kernel<true><<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(a);
  } else {
    elt::eltwise_kernel<false><<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(a);
  }
  return check_launch("eltwise launch", err);
}

int launch_maxpool(const PoolArgs& a, cudaStream_t stream, std::string* err) {
  const int64_t pixels = (int64_t)a.n * a.ho * a.wo;
  if (pixels == 0) return 0;
  // packed 2/4/8-bit rows: bit-plane maxima on whole words (16-byte units when the row allows)
  if ((a.bits == 2 || a.bits == 4 || a.bits == 8) && a.row_bytes % 4 == 0) {
    const bool v4 = a.row_bytes % 16 == 0;
    const int units = (int)(a.row_bytes / (v4 ? 16 : 4));
    int ushift = -1;
    for (int sft = 0; sft < 31; ++sft)
      if ((1 << sft) == units) ushift = sft;
    if ((int64_t)a.wo * units >= (1LL << 31) || a.ho > 65535 || a.n > 65535) {
      *err = "maxpool: output too large for the packed kernel's grid";
      return 1;
    }
    const dim3 blocks((unsigned)elt::blocks_for((int64_t)a.wo * units), (unsigned)a.ho, (unsigned)a.n);
    if (a.k == 3 && a.stride == 2) {
      const dim3 pblocks((unsigned)elt::blocks_for((int64_t)((a.wo + 1) / 2) * units), (unsigned)a.ho, (unsigned)a.n);
      if (a.bits == 2) {
        if (v4) elt::maxpool3s2_pair_kernel<2, 4><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool3s2_pair_kernel<2, 1><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
      } else if (a.bits == 4) {
        if (v4) elt::maxpool3s2_pair_kernel<4, 4><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool3s2_pair_kernel<4, 1><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
      } else {
        if (v4) elt::maxpool3s2_pair_kernel<8, 4><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool3s2_pair_kernel<8, 1><<<pblocks, elt::kThreads, 0, stream>>>(a, ushift);
      }
    } else if (a.k == 3) {
      if (a.bits == 2) {
        if (v4) elt::maxpool_packed_kernel<2, 4, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool_packed_kernel<2, 1, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      } else if (a.bits == 4) {
        if (v4) elt::maxpool_packed_kernel<4, 4, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool_packed_kernel<4, 1, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      } else {
        if (v4) elt::maxpool_packed_kernel<8, 4, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
        else elt::maxpool_packed_kernel<8, 1, 3><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      }
    } else if (a.bits == 2) {
      if (v4) elt::maxpool_packed_kernel<2, 4, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      else elt::maxpool_packed_kernel<2, 1, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
    } else if (a.bits == 4) {
      if (v4) elt::maxpool_packed_kernel<4, 4, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      else elt::maxpool_packed_kernel<4, 1, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
    } else {
      if (v4) elt::maxpool_packed_kernel<8, 4, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
      else elt::maxpool_packed_kernel<8, 1, 0><<<blocks, elt::kThreads, 0, stream>>>(a, ushift);
    }
    return check_launch("maxpool launch", err);
  }
  const int64_t total = pixels * ((a.c + 31) / 32);
  elt::maxpool_kernel<<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(a);
  return check_launch("maxpool launch", err);
}

int launch_maxpool_expand(const PoolArgs& a, uint8_t* ws, int32_t cpad, cudaStream_t stream, std::string* err) {
  if (a.k != 3 || a.stride != 2 || (a.bits != 2 && a.bits != 4) || a.row_bytes % 16 != 0 || a.c % 16 != 0) {
    *err = "maxpool_expand: needs a 3x3 stride-2 pool on 2- or 4-bit codes with 16-byte rows";
    return 2;
  }
  if (a.n == 0 || a.ho == 0 || a.wo == 0) return 0;
  const int units = (int)(a.row_bytes / 16);
  int ushift = -1;
  for (int sft = 0; sft < 31; ++sft)
    if ((1 << sft) == units) ushift = sft;
  if ((int64_t)((a.wo + 1) / 2) * units >= (1LL << 31) || a.ho + 1 > 65535 || a.n > 65535) {
    *err = "maxpool_expand: output too large for the kernel's grid";
    return 1;
  }
  const dim3 blocks((unsigned)elt::blocks_for((int64_t)((a.wo + 1) / 2) * units), (unsigned)(a.ho + 1), (unsigned)a.n);
  if (a.bits == 2) elt::maxpool3s2_expand_kernel<2, 4><<<blocks, elt::kThreads, 0, stream>>>(a, ushift, ws, cpad);
  else elt::maxpool3s2_expand_kernel<4, 4><<<blocks, elt::kThreads, 0, stream>>>(a, ushift, ws, cpad);
  return check_launch("maxpool_expand launch", err);
}

int launch_pack(const int32_t* codes, int64_t rows, int32_t c, int32_t bits, uint8_t* out,
                cudaStream_t stream, std::string* err) {
  const int64_t total = rows * ((c + 31) / 32);
  if (total == 0) return 0;
  elt::pack_kernel<<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(codes, rows, c, bits,
                                                                          row_bytes_of(c, bits), out);
  return check_launch("pack launch", err);
}

int launch_unpack(const uint8_t* packed, int64_t rows, int32_t c, int32_t bits, int32_t is_signed,
                  int32_t* out, cudaStream_t stream, std::string* err) {
  const int64_t total = rows * ((c + 31) / 32);
  if (total == 0) return 0;
  elt::unpack_kernel<<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(packed, rows, c, bits,
                                                                            row_bytes_of(c, bits), is_signed, out);
  return check_launch("unpack launch", err);
}

int launch_prepare_weights(const uint8_t* w_packed, int32_t w_bits, int32_t w_format, const WeightGeom& g,
                           uint8_t* out, cudaStream_t stream, std::string* err) {
  const int max_abs = (w_format == 0) ? (1 << (w_bits - 1)) : ((1 << w_bits) - 1);
  const int mode = max_abs <= 15 ? 1 : ((w_bits == 8 && w_format == 0) ? 2 : 0);
  const int64_t e4_rows = mode == 2 ? g.split_rows : g.cout_pad;
  const int64_t total = e4_rows * g.k_pad + (int64_t)g.cout * g.k_total;
  elt::prepare_weights_kernel<<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(
      w_packed, w_bits, w_format, g, row_bytes_of(g.cin, w_bits), mode, out);
  if (const int st = check_launch("prepare_weights launch", err)) return st;
  if (fp4_weights(w_bits, w_format)) {
    const int64_t n4 = (int64_t)g.cout_pad * (g.k_pad / 2);
    elt::prepare_fp4_kernel<<<elt::blocks_for(n4), elt::kThreads, 0, stream>>>(
        w_packed, w_bits, w_format, g, row_bytes_of(g.cin, w_bits), out);
    return check_launch("prepare_weights (fp4) launch", err);
  }
  return 0;
}

}  // namespace aqd
