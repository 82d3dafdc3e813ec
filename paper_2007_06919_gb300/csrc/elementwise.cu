// elementwise.cu -- the element-wise parts of AQD's integer inference path:
//   * requant (Eq. 6 bias + Eq. 2 fixed-point rescale and clip) of an int32 tensor,
//   * the integer skip add of Eq. 7 with Eq. 8's dyadic factor (optionally reading the
//     skip through a nearest 2x upsample, the FPN top-down add),
//   * max-pooling directly on codes (Sec. 3.2.4),
//   * code packing / unpacking and the one-time weight preparation.
// One thread handles one pixel's 32-channel group, so loads and stores are whole
// packed groups (8/12/16/32 bytes, or 128 bytes of int32).
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace aqd {
namespace elt {

constexpr int kThreads = 256;

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
// monotone quantizer, so it runs on the codes). In these layouts every byte holds 8/bits
// codes at bit offsets 0, bits, 2 bits, ..., each of a different channel, so the per-channel
// maximum is a byte-wise maximum (__vmaxu4) of each bit plane. One thread owns kVec words of
// one output pixel's row; window taps outside the input are skipped (codes are >= 0 and the
// padding is smaller than the window, so every window holds a tap).
template <int kBits, int kVec>
__global__ void __launch_bounds__(kThreads) maxpool_packed_kernel(const PoolArgs a) {
  constexpr int kPlanes = 8 / kBits;
  constexpr uint32_t kMask = kBits == 8 ? 0xFFFFFFFFu : (kBits == 4 ? 0x0F0F0F0Fu : 0x03030303u);
  const int64_t units = a.row_bytes / (4 * kVec);
  const int64_t total = (int64_t)a.n * a.ho * a.wo * units;
  const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
  if (t >= total) return;
  const int64_t pix = t / units;
  const int u = (int)(t - pix * units);
  const int hw = a.ho * a.wo;
  const int img = (int)(pix / hw);
  const int rem = (int)(pix - (int64_t)img * hw);
  const int oh = rem / a.wo, ow = rem - oh * a.wo;
  uint32_t acc[kVec][kPlanes];
#pragma unroll
  for (int v = 0; v < kVec; ++v)
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) acc[v][j] = 0u;
  for (int r = 0; r < a.k; ++r) {
    const int hi = oh * a.stride - a.pad + r;
    if (hi < 0 || hi >= a.h) continue;
    for (int s = 0; s < a.k; ++s) {
      const int wi = ow * a.stride - a.pad + s;
      if (wi < 0 || wi >= a.w) continue;
      const uint32_t* src = reinterpret_cast<const uint32_t*>(
          a.x + (((int64_t)img * a.h + hi) * a.w + wi) * a.row_bytes) + u * kVec;
      uint32_t w[kVec];
      if constexpr (kVec == 4) {
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(src));
        w[0] = q.x; w[1] = q.y; w[2] = q.z; w[3] = q.w;
      } else {
#pragma unroll
        for (int v = 0; v < kVec; ++v) w[v] = __ldg(src + v);
      }
#pragma unroll
      for (int v = 0; v < kVec; ++v)
#pragma unroll
        for (int j = 0; j < kPlanes; ++j) acc[v][j] = __vmaxu4(acc[v][j], (w[v] >> (kBits * j)) & kMask);
    }
  }
  uint32_t o[kVec];
#pragma unroll
  for (int v = 0; v < kVec; ++v) {
    o[v] = 0u;
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) o[v] |= acc[v][j] << (kBits * j);
  }
  uint32_t* dst = reinterpret_cast<uint32_t*>(a.y + pix * a.row_bytes) + u * kVec;
  if constexpr (kVec == 4) {
    *reinterpret_cast<uint4*>(dst) = make_uint4(o[0], o[1], o[2], o[3]);
  } else {
#pragma unroll
    for (int v = 0; v < kVec; ++v) dst[v] = o[v];
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

int launch_elementwise(const EltArgs& a, cudaStream_t stream, std::string* err) {
  const int64_t total = (int64_t)a.n * a.h * a.w * ((a.c + 31) / 32);
  if (total == 0) return 0;
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
    const int64_t total = pixels * (a.row_bytes / (v4 ? 16 : 4));
    const int blocks = elt::blocks_for(total);
    if (a.bits == 2) {
      if (v4) elt::maxpool_packed_kernel<2, 4><<<blocks, elt::kThreads, 0, stream>>>(a);
      else elt::maxpool_packed_kernel<2, 1><<<blocks, elt::kThreads, 0, stream>>>(a);
    } else if (a.bits == 4) {
      if (v4) elt::maxpool_packed_kernel<4, 4><<<blocks, elt::kThreads, 0, stream>>>(a);
      else elt::maxpool_packed_kernel<4, 1><<<blocks, elt::kThreads, 0, stream>>>(a);
    } else {
      if (v4) elt::maxpool_packed_kernel<8, 4><<<blocks, elt::kThreads, 0, stream>>>(a);
      else elt::maxpool_packed_kernel<8, 1><<<blocks, elt::kThreads, 0, stream>>>(a);
    }
    return check_launch("maxpool launch", err);
  }
  const int64_t total = pixels * ((a.c + 31) / 32);
  elt::maxpool_kernel<<<elt::blocks_for(total), elt::kThreads, 0, stream>>>(a);
  return check_launch("maxpool launch", err);
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
