// common.cuh -- device helpers shared by libaqd's kernels: the packed-code layout and
// the integer epilogue of AQD (Eq. 6 bias, Eq. 7/8 skip, Eq. 2 rescale + clip).
#pragma once
#include <cstdint>

namespace aqd {

enum : uint32_t {
  kStatusOk = 0,
  kStatusTimeout = 4,
  kStatusDeviceCheck = 5,
};

// ---------------------------------------------------------------- integer epilogue

__device__ __forceinline__ int64_t sat32(int64_t v) {
  return v > 2147483647LL ? 2147483647LL : (v < -2147483648LL ? -2147483648LL : v);
}

// round half up of v / 2^r, r in [0, 62]; |v| < 2^62 so the add cannot overflow
__device__ __forceinline__ int64_t rhu(int64_t v, int r) {
  return r == 0 ? v : ((v + (1LL << (r - 1))) >> r);
}

// Per-output-channel epilogue constants (one level's row of the tables).
struct EpiChan {
  int32_t bias;
  int32_t m0;
  int32_t c;      // skip multiplier of Eq. 8
  int8_t r;       // total requant right shift, 31 + shift
  int8_t d;       // skip shift of Eq. 8
  int16_t pad_;
};

// Eq. 6 -> Eq. 7 -> Eq. 2 for one accumulator value.
// out_bits == 32 returns sat32 of the BN/skip sum; else the clipped k-bit code.
template <bool kHasSkip>
__device__ __forceinline__ int32_t epilogue(int64_t acc, int64_t skip, const EpiChan& p,
                                            int scale_main, int out_bits) {
  int64_t t = acc + (int64_t)p.bias;
  if (kHasSkip) {
    if (scale_main == 0) t += rhu(skip * (int64_t)p.c, p.d);
    else t = rhu(sat32(t) * (int64_t)p.c, p.d) + skip;
  }
  int64_t u = sat32(t);
  if (out_bits == 32) return (int32_t)u;
  int64_t v = rhu(u * (int64_t)p.m0, p.r);
  int64_t hi = (1LL << out_bits) - 1;
  return (int32_t)(v < 0 ? 0 : (v > hi ? hi : v));
}

// ---------------------------------------------------------------- maxima of packed codes

// Max-pooling on codes (Sec. 3.2.4). Codes of 2, 4 or 8 bits sit in aligned kBits-bit fields of
// each 32-bit word, so w & (M << kBits j), M = (2^kBits - 1) * 0x00010001, j < 16 / kBits, are
// 16 / kBits planes of two codes each, one per 16-bit half, in place: as unsigned 16-bit
// numbers they order like the codes, so a packed 16-bit maximum (three inputs at a time) is
// the maximum of two channels, and the maxima of all planes OR back into one word. The top
// plane needs no mask before the maximum: unsigned 16-bit halves order first by their top
// field, so the maximum of the raw halves carries the maximum top code (masked once at the
// end). PoolAcc holds the planes of one word.
template <int kBits>
struct PoolAcc {
  static constexpr int kPlanes = 16 / kBits;
  static constexpr uint32_t kM = ((1u << kBits) - 1u) * 0x00010001u;
  static constexpr uint32_t kTop = kM << (kBits * (kPlanes - 1));
  uint32_t p[kPlanes];
  static __device__ __forceinline__ uint32_t plane(uint32_t w, int j) {
    return j == kPlanes - 1 ? w : w & (kM << (kBits * j));
  }
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) p[j] = 0u;  // codes are >= 0
  }
  __device__ __forceinline__ void add(uint32_t w) {
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) p[j] = __vimax3_u16x2(p[j], plane(w, j), 0u);
  }
  __device__ __forceinline__ void add2(uint32_t w0, uint32_t w1) {
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) p[j] = __vimax3_u16x2(p[j], plane(w0, j), plane(w1, j));
  }
  // the maximum of three words' planes (replaces the contents)
  __device__ __forceinline__ void set3(uint32_t w0, uint32_t w1, uint32_t w2) {
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) p[j] = __vimax3_u16x2(plane(w0, j), plane(w1, j), plane(w2, j));
  }
  // this = max(this, a, b), plane by plane
  __device__ __forceinline__ void max3(const PoolAcc& a, const PoolAcc& b) {
#pragma unroll
    for (int j = 0; j < kPlanes; ++j) p[j] = __vimax3_u16x2(p[j], a.p[j], b.p[j]);
  }
  __device__ __forceinline__ uint32_t word() const {
    uint32_t o = p[kPlanes - 1] & kTop;
#pragma unroll
    for (int j = 0; j < kPlanes - 1; ++j) o |= p[j];
    return o;
  }
};

// ---------------------------------------------------------------- packed layout
// A group = 32 consecutive channels of one pixel row: 4*bits bytes for bits 2/3/4/8.
// bits 2/4/8: word w holds channels [w*q, (w+1)*q), q = 32/bits, channel i of the word
// at bit 8*(i%4) + bits*(i/4). bits 3: two 2-bit words (low bits) + one word of bit 2.

__host__ __device__ __forceinline__ int group_bytes(int bits) { return 4 * bits; }

// Unpack one 32-channel group into 8 words of 4 byte-lane codes each:
// out[j] holds channels 4j..4j+3 in bytes 0..3 (values 0..2^bits-1).
template <int kBits>
__device__ __forceinline__ void unpack_group_bytes(const uint32_t* g, uint32_t out[8]) {
  if constexpr (kBits == 2) {
#pragma unroll
    for (int w = 0; w < 2; ++w)
#pragma unroll
      for (int j = 0; j < 4; ++j) out[4 * w + j] = (g[w] >> (2 * j)) & 0x03030303u;
  } else if constexpr (kBits == 4) {
#pragma unroll
    for (int w = 0; w < 4; ++w)
#pragma unroll
      for (int j = 0; j < 2; ++j) out[2 * w + j] = (g[w] >> (4 * j)) & 0x0F0F0F0Fu;
  } else if constexpr (kBits == 3) {
#pragma unroll
    for (int w = 0; w < 2; ++w)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint32_t lo = (g[w] >> (2 * j)) & 0x03030303u;
        uint32_t hi = ((g[2] >> (4 * w + j)) & 0x01010101u) << 2;
        out[4 * w + j] = lo | hi;
      }
  } else {  // 8
#pragma unroll
    for (int j = 0; j < 8; ++j) out[j] = g[j];
  }
}

// Pack 32 codes (already clipped to [0, 2^bits-1]) into one group.
template <int kBits>
__device__ __forceinline__ void pack_group(const int32_t v[32], uint32_t g[8]) {
  if constexpr (kBits == 2 || kBits == 4 || kBits == 8) {
    constexpr int q = 32 / kBits;
#pragma unroll
    for (int w = 0; w < kBits; ++w) {
      uint32_t word = 0;
#pragma unroll
      for (int i = 0; i < q; ++i) word |= ((uint32_t)v[w * q + i]) << (8 * (i % 4) + kBits * (i / 4));
      g[w] = word;
    }
  } else {  // 3
#pragma unroll
    for (int w = 0; w < 2; ++w) {
      uint32_t word = 0;
#pragma unroll
      for (int i = 0; i < 16; ++i) word |= ((uint32_t)v[16 * w + i] & 3u) << (8 * (i % 4) + 2 * (i / 4));
      g[w] = word;
    }
    uint32_t hw = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) hw |= (((uint32_t)v[i] >> 2) & 1u) << (8 * (i % 4) + (i / 4));
    g[2] = hw;
  }
}

// Runtime-bits dispatch helpers (elementwise kernels).
__device__ __forceinline__ void unpack_group_vals(const uint8_t* src, int bits, bool is_signed,
                                                  int32_t v[32]) {
  uint32_t g[8];
  const int nw = bits;  // words per group = 4*bits bytes / 4
#pragma unroll
  for (int i = 0; i < 8; ++i) g[i] = (i < nw) ? reinterpret_cast<const uint32_t*>(src)[i] : 0u;
  uint32_t b[8];
  switch (bits) {
    case 2: unpack_group_bytes<2>(g, b); break;
    case 3: unpack_group_bytes<3>(g, b); break;
    case 4: unpack_group_bytes<4>(g, b); break;
    default: unpack_group_bytes<8>(g, b); break;
  }
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    int32_t x = (int32_t)((b[i / 4] >> (8 * (i % 4))) & 0xFFu);
    if (is_signed && (x >> (bits - 1)) & 1) x -= (1 << bits);
    v[i] = x;
  }
}

__device__ __forceinline__ void pack_group_vals(const int32_t v[32], int bits, uint32_t g[8]) {
  int32_t m[32];
  const int32_t mask = (1 << bits) - 1;
#pragma unroll
  for (int i = 0; i < 32; ++i) m[i] = v[i] & mask;
  switch (bits) {
    case 2: pack_group<2>(m, g); break;
    case 3: pack_group<3>(m, g); break;
    case 4: pack_group<4>(m, g); break;
    default: pack_group<8>(m, g); break;
  }
}

__device__ __forceinline__ void store_group(uint8_t* dst, const uint32_t g[8], int bits) {
  uint32_t* d = reinterpret_cast<uint32_t*>(dst);
  if (bits == 2) {
    *reinterpret_cast<uint2*>(d) = make_uint2(g[0], g[1]);
  } else if (bits == 4) {
    *reinterpret_cast<uint4*>(d) = make_uint4(g[0], g[1], g[2], g[3]);
  } else if (bits == 8) {
    reinterpret_cast<uint4*>(d)[0] = make_uint4(g[0], g[1], g[2], g[3]);
    reinterpret_cast<uint4*>(d)[1] = make_uint4(g[4], g[5], g[6], g[7]);
  } else {
    d[0] = g[0]; d[1] = g[1]; d[2] = g[2];
  }
}

// Value of channel ch of a packed/int32 row (slow path for odd channel counts).
__device__ __forceinline__ int32_t read_code(const uint8_t* row, int ch, int bits, bool is_signed) {
  if (bits == 32) return reinterpret_cast<const int32_t*>(row)[ch];
  if (bits == 8) {
    int32_t x = row[ch];
    return (is_signed && x >= 128) ? x - 256 : x;
  }
  const uint8_t* grp = row + (ch / 32) * group_bytes(bits);
  int i = ch % 32;
  uint32_t x;
  if (bits == 3) {
    const uint32_t* g = reinterpret_cast<const uint32_t*>(grp);
    int il = i % 16;
    uint32_t lo = (g[i / 16] >> (8 * (il % 4) + 2 * (il / 4))) & 3u;
    uint32_t hi = (g[2] >> (8 * (i % 4) + i / 4)) & 1u;
    x = lo | (hi << 2);
  } else {
    const int q = 32 / bits;
    const uint32_t* g = reinterpret_cast<const uint32_t*>(grp);
    int w = i / q, j = i % q;
    x = (g[w] >> (8 * (j % 4) + bits * (j / 4))) & ((1u << bits) - 1u);
  }
  int32_t v = (int32_t)x;
  if (is_signed && (v >> (bits - 1)) & 1) v -= (1 << bits);
  return v;
}

__host__ __device__ __forceinline__ int64_t row_bytes_of(int c, int bits) {
  if (c <= 0) return -1;
  if (bits == 32) return 4LL * c;
  if (bits == 8) return c;
  if (bits == 2 || bits == 3 || bits == 4) return (c % 32) ? -1 : (int64_t)(c / 32) * 4 * bits;
  return -1;
}

}  // namespace aqd
