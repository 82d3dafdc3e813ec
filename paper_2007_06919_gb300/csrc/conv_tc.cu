// conv_tc.cu -- AQD's integer convolution (Eq. 4) as a persistent tcgen05 implicit GEMM
// on sm_103a, with the integer epilogue (Eq. 6 bias, Eq. 7/8 skip, Eq. 2 rescale + clip)
// fused after the TMEM accumulator.
//
// Exact integer arithmetic on the FP8 tensor pipe. sm_103a has no integer tcgen05 MMA
// (kind::i8), so codes are embedded in E4M3 bit patterns: the raw byte n (0..15) of an
// E4M3 value is exactly n * 2^-9 (0..7 subnormal, 8..15 exponent field 1), and a signed
// weight |w| <= 15 is the same byte with the sign bit set. Every product is an integer
// times 2^-18, and the FP32 accumulator holds the exact integer sum times 2^-18 as long as
// K * max|x| * max|w| < 2^24, which the host checks before choosing this kernel.
//
// 2-bit codes on the FP4 pipe (kFp4): E2M1 holds n / 2 exactly for n <= 4, so a code n and a
// weight |w| <= 4 become the E2M1 values n / 2 and w / 2 (raw nibbles n and sign | |w|), every
// product is an integer / 4, and kind::mxf4nvf4 (K = 64 per instruction, one UE8M0 scale
// per 32 K elements, all set to 2^0 in TMEM) accumulates the exact integer sum / 4 in FP32.
// Operands are nibble images (two codes per byte), so a 128-byte K chunk holds 256 codes. A
// nibble image keeps the byte image's row stride (cin bytes) and fills the first cin / 2
// bytes of each row, so its zero border lies where a byte image's does in the same workspace.
//
// Per CTA (one per SM, persistent over tiles of 128 output pixels x BN channels):
//   warps 0..E-1  epilogue (E = 4 or 8): tcgen05.ld of the accumulator, integer epilogue,
//              bit-pack, store (warp w reads TMEM lanes 32*(w%4)..; with 8 warps each takes
//              every other 32-column group)
//   warp  E    TMEM allocation + one thread issuing tcgen05.mma (kind::f8f6f4, M=128)
//   warp  E+1  one thread loading prepared weights with TMA (cp.async.bulk.tensor, SW128)
//   warps E+2..E+5 activation producers: im2col gather of packed k-bit codes with cp.async
//              (zero-fill = the padding code 0), unpack to E4M3 bytes, store into the
//              128B-swizzled K-major operand layout, signal an mbarrier
// Stages of 128 K-bytes (one 128B swizzle atom) circulate between producers and the MMA
// thread; two TMEM accumulators let the epilogue of tile i overlap the MMAs of tile i+1.
// Every wait is bounded: on expiry the CTA latches kStatusTimeout and unwinds.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace aqd {
namespace tc {

// A tile is kSub M=128 sub-tiles (each one MMA per k-step) sharing every weight stage.
// The MMA rate is full only for N = 256 (measured: two N=128 MMAs sharing B reach ~72%,
// one N=128 MMA ~31%), so tiles are 128 x 256 (kSub = 1) for 256-channel layers.
#ifndef AQD_SUBTILES
#define AQD_SUBTILES 1
#endif
constexpr int kSub = AQD_SUBTILES;
constexpr int BM = 128 * kSub;     // output pixels per tile
constexpr int kSubA = 128 * 128;   // bytes of one sub-tile's A operand per stage
constexpr int kStageA = kSub * kSubA; // bytes of A per stage
constexpr int BK = 128;            // K bytes per stage
#ifndef AQD_EPI_WARPS
#define AQD_EPI_WARPS 8
#endif
constexpr int kEpiWarps = AQD_EPI_WARPS;  // 4 or 8
static_assert(kEpiWarps == 4 || kEpiWarps == 8, "epilogue warps: 4 or 8");
constexpr int kEpiThreads = kEpiWarps * 32;
#ifndef AQD_TMA_WARPS
#define AQD_TMA_WARPS 1
#endif
constexpr int kTmaWarps = AQD_TMA_WARPS;  // weight-loading warps, alternating K chunks
constexpr int kWarpMma = kEpiWarps;
constexpr int kWarpTma = kEpiWarps + 1;
constexpr int kWarpProd0 = kEpiWarps + 1 + kTmaWarps;
constexpr int kProdWarps = 4 * kSub;  // one thread per tile row
constexpr int kThreads = (kWarpProd0 + kProdWarps) * 32;
// The expanded-activation ("flat") variant has no producer warps: TMA loads both operands,
// two boxes per K chunk. One issuing thread sustains about one box per ~700 cycles
// (measured), so that variant spreads the chunks over kTmaWarpsFlat threads.
constexpr int kTmaWarpsFlat = 3;
__host__ __device__ constexpr int tma_warps(bool flat) { return flat ? kTmaWarpsFlat : kTmaWarps; }
__host__ __device__ constexpr int threads_for(bool flat) { return flat ? (kWarpTma + kTmaWarpsFlat) * 32 : kThreads; }
constexpr int kMaxStages = 16;
constexpr int kStageRow = 36;  // words per row of an int32 staging block (16-byte aligned, conflict-free)
constexpr int kQTab = 256;  // K-chunk table entries (larger K falls back to division)

// One layer of a launch: its per-channel tables, the packed output of each job and the
// zero-padded byte image its epilogue writes for the next layer (NULL: none).
struct LayerDev {
  const int32_t* m0;
  const int8_t* shift;
  const int32_t* bias;
  uint8_t* y[kMaxJobs];
  uint8_t* ws_out;
  int32_t ws_nib;  // ws_out holds two 2-bit codes per byte (the next layer runs on the FP4 pipe)
};

// The tensor maps of a launch: the weights of each layer, the weights with half-height
// boxes (half-width tiles), and the two byte images that chained layers read in turn.
struct Maps {
  CUtensorMap w[kMaxLayers];
  CUtensorMap wh;
  CUtensorMap a[2];
};

struct Params {
  ConvJobDev jobs[kMaxJobs];
  int32_t njobs, total_tiles, n_tiles, num_kchunks;
  int32_t cin, cout, kh, kw, stride, pad, k_total;
  int32_t out_bits, skip_bits;
  int64_t x_row_bytes, y_row_bytes, skip_row_bytes;
  const int32_t* skip_c;
  const int8_t* skip_d;
  int32_t upsample, scale_main, has_skip;
  int32_t bn, stages, tmem_cols;
  int32_t acc_small;  // |acc| < 2^22 guaranteed by K * max|x| * max|w|
  int32_t cin_chunks; // cin / 128 (flat path)
  int32_t dp_tiles;   // tiles [0, dp_tiles) are bn wide; later ones are the two bn/2 halves
  int32_t contig;     // each CTA takes one contiguous range of tiles (single CTAs, one layer,
                      // no half tiles) instead of every gridDim-th tile
                      // of the remaining full tiles (the last, partial wave)
  uint32_t off_b, off_epi, off_bar, off_qtab;
  uint32_t off_ostage;  // int32 outputs: per-warp staging blocks for row-contiguous stores (0: none)
  int32_t out_pad;
  int32_t a_planes;   // K runs over this many planes of the byte image (2: 8-bit activations)
  int32_t plane_rows; // workspace rows per plane
  int32_t split_w;    // weights in the split layout: a tile's bn B rows give bn/2 channels
  uint32_t* status;
  // Several chained stride-1 layers of one shape in one launch (workspace path, CTA pairs,
  // one N tile, no half-width tiles): layer l covers the tiles [l * layer_tiles, (l + 1) *
  // layer_tiles), in that order over the persistent CTAs. Tile t of layer l reads the
  // previous layer's output rows written by its tiles t - K .. t + K of the same image
  // (K = 1 + wp / 256), which are also the only tiles of that layer that read the rows tile
  // t writes. Each epilogue warp of a tile of layer l < nlayers - 1 adds 1 to
  // dep[l * layer_tiles + t] (release) after its stores; the TMA issuers of a tile of layer
  // l > 0 wait (acquire, bounded) for dep[(l - 1) * layer_tiles + t'] >= dep_target on those
  // tiles before loading A.
  int32_t nlayers, layer_tiles;
  LayerDev layers[kMaxLayers];
  int32_t sf_col;     // FP4: first of the 32 TMEM columns that hold the unit block scales
  uint32_t* dep;
  uint32_t dep_target;
};

static_assert(kSubA == kMmaM * BK, "one sub-tile is one M=128 MMA operand");

// ---------------------------------------------------------------- tile bookkeeping

struct TileInfo {
  int layer;
  int job, mt;
  int bn;    // MMA N of this tile (weight rows): p.bn, or p.bn / 2 for a half tile
  int col0;  // first output channel
  int brow;  // first weight row
  int cn;    // output channels of this tile: bn, or bn / 2 with split weights
};
// Flat path: M tile mt of a job covers virtual rows [v0, v0 + 128) of image img, where the
// virtual grid holds the output rows at the padded input width wp (stride 1).
struct FlatTile {
  int img, v0;
};
__device__ __forceinline__ FlatTile flat_tile(const ConvJobDev& jb, int mt, int rows = 128) {
  FlatTile f;
  f.img = mt / jb.tpi;
  f.v0 = (mt - f.img * jb.tpi) * rows;
  return f;
}
// Waits until every tile of layer l - 1 that writes the rows M tile mt of job j (of layer l)
// reads has been stored (see Params::dep), then orders those stores before this thread's TMA
// loads. kTileRows: rows of a tile (every layer of a launch has the same tiles).
template <int kTileRows>
__device__ __forceinline__ bool wait_dep_tiles(const Params& p, int l, int j, int mt, volatile int* abort_flag) {
  const ConvJobDev& jb = p.jobs[j];
  const int img = mt / jb.tpi, m_in = mt - img * jb.tpi;
  const int K = 1 + jb.wp / kTileRows;
  const int lo = m_in - K < 0 ? 0 : m_in - K;
  const int hi = m_in + K > jb.tpi - 1 ? jb.tpi - 1 : m_in + K;
  const uint32_t* c = p.dep + (size_t)(l - 1) * p.layer_tiles + jb.tile_begin + img * jb.tpi;
  if (!counters_wait(c + lo, hi - lo + 1, p.dep_target, abort_flag)) return false;
  fence_proxy_async_global();
  return true;
}

// Global tile t -> (job, M tile, channel range). Tiles past dp_tiles split the remaining
// full tiles into two halves of N, so the last, partial wave covers more SMs.
__device__ __forceinline__ TileInfo tile_info(const Params& p, int t) {
  const int layer = p.nlayers > 1 ? t / p.layer_tiles : 0;
  t -= layer * p.layer_tiles;
  int half = -1;
  if (t >= p.dp_tiles) {
    const int h = t - p.dp_tiles;
    t = p.dp_tiles + (h >> 1);
    half = h & 1;
  }
  int j = 0;
#pragma unroll 1
  while (j + 1 < p.njobs && t >= p.jobs[j + 1].tile_begin) ++j;
  int local = t - p.jobs[j].tile_begin;
  TileInfo ti;
  ti.layer = layer;
  ti.job = j;
  ti.mt = local / p.n_tiles;
  const int nt = local - ti.mt * p.n_tiles;
  ti.bn = half < 0 ? p.bn : p.bn / 2;
  ti.brow = nt * p.bn + (half > 0 ? p.bn / 2 : 0);
  // split weights (no half tiles): rows [brow, brow + bn/2) hold w_lo of bn/2 channels and
  // the next bn/2 rows their w_hi
  ti.cn = p.split_w ? ti.bn / 2 : ti.bn;
  ti.col0 = p.split_w ? nt * (p.bn / 2) : ti.brow;
  return ti;
}

// ---------------------------------------------------------------- epilogue, general case

// The skip values of one row's 32-channel group (Eq. 7's second operand), loaded and
// unpacked per skip width into registers: every index is static, nothing goes through
// local memory. Channels past cout read 0.
__device__ __forceinline__ void load_skip_group(const Params& p, const uint8_t* srow, int ch0, int ncols,
                                                int32_t (&sk)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) sk[i] = 0;
  {
    const int sb = p.skip_bits;
    // a whole group of 32 channels in rows whose size is a multiple of 16 bytes: 16-byte loads
    // (the tensor base is 16-byte aligned); otherwise element by element
    const bool whole = ncols == 32 && ch0 + 32 <= p.cout && (p.skip_row_bytes & 15) == 0;
    if (sb == 32 && whole) {
      const int4* s4 = reinterpret_cast<const int4*>(reinterpret_cast<const int32_t*>(srow) + ch0);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int4 v = __ldg(s4 + q);
        sk[4 * q] = v.x; sk[4 * q + 1] = v.y; sk[4 * q + 2] = v.z; sk[4 * q + 3] = v.w;
      }
    } else if (sb == 32) {
      const int32_t* s32 = reinterpret_cast<const int32_t*>(srow) + ch0;
#pragma unroll
      for (int i = 0; i < 32; ++i) sk[i] = (i < ncols && ch0 + i < p.cout) ? __ldg(s32 + i) : 0;
    } else if (sb == 8 && whole) {
      const uint4* s16 = reinterpret_cast<const uint4*>(srow + ch0);
      const uint4 a = __ldg(s16), b = __ldg(s16 + 1);
      const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 32; ++i) sk[i] = (int32_t)((w[i / 4] >> (8 * (i % 4))) & 0xFFu);
    } else if (sb == 8) {
      const uint8_t* s8 = srow + ch0;
#pragma unroll
      for (int i = 0; i < 32; ++i) sk[i] = (i < ncols && ch0 + i < p.cout) ? (int32_t)__ldg(s8 + i) : 0;
    } else {
      // 2/3/4-bit codes: one whole packed group (the layout needs cout % 32 == 0)
      const uint32_t* g32 = reinterpret_cast<const uint32_t*>(srow + (ch0 >> 5) * group_bytes(sb));
      uint32_t g[4] = {0u, 0u, 0u, 0u};
      if (sb == 4) {  // 16-byte groups at 16-byte offsets
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(g32));
        g[0] = v.x; g[1] = v.y; g[2] = v.z; g[3] = v.w;
      } else if (sb == 2) {
        const uint2 v = __ldg(reinterpret_cast<const uint2*>(g32));
        g[0] = v.x; g[1] = v.y;
      } else {
        g[0] = __ldg(g32); g[1] = __ldg(g32 + 1); g[2] = __ldg(g32 + 2);
      }
      uint32_t b[8];
      if (sb == 2) unpack_group_bytes<2>(g, b);
      else if (sb == 3) unpack_group_bytes<3>(g, b);
      else unpack_group_bytes<4>(g, b);
#pragma unroll
      for (int i = 0; i < 32; ++i) sk[i] = (int32_t)((b[i / 4] >> (8 * (i % 4))) & 0xFFu);
    }
  }
}

// Eq. 6 -> Eq. 7 -> Eq. 2 in int64 for 32 accumulators of one row (any shift, any skip),
// element by element as the definition states it; the common cases take 32-bit forms.
// (sc: the FP32 accumulator holds the integer sum / sc: 2^18 on the E4M3 pipe, 4 on the FP4 one)
template <bool kSkip, bool kIntAcc = false>
__device__ __forceinline__ void general_group(const Params& p, const uint32_t* v, const EpiChan* ep,
                                              const uint8_t* srow, int ch0, int ncols, float sc, int32_t (&out)[32]) {
  int32_t sk[32];
  if (kSkip) load_skip_group(p, srow, ch0, ncols, sk);
  else {
#pragma unroll
    for (int i = 0; i < 32; ++i) sk[i] = 0;
  }
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    // v: FP32 accumulators of exact integers x 2^-18, or (kIntAcc) int32 sums already
    const int64_t acc = kIntAcc ? (int64_t)(int32_t)v[i]
                                : (int64_t)__float2int_rn(__uint_as_float(v[i]) * sc);
    const EpiChan ec = ep[i];
    out[i] = kSkip ? epilogue<true>(acc, sk[i], ec, p.scale_main, p.out_bits)
                        : epilogue<false>(acc, 0, ec, p.scale_main, p.out_bits);
  }
}

// In the 32-bit forms below, Eq. 2's clip to [0, qmax] is __vimin_s32_relu(x, qmax) =
// max(min(x, qmax), 0), one min.relu instruction instead of a min and a max.

// Skip epilogue in 32-bit arithmetic (Eq. 6, Eq. 7 with the skip rescaled, Eq. 2) when, for
// every column of the tile, R = 31 + shift >= 33, |bias| <= 2^30 and d >= 8, and the skip
// holds k-bit codes (s <= 255): then rhu(s * c, d) = (s * c + 2^(d-1)) >> d fits in int32,
// acc + bias cannot overflow (|acc| < 2^24), and one saturating add gives sat32 of the
// exact sum; the requant is the same 32-bit form as fast_requant_group.
// (y may be sk itself: element i is read before it is written)
__device__ __forceinline__ void fast_skip_group(const uint32_t* v, const EpiChan* ep, const int32_t (&sk)[32],
                                                int qmax, float sc, int32_t (&y)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const EpiChan c = ep[i];
    const int32_t acc = __float2int_rn(__uint_as_float(v[i]) * sc);  // exact integer
    const int64_t sc = (int64_t)sk[i] * (int64_t)c.c;
    const int32_t st = (int32_t)((sc + (1LL << (c.d - 1))) >> c.d);
    const int32_t u = add_sat(acc + c.bias, st);
    const int r = c.r;
    y[i] = __vimin_s32_relu((__mulhi(u, c.m0) + (1 << (r - 33))) >> (r - 32), qmax);
  }
}

// Skip epilogue for an int32 skip (a downsample branch in accumulator units), default
// direction, when every column has R >= 33, |bias| <= 2^30 and d >= 1: Eq. 7's rescaled skip
// rhu(s * c, d) is one 64-bit product, add and shift (|s * c| < 2^62); acc + bias fits in
// int32 (|acc| < 2^24); the sum is saturated to int32 as in Eq. 7's int64 form, and the requant
// is the 32-bit form of fast_requant_group.
__device__ __forceinline__ void fast_skip32_group(const uint32_t* v, const EpiChan* ep, const int32_t (&sk)[32],
                                                  int qmax, float sc, int32_t (&y)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const EpiChan c = ep[i];
    const int32_t acc = __float2int_rn(__uint_as_float(v[i]) * sc);  // exact integer
    const int64_t st = ((int64_t)sk[i] * (int64_t)c.c + (1LL << (c.d - 1))) >> c.d;
    int64_t t = (int64_t)(acc + c.bias) + st;
    t = t > 2147483647LL ? 2147483647LL : (t < -2147483648LL ? -2147483648LL : t);
    const int32_t u = (int32_t)t;
    const int r = c.r;
    y[i] = __vimin_s32_relu((__mulhi(u, c.m0) + (1 << (r - 33))) >> (r - 32), qmax);
  }
}

// 1.5 * 2^23: adding it to an integer-valued float |x| < 2^22 puts x in the low mantissa bits
constexpr float kMagic = 12582912.0f;
constexpr uint32_t kMagicBits = 0x4B400000u;

// Fast requant of 32 accumulators of one row into one packed group (no skip, R >= 33,
// any bias): u = sat32(acc + bias), y = clamp((mulhi(u, M0) + 2^(R-33)) >> (R-32), 0, 2^k-1).
template <int kOut>
__device__ __forceinline__ void fast_requant_group(const uint32_t* v, const EpiChan* ep, int g0, int qmax, float sc,
                                                   uint32_t gw[8]) {
#pragma unroll
  for (int w = 0; w < 8; ++w) gw[w] = 0u;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const EpiChan c = ep[g0 + i];
    const int32_t acc = __float2int_rn(__uint_as_float(v[i]) * sc);  // exact integer
    const int32_t u = add_sat(acc, c.bias);
    const int r = c.r;
    const uint32_t y = (uint32_t)__vimin_s32_relu((__mulhi(u, c.m0) + (1 << (r - 33))) >> (r - 32), qmax);
    if constexpr (kOut == 3) {
      gw[i / 16] |= (y & 3u) << (8 * (i % 4) + 2 * ((i % 16) / 4));
      gw[2] |= (y >> 2) << (8 * (i % 4) + i / 4);
    } else {
      constexpr int q = 32 / kOut;
      gw[i / q] |= y << (8 * (i % 4) + kOut * ((i % q) / 4));
    }
  }
}

// Fastest requant (no skip, R >= 33, |acc| < 2^22, |bias| <= 2^30) of 32 accumulators of one
// row, straight into 8 byte-words (word j holds channels 4j..4j+3, one code per byte: the
// layout of the chained byte image, and one step from every packed layout). One FMA turns
// the accumulator float acc / sc into the int32 acc + 0x4B400000; c.x holds
// bias - 0x4B400000, so one add gives acc + bias exactly (no int32 overflow under the stated
// bounds); c.y, c.z, c.w are M0, 2^(R-33) and R-32.
__device__ __forceinline__ void magic_requant_bytes(const uint32_t* v, const int4* f, int qmax, float sc,
                                                    uint32_t (&bw)[8]) {
#pragma unroll
  for (int j = 0; j < 8; ++j) bw[j] = 0u;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int4 c = f[i];
    const int32_t u = __float_as_int(__fmaf_rn(__uint_as_float(v[i]), sc, kMagic)) + c.x;
    const uint32_t y = (uint32_t)__vimin_s32_relu((__mulhi(u, c.y) + c.z) >> c.w, qmax);
    bw[i / 4] += y << (8 * (i % 4));  // codes < 256: the add is an or
  }
}
// Byte-words of codes < 2^kBits -> the packed group (the layout of common.cuh: word w of the
// 2/4/8-bit layout holds its channels 4k..4k+3 in bit field k of every byte; the 3-bit layout
// is two 2-bit words of the low bits and one word of bit 2, channel i at bit 8 (i%4) + i/4).
template <int kBits>
__device__ __forceinline__ void pack_bytewords(const uint32_t (&bw)[8], uint32_t (&gw)[8]) {
  if constexpr (kBits == 8) {
#pragma unroll
    for (int j = 0; j < 8; ++j) gw[j] = bw[j];
  } else if constexpr (kBits == 4) {
#pragma unroll
    for (int w = 0; w < 4; ++w) gw[w] = bw[2 * w] | (bw[2 * w + 1] << 4);
  } else if constexpr (kBits == 2) {
#pragma unroll
    for (int w = 0; w < 2; ++w)
      gw[w] = bw[4 * w] | (bw[4 * w + 1] << 2) | (bw[4 * w + 2] << 4) | (bw[4 * w + 3] << 6);
  } else {
#pragma unroll
    for (int w = 0; w < 2; ++w)
      gw[w] = (bw[4 * w] & 0x03030303u) | ((bw[4 * w + 1] & 0x03030303u) << 2) |
              ((bw[4 * w + 2] & 0x03030303u) << 4) | ((bw[4 * w + 3] & 0x03030303u) << 6);
    uint32_t h = 0u;
#pragma unroll
    for (int j = 0; j < 8; ++j) h |= ((bw[j] >> 2) & 0x01010101u) << j;
    gw[2] = h;
  }
}
// Chained output: the 32 codes of one packed group (byte-words bw: channels 4j..4j+3 in word
// j) at their place in the zero-padded image that the next stride-1 conv (padding out_pad)
// reads: one byte per code, or, when that conv runs on the FP4 pipe (nib), two codes per byte
// (channel 2k in the low nibble of byte k) in the first half of the same row.
__device__ __forceinline__ void chain_store_bw(const Params& p, uint8_t* ws_out, int nib, const ConvJobDev& jb,
                                               int img, int oh, int ow, int ch0, const uint32_t (&bw)[8]) {
  const int row = jb.orow_off + (img * jb.ohp + oh + p.out_pad) * jb.owp + ow + p.out_pad;
  if (nib) {
    uint32_t o[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      // bytes 0 and 2 of t hold the nibble pairs (c0, c1) and (c2, c3) of a byte-word
      const uint32_t t0 = bw[2 * m] | (bw[2 * m] >> 4), t1 = bw[2 * m + 1] | (bw[2 * m + 1] >> 4);
      o[m] = __byte_perm(t0, t1, 0x6420);
    }
    *reinterpret_cast<uint4*>(ws_out + (size_t)row * p.cout + (ch0 >> 1)) = make_uint4(o[0], o[1], o[2], o[3]);
  } else {
    uint4* dst = reinterpret_cast<uint4*>(ws_out + (size_t)row * p.cout + ch0);
    dst[0] = make_uint4(bw[0], bw[1], bw[2], bw[3]);
    dst[1] = make_uint4(bw[4], bw[5], bw[6], bw[7]);
  }
}

// The same from a packed group gw of out_bits codes.
__device__ __forceinline__ void chain_store(const Params& p, uint8_t* ws_out, int nib, const ConvJobDev& jb, int img,
                                            int oh, int ow, int ch0, const uint32_t gw[8], int out_bits) {
  uint32_t o[8];
  switch (out_bits) {
    case 2: unpack_group_bytes<2>(gw, o); break;
    case 3: unpack_group_bytes<3>(gw, o); break;
    default: unpack_group_bytes<4>(gw, o); break;
  }
  chain_store_bw(p, ws_out, nib, jb, img, oh, ow, ch0, o);
}

// ---------------------------------------------------------------- the kernel

// Loads the packed codes of one 128-channel K chunk of one output row into registers
// (4 * kXBits words; group g = channels 32g..32g+31 of the chunk at words [g*kXBits, ...)).
// Taps outside the image (and rows past the end of the job) read zeros = code 0.
template <int kXBits>
struct RowCursor {
  const uint8_t* xbase;  // image base of this row's pixel
  int hb, wb, H, W;      // top-left input coordinate of the window, image size
  bool valid;
  int tr, ts, tc0;       // tap (r, s) and channel offset of the next 32-channel group
};

template <int kXBits, bool kChunkInTap>
__device__ __forceinline__ void load_chunk(const Params& p, RowCursor<kXBits>& rc, int q, uint32_t (&w)[4 * kXBits]) {
  constexpr int kGB = 4 * kXBits;
  if constexpr (kChunkInTap) {
    // cin % 128 == 0: the chunk is 128 consecutive channels of one tap
    const int hi = rc.hb + rc.tr, wi = rc.wb + rc.ts;
    const bool ok = rc.valid && hi >= 0 && hi < rc.H && wi >= 0 && wi < rc.W;
    const uint4* src = reinterpret_cast<const uint4*>(rc.xbase + ((int64_t)hi * rc.W + wi) * p.x_row_bytes +
                                                      (rc.tc0 >> 5) * kGB);
#pragma unroll
    for (int i = 0; i < kXBits; ++i) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (ok) v = __ldg(src + i);
      w[4 * i] = v.x; w[4 * i + 1] = v.y; w[4 * i + 2] = v.z; w[4 * i + 3] = v.w;
    }
    rc.tc0 += 128;
    if (rc.tc0 == p.cin) { rc.tc0 = 0; if (++rc.ts == p.kw) { rc.ts = 0; ++rc.tr; } }
  } else {
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const int k0 = q * BK + 32 * g;
      bool ok = false;
      const uint8_t* src = rc.xbase;
      if (k0 < p.k_total) {
        const int hi = rc.hb + rc.tr, wi = rc.wb + rc.ts;
        ok = rc.valid && hi >= 0 && hi < rc.H && wi >= 0 && wi < rc.W;
        src = rc.xbase + ((int64_t)hi * rc.W + wi) * p.x_row_bytes + (rc.tc0 >> 5) * kGB;
        rc.tc0 += 32;
        if (rc.tc0 == p.cin) { rc.tc0 = 0; if (++rc.ts == p.kw) { rc.ts = 0; ++rc.tr; } }
      }
      if constexpr (kXBits == 2) {
        uint2 v = make_uint2(0, 0);
        if (ok) v = __ldg(reinterpret_cast<const uint2*>(src));
        w[2 * g] = v.x; w[2 * g + 1] = v.y;
      } else if constexpr (kXBits == 4) {
        uint4 v = make_uint4(0, 0, 0, 0);
        if (ok) v = __ldg(reinterpret_cast<const uint4*>(src));
        w[4 * g] = v.x; w[4 * g + 1] = v.y; w[4 * g + 2] = v.z; w[4 * g + 3] = v.w;
      } else {
#pragma unroll
        for (int i = 0; i < 3; ++i) w[3 * g + i] = ok ? __ldg(reinterpret_cast<const uint32_t*>(src) + i) : 0u;
      }
    }
  }
}

// kSkip: the instantiation that handles a skip tensor (Eq. 7); the others carry no skip code,
// which keeps the common path's registers free.
// kSplit: the 8-bit split form (split weights combined as D1 + 16 D2 in the epilogue).
// kOStage: int32 outputs go through per-warp shared-memory staging blocks (an instantiation of
// its own, so that the other forms keep their registers)
template <int kXBits, bool kChunkInTap, bool kFlat, bool kPair, bool kSkip, bool kSplit, int kBK, bool kFp4,
          bool kOStage>
__global__ void __launch_bounds__(threads_for(kFlat), 1)
conv_tc_kernel(const __grid_constant__ Maps maps, const __grid_constant__ Params p) {
  static_assert(!kPair || kFlat, "the CTA-pair form exists for the workspace path only");
  static_assert(kBK == BK || kFlat, "64-byte K chunks exist for the workspace path only");
  static_assert(!kFp4 || (kFlat && kBK == BK && !kSplit), "the FP4 pipe reads nibble images in 128-byte chunks");
  // the FP32 accumulator holds the integer sum / kAccSc
  constexpr float kAccSc = kFp4 ? 4.0f : 262144.0f;
  // bytes of one stage's A operand: kSub sub-tiles of 128 rows x kBK bytes
  constexpr int kStA = kSub * 128 * kBK;
  constexpr int kTma = tma_warps(kFlat);
  // CTA pair: this CTA's rank; the even CTA issues the MMAs; a tile has 256 rows
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;
  const bool leader = rank == 0;
  constexpr int kTileRows = kPair ? 256 : 128;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // align by pointer arithmetic on the shared array itself (no integer round trip), so the
  // compiler keeps every access through `smem` in the shared state space (lds/sts)
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t s_a = sbase;
  const uint32_t s_b = sbase + p.off_b;
  EpiChan* epi = reinterpret_cast<EpiChan*>(smem + p.off_epi);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + p.off_bar);
  // barrier slots: full[0..S), empty[0..S), tfull[2], tempty[2], final
  const int S = p.stages;
  const uint32_t b_full = smem_u32(bars);
  const uint32_t b_empty = b_full + 8 * S;
  const uint32_t b_tfull = b_empty + 8 * S;
  const uint32_t b_tempty = b_tfull + 16;
  const uint32_t b_final = b_tempty + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x / 32;
  const int lane = threadIdx.x % 32;
  const int BN = p.bn;
  const uint32_t stage_b_bytes = (uint32_t)(kPair ? BN / 2 : BN) * kBK;  // this CTA's rows of B

  // K chunk q -> (tap row r, tap column sx, 128-channel block cb), for the TMA issuers
  uint32_t* qtab = reinterpret_cast<uint32_t*>(smem + p.off_qtab);
  for (int q = threadIdx.x; q < p.num_kchunks && q < kQTab; q += blockDim.x) {
    const int tap = q / p.cin_chunks, cb = q - tap * p.cin_chunks;
    const int r = tap / p.kw, sx = tap - r * p.kw;
    qtab[q] = ((uint32_t)r << 24) | ((uint32_t)sx << 16) | (uint32_t)cb;
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(b_full + 8 * s, kFlat ? 1 : kProdWarps + 1);  // per producer warp + TMA
      mbar_init(b_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(b_tfull + 8 * b, 1);
      mbar_init(b_tempty + 8 * b, kPair ? 2 * kEpiWarps : kEpiWarps);  // one arrive per epilogue warp
    }
    mbar_init(b_final, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kWarpMma) {
    if constexpr (kPair) {
      // one warp of each CTA of the pair allocates, collectively, the same columns in both
      asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;"
                   ::"r"(smem_u32(tmem_slot)), "r"(p.tmem_cols) : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    } else {
      asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                   ::"r"(smem_u32(tmem_slot)), "r"(p.tmem_cols) : "memory");
      asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
  }
  if (warp >= kWarpTma && warp < kWarpTma + kTma && lane == 0) {
    for (int l = 0; l < p.nlayers; ++l) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.w[l]) : "memory");
    if (p.dp_tiles < p.layer_tiles) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.wh) : "memory");
    if (kFlat) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.a[0]) : "memory");
      if (p.nlayers > 1) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&maps.a[1]) : "memory");
    }
  }
  tc_fence_before();
  __syncthreads();
  // the peer signals this CTA's barriers (and the leader's MMAs read the peer's shared
  // memory) only after both CTAs have initialised them
  if constexpr (kPair) cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  if constexpr (kFp4) {
    // unit block scales (UE8M0 127 = 2^0) in the 32 TMEM columns from sf_col, every lane of
    // both CTAs of a pair: the MMAs read the A scales from the first 16, the B scales from
    // the next 16, whatever the scale vectors' layout inside them
    if (warp < 4) {
      const uint32_t ta = tmem_base + ((uint32_t)(32 * warp) << 16) + (uint32_t)p.sf_col;
      tmem_st16_fill(ta, 0x7F7F7F7Fu);
      tmem_st16_fill(ta + 16, 0x7F7F7F7Fu);
      tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (kPair) cluster_sync();
    tc_fence_after();
  }
  // everything above overlaps the previous kernel; global memory is touched only after this
  grid_dep_wait();
  if (threadIdx.x == 0) grid_dep_launch();

  const int nk = p.num_kchunks * p.a_planes;  // K chunks, over every plane of the image
  // This CTA's tiles: every tile_stride-th from first_tile, or (contig) the range
  // [first_tile, tile_end) of a balanced split of the tiles over the grid, so that a CTA's
  // consecutive tiles are neighbours (one level's table, adjacent rows in L2)
  int first_tile = kPair ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  int tile_stride = kPair ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  int tile_end = p.total_tiles;
  if (!kPair && p.contig) {
    const int q = p.total_tiles / (int)gridDim.x, r = p.total_tiles % (int)gridDim.x;
    const int b = (int)blockIdx.x;
    first_tile = b * q + (b < r ? b : r);
    tile_end = first_tile + q + (b < r ? 1 : 0);
    tile_stride = 1;
  }

  if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && leader) {
      const uint32_t idesc_full = kFp4 ? idesc_fp4(BN, kPair ? 2 * kMmaM : kMmaM) : idesc_e4m3(BN, kPair ? 2 * kMmaM : kMmaM);
      const uint32_t idesc_half =
          kFp4 ? idesc_fp4(BN / 2, kPair ? 2 * kMmaM : kMmaM) : idesc_e4m3(BN / 2, kPair ? 2 * kMmaM : kMmaM);
      const uint32_t sfa = tmem_base + (uint32_t)p.sf_col, sfb = sfa + 16;  // (FP4 only)
      // descriptors of stage 0, k-step 0; later stages / sub-tiles / k-steps add
      // (byte offset >> 4) to the 14-bit start-address field (shared addresses < 2^18)
      // the descriptors' high words are constant; stages / sub-tiles / k-steps only move the
      // 14-bit start-address field in the low word (shared addresses < 2^18, no carry)
      const uint64_t da0 = sdesc_k<kBK>(s_a), db0 = sdesc_k<kBK>(s_b);
      const uint32_t a_lo0 = (uint32_t)da0, b_lo0 = (uint32_t)db0;
      const uint32_t a_hi = (uint32_t)(da0 >> 32), b_hi = (uint32_t)(db0 >> 32);
      uint32_t it = 0, lt = 0, s = 0, ph = 0;
      bool ok = true;
      bool next_ready = false;  // the stage after the current one is known to be full
      for (int t = first_tile; t < tile_end && ok; t += tile_stride, ++lt) {
        const uint32_t buf = lt & 1;
        // (half-width tiles are counted within a layer; a launch of several layers has none)
        const int t_in_layer = p.nlayers > 1 ? t - (t / p.layer_tiles) * p.layer_tiles : t;
        const uint32_t idesc = t_in_layer < p.dp_tiles ? idesc_full : idesc_half;
        if (!mbar_poll(b_tempty + 8 * buf, ((lt >> 1) & 1) ^ 1, abort_flag)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d0 = tmem_base + buf * (uint32_t)(kSub * BN);  // sub-tile j at +j*BN
        for (int q = 0; q < nk; ++q, ++it) {
          // (operands written by TMA, or by producer threads followed by fence.proxy.async,
          // are ordered for the MMA by the mbarrier phase alone; tcgen05.fence is needed only
          // where TMEM changes hands, after the accumulator-empty wait above)
          if (!next_ready && !mbar_poll(b_full + 8 * s, ph, abort_flag)) { ok = false; break; }
          const uint32_t a_lo = a_lo0 + ((s * kStA) >> 4);
          const uint32_t b_lo = b_lo0 + ((s * stage_b_bytes) >> 4);
          const uint32_t s_next = s + 1 == (uint32_t)S ? 0u : s + 1;
          const uint32_t ph_next = s_next == 0 ? ph ^ 1u : ph;
#pragma unroll
          for (int kk = 0; kk < kBK / 32; ++kk) {
            // The tensor pipe takes about one instruction at a time, so each issue waits for
            // the previous MMA. Testing the next stage here, while the last MMAs of this
            // chunk run, lets the next chunk's first MMA follow this chunk's commit at once.
            if (kk == kBK / 32 - 1) next_ready = mbar_test(b_full + 8 * s_next, ph_next);
            const uint32_t acc = (q > 0 || kk > 0) ? 1u : 0u;
            const uint64_t db = ((uint64_t)b_hi << 32) | (b_lo + 2 * kk);
            if constexpr (kPair && kFp4) {
              mma_fp4_pair(d0, ((uint64_t)a_hi << 32) | (a_lo + 2 * kk), db, idesc, sfa, sfb, acc);
            } else if constexpr (kPair) {
              mma_e4m3_pair(d0, ((uint64_t)a_hi << 32) | (a_lo + 2 * kk), db, idesc, acc);
            } else {
#pragma unroll
              for (int j = 0; j < kSub; ++j) {
                const uint64_t da = ((uint64_t)a_hi << 32) | (a_lo + j * (kSubA >> 4) + 2 * kk);
                if constexpr (kFp4) mma_fp4(d0 + j * BN, da, db, idesc, sfa, sfb, acc);
                else mma_e4m3(d0 + j * BN, da, db, idesc, acc);
              }
            }
          }
          if constexpr (kPair) mma_commit_pair_both(b_empty + 8 * s);
          else mma_commit(b_empty + 8 * s);
          if (++s == (uint32_t)S) { s = 0; ph ^= 1; }
        }
        if (ok) {
          if constexpr (kPair) mma_commit_pair_both(b_tfull + 8 * buf);
          else mma_commit(b_tfull + 8 * buf);
        }
      }
      if (!ok) fail(abort_flag, p.status);
      // drain: every MMA issued above has completed once this barrier flips
      if constexpr (kPair) mma_commit_pair(b_final);
      else mma_commit(b_final);
      if (!mbar_wait(b_final, 0, abort_flag)) fail(abort_flag, p.status);
    }
  } else if (warp >= kWarpTma && warp < kWarpTma + kTma) {
    // ------------------------------------------------------------ weight loaders (TMA)
    // One thread of each TMA warp issues every kTmaWarps-th chunk: a thread sustains
    // about one tensor copy at a time, so two threads keep two copies in flight.
    const int tw = warp - kWarpTma;
    if (lane == 0) {
      uint32_t it = 0, s = 0, ph = 0;
      bool ok = true;
      for (int t = first_tile; t < tile_end && ok; t += tile_stride) {
        const TileInfo ti = tile_info(p, t);
        // per tile: the first workspace row of this CTA's A rows (flat path) and the image width
        int row0 = 0, wp = 0;
        if constexpr (kFlat) {
          const ConvJobDev& jb = p.jobs[ti.job];
          const FlatTile ft = flat_tile(jb, ti.mt, kTileRows);
          row0 = jb.row_off + ft.img * jb.hp * jb.wp + ft.v0 + (int)rank * 128;
          wp = jb.wp;
        }
        const CUtensorMap* wm = ti.bn == BN ? &maps.w[ti.layer] : &maps.wh;
        const CUtensorMap* am = &maps.a[ti.layer & 1];  // layers read the two images in turn
        bool deps_ready = !kFlat || ti.layer == 0;
        for (int q2 = 0; q2 < nk; ++q2, ++it, s = (s + 1 == (uint32_t)S) ? 0 : s + 1, ph ^= (s == 0)) {
          if ((int)(it % kTma) != tw) continue;
          if (!deps_ready) {
            // the previous layer's tiles that this tile reads (and that read what it writes)
            if (!wait_dep_tiles<kTileRows>(p, ti.layer, ti.job, ti.mt, abort_flag)) { ok = false; break; }
            deps_ready = true;
          }
          if (!mbar_wait(b_empty + 8 * s, ph ^ 1, abort_flag)) { ok = false; break; }
          // plane of the byte image (8-bit activations: x_lo, then 16 x_hi) and K chunk in it
          const int plane = q2 >= p.num_kchunks ? 1 : 0;
          const int q = q2 - plane * p.num_kchunks;
          const int prow = plane * p.plane_rows;
          int r, sx, cb;
          if (q < kQTab) {
            const uint32_t e = qtab[q];
            r = (int)(e >> 24); sx = (int)((e >> 16) & 255u); cb = (int)(e & 0xFFFFu);
          } else {
            const int tap = q / p.cin_chunks;
            cb = q - tap * p.cin_chunks;
            r = tap / p.kw; sx = tap - r * p.kw;
          }
          if constexpr (kPair) {
            // this CTA's 128 rows of A and its half of B; both CTAs' copies complete on the
            // leader's "full" barrier, which the leader arms with the bytes of all four
            const int row = row0 + prow + r * wp + sx;
            const int brow = ti.brow + (int)rank * (ti.bn / 2);
            const uint32_t b_bytes = (uint32_t)(ti.bn / 2) * kBK;
            if (leader) {
              mbar_arrive_expect_tx(b_full + 8 * s, 2 * (b_bytes + kStA));
              tma_load_2d(s_a + s * kStA, am, cb * kBK, row, b_full + 8 * s);
              tma_load_2d(s_b + s * stage_b_bytes, wm, q * kBK, brow, b_full + 8 * s);
            } else {
              const uint32_t fb = mapa_shared(b_full + 8 * s, 0);
              tma_load_2d_pair(s_a + s * kStA, am, cb * kBK, row, fb);
              tma_load_2d_pair(s_b + s * stage_b_bytes, wm, q * kBK, brow, fb);
            }
            continue;
          } else if constexpr (kFlat) {
            // A: 128 consecutive rows of the padded byte image, shifted by the tap (r, s)
            const int row = row0 + prow + r * wp + sx;
            mbar_arrive_expect_tx(b_full + 8 * s, (uint32_t)ti.bn * kBK + kStA);
            tma_load_2d(s_a + s * kStA, am, cb * kBK, row, b_full + 8 * s);
          } else {
            (void)r; (void)sx; (void)cb;
            mbar_arrive_expect_tx(b_full + 8 * s, (uint32_t)ti.bn * kBK);
          }
          tma_load_2d(s_b + s * stage_b_bytes, wm, q * kBK, ti.brow, b_full + 8 * s);
        }
      }
      if (!ok) fail(abort_flag, p.status);
    }
  } else if (!kFlat && warp >= kWarpProd0) {
    // ------------------------------------------------------------ activation producers
    const int row = threadIdx.x - kWarpProd0 * 32;  // 0..255: tile row owned by this thread
    const int sub = row >> 7, r7 = row & 7;
    uint8_t* arow = smem + sub * kSubA + (row & 127) * BK;
    int my_tiles = 0;
    for (int t = first_tile; t < tile_end; t += tile_stride) ++my_tiles;
    const int total = my_tiles * nk;

    RowCursor<kXBits> rc{};
    int l_tile = first_tile, l_q = 0;  // load cursor (runs kDepth chunks ahead)
    auto start_tile = [&](int t) {
      const TileInfo ti = tile_info(p, t);
      const ConvJobDev& jb = p.jobs[ti.job];
      const int m = ti.mt * BM + row;
      rc.valid = m < jb.m_total;
      const int mm = rc.valid ? m : 0;
      const int hw = jb.ho * jb.wo;
      const int img = mm / hw;
      const int rem = mm - img * hw;
      const int ho = rem / jb.wo, wo = rem - (rem / jb.wo) * jb.wo;
      rc.hb = ho * p.stride - p.pad;
      rc.wb = wo * p.stride - p.pad;
      rc.H = jb.h;
      rc.W = jb.w;
      rc.xbase = jb.x + (int64_t)img * jb.h * jb.w * p.x_row_bytes;
      rc.tr = 0; rc.ts = 0; rc.tc0 = 0;
    };
    auto load_next = [&](uint32_t (&w)[4 * kXBits]) {
      if (l_q == 0) start_tile(l_tile);
      load_chunk<kXBits, kChunkInTap>(p, rc, l_q, w);
      if (++l_q == nk) { l_q = 0; l_tile += tile_stride; }
    };
    bool ok = true;
    auto consume = [&](int c, const uint32_t (&w)[4 * kXBits]) -> bool {
      const uint32_t s = c % S, ph = (c / S) & 1;
      if (!mbar_wait(b_empty + 8 * s, ph ^ 1, abort_flag)) return false;
      uint8_t* dst = arow + (size_t)s * kStageA;
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        uint32_t o[8];
        unpack_group_bytes<kXBits>(w + g * kXBits, o);  // raw E4M3 byte = code
        *reinterpret_cast<uint4*>(dst + 16 * ((2 * g) ^ r7)) = make_uint4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<uint4*>(dst + 16 * ((2 * g + 1) ^ r7)) = make_uint4(o[4], o[5], o[6], o[7]);
      }
      fence_proxy_async();  // this thread's generic-proxy stores -> visible to the MMA
      __syncwarp();
      if (lane == 0) mbar_arrive(b_full + 8 * s);
      return true;
    };
    uint32_t w0[4 * kXBits], w1[4 * kXBits], w2[4 * kXBits];
    if (total > 0) load_next(w0);
    if (total > 1) load_next(w1);
    if (total > 2) load_next(w2);
    for (int c = 0; c < total && ok; c += 3) {
      if (!consume(c, w0)) { ok = false; break; }
      if (c + 3 < total) load_next(w0);
      if (c + 1 < total) {
        if (!consume(c + 1, w1)) { ok = false; break; }
        if (c + 4 < total) load_next(w1);
      }
      if (c + 2 < total) {
        if (!consume(c + 2, w2)) { ok = false; break; }
        if (c + 5 < total) load_next(w2);
      }
    }
    if (!ok) fail(abort_flag, p.status);
  } else {
    // ------------------------------------------------------------ epilogue (warps 0..E-1)
    // Warp w reads TMEM lanes 32*(w%4).. (the hardware lane quarter of its warp index).
    // Warp group gi = w/4 takes sub-tiles / column groups in turn, so with 8 warps two
    // warps share each lane quarter.
    const int quarter = warp & 3;
    const int gi = warp >> 2;
    constexpr int kGroups = kEpiWarps / 4;
    const int et = threadIdx.x;  // 0 .. kEpiThreads-1
    const uint32_t lane_base = tmem_base + ((uint32_t)(quarter * 32) << 16);
    const int4* epf = reinterpret_cast<const int4*>(epi + 256);  // per-column fast constants
    uint32_t lt = 0;
    bool ok = true;
    const int out_bits = p.out_bits;
    const int qmax = (1 << (out_bits & 15)) - 1;
    // the per-column constant tables of the last tile's level and channel range: rebuilt only
    // when a tile needs others (tiles of one job and N range keep them), so most tiles start
    // without table loads or barriers
    long long cur_key = -1;  // (level, first channel, width) of the tables
    int flags = 0;           // bit 0: 32-bit requant form, 1: |bias| <= 2^30, 2: 32-bit skip form
    for (int t = first_tile; t < tile_end; t += tile_stride, ++lt) {
      const TileInfo ti = tile_info(p, t);
      const ConvJobDev& jb = p.jobs[ti.job];
      // this tile's output channels that exist (a last N tile may reach past cout; packed
      // groups past it must not be written)
      const int TBN = ti.cn < p.cout - ti.col0 ? ti.cn : p.cout - ti.col0;
      const LayerDev& ly = p.layers[ti.layer];
      const long long key =
          ((long long)ti.layer << 48) | ((long long)jb.level << 32) | ((long long)ti.col0 << 10) | TBN;
      if (key != cur_key) {
        // (the same decision in every epilogue thread: all of them see the same tiles)
        named_bar(1, kEpiThreads);  // every epilogue warp is done with the previous tables
        // Per-column constants of this tile's level. The 32-bit fast path applies when the
        // total requant shift R = 31 + shift is >= 33 (then y = (mulhi(u, M0) + 2^(R-33)) >>
        // (R-32) equals rhu(u * M0, R): the low product word cannot carry into the result)
        // and |bias| <= 2^30 (acc + bias cannot leave int32 when |acc| < 2^24).
        int fq = 1, sbias = 1;
        for (int col = et; col < 256; col += kEpiThreads) {
          const int ch = ti.col0 + col;
          EpiChan ec{};
          int4 ef = make_int4((int32_t)(0u - kMagicBits), 0, 0, 1);
          if (col < TBN && ch < p.cout) {
            const int64_t idx = (int64_t)jb.level * p.cout + ch;
            ec.bias = ly.bias ? ly.bias[idx] : 0;
            const bool sb = ec.bias >= -(1 << 30) && ec.bias <= (1 << 30);
            sbias &= sb;
            ef.x = (int32_t)((uint32_t)ec.bias - kMagicBits);
            if (out_bits != 32) {
              ec.m0 = ly.m0[idx];
              const int r = 31 + ly.shift[idx];
              ec.r = (int8_t)r;
              if (r >= 33 && sb) { ef.y = ec.m0; ef.z = 1 << (r - 33); ef.w = r - 32; }
              else fq = 0;
            }
            if (kSkip) { ec.c = p.skip_c[idx]; ec.d = p.skip_d[idx]; }
          }
          epi[col] = ec;
          reinterpret_cast<int4*>(epi + 256)[col] = ef;
        }
        fq = named_bar_and(1, kEpiThreads, fq);
        sbias = named_bar_and(1, kEpiThreads, sbias);
        // 32-bit skip path (fast_skip_group): default direction, code skips, d >= 8 everywhere
        // (int32 skips: 64-bit product, any d >= 1)
        int fsk = 0;
        if (kSkip && p.scale_main == 0 && out_bits != 32 && fq && sbias) {
          const int dmin = p.skip_bits <= 8 ? 8 : 1;
          int okd = 1;
          for (int col = et; col < TBN; col += kEpiThreads)
            if (ti.col0 + col < p.cout && epi[col].d < dmin) okd = 0;
          fsk = named_bar_and(1, kEpiThreads, okd);
        }
        flags = fq | (sbias << 1) | (fsk << 2);
        cur_key = key;
      }
      const int fast_req = flags & 1, small_bias = (flags >> 1) & 1, fast_skip = (flags >> 2) & 1;
      // 0: general int64 epilogue; 1: fast requant to codes; 2: int32 output, no skip
      // (kSkip: the skip instantiation runs exactly the calls with a skip, so its mode is 0 at
      // compile time and it carries no code or registers of the other modes)
      const int mode = (kSplit || kSkip) ? 0 : (out_bits == 32 ? 2 : (fast_req ? 1 : 0));
      const bool magic = p.acc_small && (mode == 2 ? small_bias : fast_req);
      const uint32_t buf = lt & 1;
      if (!mbar_wait(b_tfull + 8 * buf, (lt >> 1) & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();

      // This warp's (sub-tile, 32-column group) units. The TMEM load of the next unit is in
      // flight while the current one is converted and stored; no register written by a
      // tcgen05.ld is read before the tcgen05.wait::ld that covers it.
      const int ngrp = (TBN + 31) / 32;
      const int nunits = kSub * ngrp;
      const uint32_t tbuf = lane_base + buf * (uint32_t)(kSub * BN);
      uint32_t va[32], vn[32];
      __syncwarp();
      if (gi < nunits) {
        tmem_ld32(tbuf + (gi / ngrp) * (uint32_t)BN + (gi % ngrp) * 32, ti.cn - (gi % ngrp) * 32 >= 32, va);
        tmem_wait_ld();
        reg_fence32(va);
      }
      for (int u0 = gi; u0 < nunits; u0 += kGroups) {
        const int un = u0 + kGroups;
        // the next unit's TMEM load overlaps this unit's work in the light modes; the general /
        // skip mode (0) holds more registers and loads it afterwards
        if (un < nunits && mode != 0)
          tmem_ld32(tbuf + (un / ngrp) * (uint32_t)BN + (un % ngrp) * 32, ti.cn - (un % ngrp) * 32 >= 32, vn);
        const int sub = u0 / ngrp, g0 = (u0 % ngrp) * 32;
        const int ncols = (TBN - g0) < 32 ? (TBN - g0) : 32;
        // 32 TMEM columns were loaded when the tile's MMA width covers them (else 16)
        const bool full = ti.cn - g0 >= 32;
        if (!full) {
#pragma unroll
          for (int i = 16; i < 32; ++i) va[i] = 0u;  // only the first 16 columns were loaded
        }
        if constexpr (kSplit) {
          // split weights: va holds D1 (w_lo rows); D2 (w_hi rows) sits TBN columns on;
          // the exact sum is D1 + 16 D2, each an integer x 2^-18 below 2^24
          uint32_t vb[32];
          tmem_ld32(tbuf + (uint32_t)ti.cn + g0, full, vb);
          tmem_wait_ld();
          reg_fence32(vb);
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int32_t d1 = __float2int_rn(__uint_as_float(va[i]) * kAccSc);
            const int32_t d2 = (full || i < 16) ? __float2int_rn(__uint_as_float(vb[i]) * kAccSc) : 0;
            va[i] = (uint32_t)(d1 + 16 * d2);
          }
        }
        const uint32_t* v = va;
        int m;  // output pixel index within the job
        bool row_ok;
        int oimg = 0, oh = 0, ow = 0;  // the pixel (flat path)
        if constexpr (kFlat) {
          const FlatTile ft = flat_tile(jb, ti.mt, kTileRows);
          const int vr = ft.v0 + (int)rank * 128 + quarter * 32 + lane;  // virtual row at the padded width
          const int ho = vr / jb.wp, wo = vr - (vr / jb.wp) * jb.wp;
          row_ok = vr < jb.vimg && wo < jb.wo;  // else a junk column or past the image
          m = (ft.img * jb.ho + ho) * jb.wo + wo;
          oimg = ft.img; oh = ho; ow = wo;
        } else {
          m = ti.mt * BM + sub * 128 + quarter * 32 + lane;
          row_ok = m < jb.m_total;
        }
        if constexpr (kOStage) {
          // (launched for int32 outputs without a skip only: mode 2)
          // int32 outputs through this warp's staging block: each lane holds its row's 32
          // values; stored back four rows at a time, so every warp store covers four whole
          // 128-byte row segments instead of 32 scattered 16-byte pieces (cout % 4 == 0)
          uint32_t* stg = reinterpret_cast<uint32_t*>(smem + p.off_ostage) + warp * (32 * kStageRow);
          const int ch0 = ti.col0 + g0;
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            int32_t o[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float f = __uint_as_float(v[4 * q + k]);
              o[k] = magic ? __float_as_int(__fmaf_rn(f, kAccSc, kMagic)) + epf[g0 + 4 * q + k].x
                           : add_sat(__float2int_rn(f * kAccSc), epi[g0 + 4 * q + k].bias);
            }
            *reinterpret_cast<int4*>(stg + lane * kStageRow + 4 * q) = make_int4(o[0], o[1], o[2], o[3]);
          }
          __syncwarp();
          const uint32_t rows_ok = __ballot_sync(0xffffffffu, row_ok);
          const int nq = (ncols < p.cout - ch0 ? ncols : p.cout - ch0) >> 2;  // whole 16-byte pieces
#pragma unroll
          for (int r4 = 0; r4 < 8; ++r4) {
            const int r = 4 * r4 + (lane >> 3), c4 = lane & 7;
            const int mr = __shfl_sync(0xffffffffu, m, r);
            if (((rows_ok >> r) & 1u) && c4 < nq) {
              const int4 val = *reinterpret_cast<const int4*>(stg + r * kStageRow + 4 * c4);
              *reinterpret_cast<int4*>(ly.y[ti.job] + (int64_t)mr * p.y_row_bytes + (int64_t)(ch0 + 4 * c4) * 4) = val;
            }
          }
          __syncwarp();
        } else {
  if (row_ok) {
            uint8_t* yrow = ly.y[ti.job] + (int64_t)m * p.y_row_bytes;
            const int ch0 = ti.col0 + g0;
            if (mode == 1 && magic) {
              // codes as byte-words: the chained image takes them as they are, the packed
              // output a couple of shifts per 8 codes
              uint32_t bw[8], gw[8];
              magic_requant_bytes(v, epf + g0, qmax, kAccSc, bw);
              switch (out_bits) {
                case 2: pack_bytewords<2>(bw, gw); break;
                case 3: pack_bytewords<3>(bw, gw); break;
                case 4: pack_bytewords<4>(bw, gw); break;
                default: pack_bytewords<8>(bw, gw); break;
              }
              store_group(yrow + (ch0 >> 5) * group_bytes(out_bits), gw, out_bits);
              if (kFlat && ly.ws_out) chain_store_bw(p, ly.ws_out, ly.ws_nib, jb, oimg, oh, ow, ch0, bw);
            } else if (mode == 1) {
              uint32_t gw[8];
              {
                switch (out_bits) {
                  case 2: fast_requant_group<2>(v, epi, g0, qmax, kAccSc, gw); break;
                  case 3: fast_requant_group<3>(v, epi, g0, qmax, kAccSc, gw); break;
                  case 4: fast_requant_group<4>(v, epi, g0, qmax, kAccSc, gw); break;
                  default: fast_requant_group<8>(v, epi, g0, qmax, kAccSc, gw); break;
                }
              }
              store_group(yrow + (ch0 >> 5) * group_bytes(out_bits), gw, out_bits);
              if (kFlat && ly.ws_out) chain_store(p, ly.ws_out, ly.ws_nib, jb, oimg, oh, ow, ch0, gw, out_bits);
            } else if (mode == 2) {
              int32_t* yr = reinterpret_cast<int32_t*>(yrow) + ch0;
              const bool whole = ncols == 32 && ch0 + 32 <= p.cout;
    #pragma unroll
              for (int q = 0; q < 8; ++q) {
                int32_t o[4];
    #pragma unroll
                for (int k = 0; k < 4; ++k) {
                  const float f = __uint_as_float(v[4 * q + k]);
                  o[k] = magic ? __float_as_int(__fmaf_rn(f, kAccSc, kMagic)) + epf[g0 + 4 * q + k].x
                               : add_sat(__float2int_rn(f * kAccSc), epi[g0 + 4 * q + k].bias);
                }
                if (whole) {
                  reinterpret_cast<int4*>(yr)[q] = make_int4(o[0], o[1], o[2], o[3]);
                } else {
    #pragma unroll
                  for (int k = 0; k < 4; ++k)
                    if (4 * q + k < ncols && ch0 + 4 * q + k < p.cout) yr[4 * q + k] = o[k];
                }
              }
            } else {
              const uint8_t* srow = nullptr;
              if (kSkip) {
                int img, ho, wo;
                if constexpr (kFlat) {
                  img = oimg; ho = oh; wo = ow;
                } else {
                  const int hw = jb.ho * jb.wo;
                  img = m / hw;
                  const int rem = m - img * hw;
                  ho = rem / jb.wo; wo = rem - ho * jb.wo;
                }
                const int sh = p.upsample == 2 ? ho >> 1 : ho, sw = p.upsample == 2 ? wo >> 1 : wo;
                srow = jb.skip + (((int64_t)img * jb.skip_h + sh) * jb.skip_w + sw) * p.skip_row_bytes;
              }
              int32_t oo[32];
              if (kSkip && fast_skip && p.skip_bits <= 8) {
                load_skip_group(p, srow, ch0, ncols, oo);   // skip codes, replaced by the results
                fast_skip_group(v, epi + g0, oo, qmax, kAccSc, oo);
              } else if (kSkip && fast_skip) {
                load_skip_group(p, srow, ch0, ncols, oo);   // int32 skip, replaced by the results
                fast_skip32_group(v, epi + g0, oo, qmax, kAccSc, oo);
              } else {
                general_group<kSkip, kSplit>(p, v, epi + g0, srow, ch0, ncols, kAccSc, oo);
              }
              if (out_bits == 32) {
                int32_t* yr = reinterpret_cast<int32_t*>(yrow) + ch0;
  #pragma unroll
                for (int i = 0; i < 32; ++i)
                  if (i < ncols && ch0 + i < p.cout) yr[i] = oo[i];
              } else {
                // clipped codes (< 2^out_bits) as byte-words, then the packed group
                uint32_t bw[8], gw[8];
  #pragma unroll
                for (int j = 0; j < 8; ++j)
                  bw[j] = (uint32_t)oo[4 * j] | ((uint32_t)oo[4 * j + 1] << 8) | ((uint32_t)oo[4 * j + 2] << 16) |
                          ((uint32_t)oo[4 * j + 3] << 24);
                switch (out_bits) {
                  case 2: pack_bytewords<2>(bw, gw); break;
                  case 3: pack_bytewords<3>(bw, gw); break;
                  case 4: pack_bytewords<4>(bw, gw); break;
                  default: pack_bytewords<8>(bw, gw); break;
                }
                store_group(yrow + (ch0 >> 5) * group_bytes(out_bits), gw, out_bits);
                if (kFlat && ly.ws_out) chain_store_bw(p, ly.ws_out, ly.ws_nib, jb, oimg, oh, ow, ch0, bw);
              }
            }
          }
        }
        if (un < nunits) {
          if (mode == 0)
            tmem_ld32(tbuf + (un / ngrp) * (uint32_t)BN + (un % ngrp) * 32, ti.cn - (un % ngrp) * 32 >= 32, vn);
          tmem_wait_ld();
          reg_fence32(vn);
#pragma unroll
          for (int i = 0; i < 32; ++i) va[i] = vn[i];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (kPair && !leader) mbar_arrive_cluster(mapa_shared(b_tempty + 8 * buf, 0));
        else mbar_arrive(b_tempty + 8 * buf);
      }
      if (kFlat && p.dep && ti.layer < p.nlayers - 1) {
        // this warp's stores of tile t are done: order them for the next layer's TMA (async
        // proxy) loads, gather the warp (__syncwarp orders its lanes' stores before lane 0's
        // next operations), and count the warp in with one release (cumulative over them)
        fence_proxy_async_global();
        __syncwarp();
        // (a tower launch has no half-width tiles: t is layer * layer_tiles + the tile)
        if (lane == 0) red_release_gpu_add(p.dep + t, 1u);
      }
    }
    if (!ok) fail(abort_flag, p.status);
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA of a pair leaves while the leader's MMAs may still read the peer's shared
  // memory or write its TMEM (the leader's MMA thread drained them before the barrier)
  if constexpr (kPair) cluster_sync();
  if (warp == kWarpMma) {
    tc_fence_after();
    if constexpr (kPair)
      asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;"
                   ::"r"(tmem_base), "r"(p.tmem_cols) : "memory");
    else
      asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                   ::"r"(tmem_base), "r"(p.tmem_cols) : "memory");
  }
}

// ---------------------------------------------------------------- activation expansion

// Writes every job's input as a zero-padded byte image: workspace row
// row_off + (img * hp + hp_i) * wp + wp_i holds the cin E4M3 bytes (raw byte = code) of
// input pixel (img, hp_i - pad, wp_i - pad), or zeros in the padding border.
struct ExpandArgs {
  ConvJobDev jobs[kMaxJobs];
  int32_t njobs, cin, pad;
  int64_t x_row_bytes;
  int64_t total_rows;     // rows of one plane
  uint8_t* ws;
  // per-tile counters of a chained tower, cleared here (before the first layer, which waits
  // for this grid, can raise them)
  uint32_t* zero;
  int32_t zero_words;
};

// E4M3 byte of the value 16 n * 2^-9 = n * 2^-5, n in [0, 15] (the raw byte n is n * 2^-9):
// n = 2^e (1 + m/8) with 8-bit exponent field e + 2, packed as two 64-bit tables of 8 bytes.
__device__ __forceinline__ uint32_t e4m3_times16(uint32_t n) {
  constexpr uint64_t lo = 0x26242220'1C181000ull;  // n = 7 .. 0
  constexpr uint64_t hi = 0x2F2E2D2C'2B2A2928ull;  // n = 15 .. 8
  return (uint32_t)(((n < 8 ? lo : hi) >> (8 * (n & 7))) & 0xFFu);
}

// Position of one workspace row: its job, image, padded row / column and input pointer.
struct ExpandPos {
  int row, job, img, hr, wc;  // workspace row; job; image; padded row and column
  int next_off;               // first row of the next job (INT_MAX for the last)
};

__device__ __forceinline__ void expand_locate(const ExpandArgs& a, int row, ExpandPos& ps) {
  int j = 0;
#pragma unroll 1
  while (j + 1 < a.njobs && row >= a.jobs[j + 1].row_off) ++j;
  const ConvJobDev& jb = a.jobs[j];
  const int local = row - jb.row_off;
  const int plane = jb.hp * jb.wp;
  ps.row = row;
  ps.job = j;
  ps.img = local / plane;
  const int rem = local - ps.img * plane;
  ps.hr = rem / jb.wp;
  ps.wc = rem - ps.hr * jb.wp;
  ps.next_off = j + 1 < a.njobs ? a.jobs[j + 1].row_off : 0x7fffffff;
}

// Moves the position forward by d rows (d small: at most 4 here).
__device__ __forceinline__ void expand_advance(const ExpandArgs& a, int d, ExpandPos& ps) {
  ps.row += d;
  if (ps.row >= ps.next_off) { expand_locate(a, ps.row, ps); return; }
  const ConvJobDev& jb = a.jobs[ps.job];
  ps.wc += d;
#pragma unroll 1
  while (ps.wc >= jb.wp) {
    ps.wc -= jb.wp;
    if (++ps.hr == jb.hp) { ps.hr = 0; ++ps.img; }
  }
}

template <int kXBits>
__global__ void __launch_bounds__(256) expand_kernel(const __grid_constant__ ExpandArgs a) {
  // The (row, 16-byte chunk) pairs of the workspace, row-major, are split into runs of
  // 32 * kPerLane; a warp takes one run, lane l the pairs l, l + 32, ... of it, so every
  // warp-wide step reads consecutive packed words and writes 512 consecutive bytes. The
  // position is divided out once per lane and then advanced incrementally; the loads of
  // all steps are issued before the stores. All index arithmetic is 32-bit (the host
  // checks rows * cin / 16 < 2^31).
  constexpr int kPerLane = 4;  // (measured: 4 beats 8 and 2 on the head step, 120.6 / 121.7 / 121.5 us)
  // the previous kernel in the stream may still be reading the workspace or writing x
  grid_dep_wait();
  if (threadIdx.x == 0) grid_dep_launch();
  if (blockIdx.x == 0)
    for (int i = threadIdx.x; i < a.zero_words; i += blockDim.x) a.zero[i] = 0u;
  const int chunks = a.cin >> 4;
  const int total = (int)a.total_rows * chunks;
  const int lane = threadIdx.x & 31;
  const int e0 = (blockIdx.x * 8 + (threadIdx.x >> 5)) * (32 * kPerLane) + lane;
  if (e0 >= total) return;
  const int drow = 32 / chunks, dq = 32 - drow * chunks;
  ExpandPos ps;
  int q = e0 % chunks;
  expand_locate(a, e0 / chunks, ps);
  uint32_t w[kPerLane][kXBits == 2 ? 1 : (kXBits == 8 ? 4 : 2)];
  uint8_t* dst[kPerLane];
  bool inside[kPerLane];
  int hsel[kPerLane];
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    const int e = e0 + 32 * i;
    const bool live = e < total;
    const ConvJobDev& jb = a.jobs[ps.job];
    const int hi = ps.hr - a.pad, wi = ps.wc - a.pad;
    inside[i] = live && hi >= 0 && hi < jb.h && wi >= 0 && wi < jb.w;
    dst[i] = live ? a.ws + (size_t)ps.row * a.cin + q * 16 : nullptr;
    hsel[i] = q & 1;
    if (inside[i]) {
      const uint32_t* grp = reinterpret_cast<const uint32_t*>(
          jb.x + ((size_t)(ps.img * jb.h + hi) * jb.w + wi) * a.x_row_bytes + (q >> 1) * 4 * kXBits);
      if constexpr (kXBits == 8) {
        // 16 one-byte codes: channels 16 q .. 16 q + 15
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(jb.x + ((size_t)(ps.img * jb.h + hi) * jb.w + wi) *
                                                             a.x_row_bytes) + q);
        w[i][0] = v.x; w[i][1] = v.y; w[i][2] = v.z; w[i][3] = v.w;
      } else if constexpr (kXBits == 2) {
        w[i][0] = __ldg(grp + (q & 1));
      } else if constexpr (kXBits == 4) {
        const uint2 v = __ldg(reinterpret_cast<const uint2*>(grp) + (q & 1));
        w[i][0] = v.x; w[i][1] = v.y;
      } else {
        w[i][0] = __ldg(grp + (q & 1)); w[i][1] = __ldg(grp + 2);
      }
    }
    if (i + 1 < kPerLane) {
      q += dq;
      int step = drow;
      if (q >= chunks) { q -= chunks; ++step; }
      if (step) expand_advance(a, step, ps);
    }
  }
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    if (!dst[i]) continue;
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if constexpr (kXBits == 8) {
      // plane 0: x_lo = x & 15 (raw byte); plane 1, total_rows rows on: 16 x_hi as E4M3
      uint32_t o1[4] = {0u, 0u, 0u, 0u};
      if (inside[i]) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          o[j] = w[i][j] & 0x0F0F0F0Fu;
          const uint32_t hn = (w[i][j] >> 4) & 0x0F0F0F0Fu;
          o1[j] = e4m3_times16(hn & 0xFFu) | (e4m3_times16((hn >> 8) & 0xFFu) << 8) |
                  (e4m3_times16((hn >> 16) & 0xFFu) << 16) | (e4m3_times16(hn >> 24) << 24);
        }
      }
      *reinterpret_cast<uint4*>(dst[i]) = make_uint4(o[0], o[1], o[2], o[3]);
      *reinterpret_cast<uint4*>(dst[i] + (size_t)a.total_rows * a.cin) = make_uint4(o1[0], o1[1], o1[2], o1[3]);
      continue;
    }
    if (inside[i]) {
      const int h = hsel[i];
      if constexpr (kXBits == 2) {
#pragma unroll
        for (int j = 0; j < 4; ++j) o[j] = (w[i][0] >> (2 * j)) & 0x03030303u;
      } else if constexpr (kXBits == 4) {
        o[0] = w[i][0] & 0x0F0F0F0Fu; o[1] = (w[i][0] >> 4) & 0x0F0F0F0Fu;
        o[2] = w[i][1] & 0x0F0F0F0Fu; o[3] = (w[i][1] >> 4) & 0x0F0F0F0Fu;
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          o[j] = ((w[i][0] >> (2 * j)) & 0x03030303u) | (((w[i][1] >> (4 * h + j)) & 0x01010101u) << 2);
      }
    }
    *reinterpret_cast<uint4*>(dst[i]) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// The zero-padded nibble image of 2-bit codes for the FP4 pipe: the first cin / 2 bytes of
// workspace row r (rows cin bytes apart, as in the byte image) hold two codes per byte,
// channel 2k in the low nibble of byte k, of input pixel (img, hp - pad, wp - pad), or zeros
// in the border (code 0 is the E2M1 value 0). One thread
// per 16 output bytes, i.e. one 32-channel packed group of 8 input bytes; consecutive threads
// take consecutive groups of a row.
__global__ void __launch_bounds__(256) expand_nib_kernel(const __grid_constant__ ExpandArgs a) {
  grid_dep_wait();
  if (threadIdx.x == 0) grid_dep_launch();
  const int groups = a.cin >> 5;
  const int64_t total = a.total_rows * groups;
  for (int64_t e = (int64_t)blockIdx.x * 256 + threadIdx.x; e < total; e += (int64_t)gridDim.x * 256) {
    const int row = (int)(e / groups), g = (int)(e - (int64_t)row * groups);
    ExpandPos ps;
    expand_locate(a, row, ps);
    const ConvJobDev& jb = a.jobs[ps.job];
    const int hi = ps.hr - a.pad, wi = ps.wc - a.pad;
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if (hi >= 0 && hi < jb.h && wi >= 0 && wi < jb.w) {
      const uint2 v = __ldg(reinterpret_cast<const uint2*>(jb.x + ((size_t)(ps.img * jb.h + hi) * jb.w + wi) *
                                                                   a.x_row_bytes) + g);
#pragma unroll
      for (int m = 0; m < 4; ++m) {
        // output word m: channels 8m .. 8m + 7, the byte-words 2(m % 2) and 2(m % 2) + 1 of
        // packed word m / 2 (byte-word j of a 2-bit word: channels 4j .. 4j + 3, one per byte)
        const uint32_t wd = (m >> 1) ? v.y : v.x;
        const int j0 = 2 * (m & 1);
        const uint32_t b0 = (wd >> (2 * j0)) & 0x03030303u, b1 = (wd >> (2 * j0 + 2)) & 0x03030303u;
        o[m] = __byte_perm(b0 | (b0 >> 4), b1 | (b1 >> 4), 0x6420);
      }
    }
    *reinterpret_cast<uint4*>(a.ws + (size_t)row * a.cin + (size_t)g * 16) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// ---------------------------------------------------------------- host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn(std::string* err) {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  static cudaError_t st = cudaSuccess;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    st = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q);
    if (st == cudaSuccess && q == cudaDriverEntryPointSuccess) fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  if (!fn && err) *err = "cuTensorMapEncodeTiled entry point unavailable";
  return fn;
}

template <int kXBits, bool kChunkInTap, bool kFlat, bool kPair = false, bool kSkip = true, bool kSplit = false,
          int kBK = BK, bool kFp4 = false, bool kOStage = false>
static int launch_bits(const Params& prm, const Maps& maps, int grid, size_t smem, cudaStream_t stream,
                       std::string* err) {
  auto kern = conv_tc_kernel<kXBits, kChunkInTap, kFlat, kPair, kSkip, kSplit, kBK, kFp4, kOStage>;
  // The opt-in limit is raised to the device maximum, never lowered to this call's size:
  // a CUDA graph node captured earlier with a larger plan must stay launchable (a graph
  // node, or a tool relaunching it, is checked against the function's current limit).
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if ((size_t)optin < smem) { *err = "conv_tc: shared memory plan exceeds the device limit"; return 2; }
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
  if (e != cudaSuccess) { *err = std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e); return 3; }
  // programmatic dependent launch: the prologue (barriers, TMEM allocation, tensor-map
  // prefetch) overlaps the previous kernel; the kernel waits for it before touching global
  // memory. CTA pairs run as clusters of two.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3((unsigned)threads_for(kFlat));
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = kPair ? 2 : 1;
  e = cudaLaunchKernelEx(&cfg, kern, maps, prm);
  if (e != cudaSuccess) { *err = std::string("conv_tc launch: ") + cudaGetErrorString(e); return 3; }
  e = cudaGetLastError();
  if (e != cudaSuccess) { *err = std::string("conv_tc launch: ") + cudaGetErrorString(e); return 3; }
  return 0;
}

}  // namespace tc

bool conv_tc_uses_pair(const ConvArgs& a) {
  // every N tile width of the workspace path (BN is a multiple of 16, so each CTA's half of
  // the weight tile is whole 8-row swizzle atoms and M = 256 MMAs take N = BN), except narrow
  // tiles on the FP4 pipe: the 256->84 output conv of the head measured 35.7 us on single
  // CTAs against 39.4 us on pairs (same box, expansion included)
  if (a.fp4 && a.bn <= 128) return false;
  return a.ws != nullptr && a.bn >= 16 && a.bn % 16 == 0 && tc::kSub == 1 && !a.no_pair;
}

// Last-wave balancing: with `workers` persistent CTAs (or CTA pairs), the full tiles past the
// last complete wave run as two half-width (N/2) tiles each, when those halves still fit in
// one wave; half as long per tile, they end the kernel sooner. A half tile must start on a
// 32-channel packing group (bn / 2 a multiple of 32). Returns the first split tile.
static int split_start(int tiles, int workers, int bn, bool split_w) {
  const int rem = tiles % workers;
  return (bn % 64 == 0 && !split_w && rem > 0 && 2 * rem <= workers) ? tiles - rem : tiles;
}

int64_t conv_tc_pair_tiles(const ConvArgs& a) {
  int64_t tiles = 0;
  for (int j = 0; j < a.njobs; ++j) {
    const ConvJobDev& jb = a.jobs[j];
    const int64_t wp = jb.w + 2 * a.pad;
    tiles += (int64_t)jb.n * ((jb.ho * wp + 255) / 256);
  }
  return tiles;
}

int launch_conv_tc(const ConvArgs& a, cudaStream_t stream, std::string* err) {
  using namespace tc;
  Params prm{};
  // split (8-bit) weights: tiles of 256 weight rows = 128 output channels
  const int BN = a.split_w ? 256 : a.bn;
  const int w_rows = a.split_w ? a.split_rows : a.cout_pad;  // rows of the weight block
  prm.njobs = a.njobs;
  prm.n_tiles = w_rows / BN;
  // flat path: the activations are expanded into the workspace first (stride 1,
  // cin % 128 == 0; the API checks both before passing a workspace)
  const bool flat = a.ws != nullptr;
  // CTA pairs (cta_group::2, M = 256 per tile) on the workspace path: each SM streams half
  // of the weight tile per K chunk, and one MMA instruction covers both SMs' rows
  const bool pair = conv_tc_uses_pair(a);
  const int tile_rows = pair ? 256 : 128;
  int tiles = 0;
  int64_t rows = 0;
  for (int j = 0; j < a.njobs; ++j) {
    prm.jobs[j] = a.jobs[j];
    prm.jobs[j].tile_begin = tiles;
    if (flat) {
      ConvJobDev& jb = prm.jobs[j];
      jb.hp = jb.h + 2 * a.pad;
      jb.wp = jb.w + 2 * a.pad;
      jb.vimg = jb.ho * jb.wp;
      jb.tpi = (jb.vimg + tile_rows - 1) / tile_rows;
      jb.row_off = (int32_t)rows;
      rows += (int64_t)jb.n * jb.hp * jb.wp;
      tiles += jb.n * jb.tpi * prm.n_tiles;
    } else {
      tiles += ((a.jobs[j].m_total + BM - 1) / BM) * prm.n_tiles;
    }
  }
  // K chunk width: 128 bytes of one tap, or on the workspace path with cin % 128 != 0 the 64
  // channels of one tap (cin % 64 == 0; 64-byte swizzled operand rows, two MMAs per chunk)
  const bool fp4 = a.fp4 != 0;
  // bytes per row of the image: one code per byte, or two (nibbles) on the FP4 pipe
  const int img_row = fp4 ? a.cin / 2 : a.cin;
  const int bk = (flat && img_row % BK != 0) ? 64 : BK;
  if (flat && (kSub != 1 || a.stride != 1 || img_row % bk != 0 || rows > a.ws_rows || (a.split_w && bk != BK))) {
    *err = "conv_tc: workspace path needs stride 1, cin % 64 == 0 (128 for split weights) and a large enough workspace";
    return 1;
  }
  if (fp4 && !(flat && bk == BK && a.x_bits == 2 && !a.split_w && a.a_planes <= 1 && a.zero_words == 0 && !a.ws_out &&
               a.nlayers <= 1 && a.w_fp4)) {
    *err = "conv_tc: the FP4 pipe takes 2-bit codes from a nibble image (cin % 256 == 0), one layer, no chained output";
    return 1;
  }
  if (tiles == 0) return 0;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms < 2) sms = 2;
  // Last-wave balancing: with `workers` persistent CTAs (or CTA pairs), the full tiles past
  // the last complete wave run as two half-width (N/2) tiles each, when those halves still
  // fit in one wave; half as long per tile, they end the kernel sooner.
  const int nlayers = a.nlayers > 1 ? a.nlayers : 1;
  if (nlayers > 1 && !(flat && pair && prm.n_tiles == 1 && !a.split_w && a.a_planes <= 1 && a.ws2 && a.dep &&
                       nlayers <= kMaxLayers)) {
    *err = "conv_tc: chained layers in one launch need the workspace path on CTA pairs with one N tile";
    return 1;
  }
  // (a launch of several layers has no half-width tiles: every layer keeps the same tiles)
  prm.dp_tiles = nlayers > 1 ? tiles : split_start(tiles, pair ? sms / 2 : sms, BN, a.split_w != 0);
  prm.total_tiles = nlayers * (prm.dp_tiles + 2 * (tiles - prm.dp_tiles));
  // contiguous tile ranges for single-CTA launches of one layer on the workspace path with no
  // half tiles (the FP4 output conv): neighbouring tiles share a level's tables and halo rows
  prm.contig = (!pair && flat && nlayers <= 1 && prm.dp_tiles == tiles) ? 1 : 0;
  prm.nlayers = nlayers;
  prm.layer_tiles = prm.total_tiles / nlayers;
  prm.num_kchunks = flat ? (fp4 ? a.k_total / 2 : a.k_total) / bk : a.k_pad / BK;
  prm.cin = a.cin; prm.cout = a.cout; prm.kh = a.kh; prm.kw = a.kw;
  prm.stride = a.stride; prm.pad = a.pad; prm.k_total = a.k_total;
  prm.out_bits = a.out_bits; prm.skip_bits = a.skip_bits;
  prm.x_row_bytes = a.x_row_bytes; prm.y_row_bytes = a.y_row_bytes; prm.skip_row_bytes = a.skip_row_bytes;
  if (nlayers > 1) {
    for (int l = 0; l < nlayers; ++l) {
      LayerDev& ly = prm.layers[l];
      ly.m0 = a.layer[l].m0; ly.shift = a.layer[l].shift; ly.bias = a.layer[l].bias;
      for (int j = 0; j < a.njobs; ++j) ly.y[j] = a.layer[l].y[j];
      ly.ws_out = a.layer[l].ws_out;
      ly.ws_nib = a.layer[l].ws_nib;
    }
  } else {
    LayerDev& ly = prm.layers[0];
    ly.m0 = a.m0; ly.shift = a.shift; ly.bias = a.bias;
    for (int j = 0; j < a.njobs; ++j) ly.y[j] = a.jobs[j].y;
    ly.ws_out = a.ws_out;
    ly.ws_nib = a.ws_out_nib;
  }
  prm.skip_c = a.skip_c; prm.skip_d = a.skip_d;
  prm.upsample = a.upsample; prm.scale_main = a.scale_main; prm.has_skip = a.has_skip;
  prm.bn = BN;
  prm.acc_small = a.acc_bound < (1LL << 22) ? 1 : 0;
  prm.cin_chunks = img_row / bk;
  prm.out_pad = a.out_pad;
  prm.a_planes = flat ? (a.a_planes > 1 ? a.a_planes : 1) : 1;
  prm.plane_rows = (int32_t)rows;
  prm.split_w = a.split_w;
  bool chained = a.ws_out != nullptr;
  for (int l = 0; l < nlayers && nlayers > 1; ++l) chained |= a.layer[l].ws_out != nullptr;
  if (chained) {
    int64_t orows = 0;
    for (int j = 0; j < a.njobs; ++j) {
      ConvJobDev& jb = prm.jobs[j];
      jb.ohp = jb.ho + 2 * a.out_pad;
      jb.owp = jb.wo + 2 * a.out_pad;
      jb.orow_off = (int32_t)orows;
      orows += (int64_t)jb.n * jb.ohp * jb.owp;
    }
  }
  prm.status = a.status;
  prm.dep = nlayers > 1 ? a.dep : nullptr;
  prm.dep_target = (uint32_t)(2 * kEpiWarps);  // epilogue warps of both CTAs of a pair
  // shared memory plan: stages of (BM x bk A bytes + this CTA's B rows x bk bytes)
  const int b_rows = pair ? BN / 2 : BN;
  const size_t stage_a = (size_t)kSub * 128 * bk;
  const size_t stage_bytes = stage_a + (size_t)b_rows * bk;
  const size_t epi_bytes = 256 * sizeof(EpiChan) + 256 * sizeof(int4);
  const size_t bar_bytes = 8 * (2 * kMaxStages + 5) + 16;
  const size_t qtab_bytes = kQTab * sizeof(uint32_t);
  const size_t budget = 232448 - 1024;  // max dynamic smem per block minus alignment slack
  // int32 outputs with cout % 4 == 0: per-warp staging blocks when at least 6 stages remain
  const size_t ostage_bytes = (size_t)kEpiWarps * 32 * kStageRow * sizeof(uint32_t);
  const bool ostage = flat && bk == BK && a.out_bits == 32 && a.cout % 4 == 0 && !a.has_skip && !a.split_w &&
                      (budget - epi_bytes - bar_bytes - qtab_bytes - ostage_bytes) / stage_bytes >= 6;
  int stages = (int)((budget - epi_bytes - bar_bytes - qtab_bytes - (ostage ? ostage_bytes : 0)) / stage_bytes);
  if (stages > kMaxStages) stages = kMaxStages;
  if (stages < 2) { *err = "conv_tc: shared memory plan does not fit"; return 2; }
  // The TMA issuers take K chunks round-robin and each waits on its stage's "empty"
  // barrier by phase parity. That parity is unambiguous only while no issuer can run more
  // than one phase ahead of the last completed one, which holds when the issuers are at
  // most as many as the stages.
  if (stages < tma_warps(flat)) { *err = "conv_tc: fewer pipeline stages than TMA issuers"; return 2; }
  prm.stages = stages;
  prm.off_b = (uint32_t)(stages * stage_a);
  prm.off_epi = prm.off_b + (uint32_t)(stages * b_rows * bk);
  prm.off_bar = prm.off_epi + (uint32_t)epi_bytes;
  prm.off_qtab = prm.off_bar + (uint32_t)bar_bytes;
  prm.off_ostage = ostage ? (uint32_t)((prm.off_qtab + qtab_bytes + 15) / 16 * 16) : 0u;
  const size_t smem = 1024 + (ostage ? prm.off_ostage + ostage_bytes : prm.off_qtab + qtab_bytes);
  // two buffers x kSub sub-tiles x BN fp32 columns (and, on the FP4 pipe, 32 columns of scales)
  const int acc_cols = 2 * kSub * BN;
  if (fp4 && acc_cols + 32 > 512) { *err = "conv_tc: FP4 tiles wider than 240 channels do not fit in TMEM"; return 2; }
  int cols = 32;
  while (cols < acc_cols + (fp4 ? 32 : 0)) cols *= 2;
  prm.tmem_cols = cols;
  prm.sf_col = acc_cols;

  EncodeTiledFn enc = get_encode_fn(err);
  if (!enc) return 3;
  Maps maps{};
  // weight rows: k_pad E4M3 bytes, or k_pad / 2 bytes of E2M1 nibbles on the FP4 pipe
  const int w_row = fp4 ? a.k_pad / 2 : a.k_pad;
  cuuint64_t gdim[2] = {(cuuint64_t)w_row, (cuuint64_t)w_rows};
  cuuint64_t gstride[1] = {(cuuint64_t)w_row};
  cuuint32_t box[2] = {(cuuint32_t)bk, (cuuint32_t)b_rows};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapSwizzle swz = bk == 64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B;
  for (int l = 0; l < nlayers; ++l) {
    const uint8_t* wl = nlayers > 1 ? a.layer[l].w_e4m3 : (fp4 ? a.w_fp4 : a.w_e4m3);
    const CUresult r = enc(&maps.w[l], CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, (void*)wl, gdim, gstride, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { *err = "cuTensorMapEncodeTiled failed: " + std::to_string((int)r); return 3; }
  }
  // the same weights with boxes of half the rows, for the half-width tiles
  maps.wh = maps.w[0];
  if (prm.dp_tiles < prm.layer_tiles) {
    cuuint32_t box_h[2] = {(cuuint32_t)bk, (cuuint32_t)(b_rows / 2)};
    const CUresult r = enc(&maps.wh, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, (void*)(fp4 ? a.w_fp4 : a.w_e4m3), gdim,
                           gstride, box_h, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) { *err = "cuTensorMapEncodeTiled (half) failed: " + std::to_string((int)r); return 3; }
  }

  const int units = prm.total_tiles;
  int grid = units < sms ? units : sms;
  if (pair) grid = 2 * (units < sms / 2 ? units : sms / 2);
  const bool in_tap = (a.cin % BK) == 0;
  if (flat) {
    // 1) expand the packed codes of every job into the zero-padded byte workspace (unless
    //    the caller expanded them already)
    if (!a.skip_expand || a.zero_words > 0) {
      // (with skip_expand, only the counters are cleared: an expansion of no rows)
      ExpandArgs ea{};
      for (int j = 0; j < a.njobs; ++j) ea.jobs[j] = prm.jobs[j];
      ea.njobs = a.njobs; ea.cin = a.cin; ea.pad = a.pad; ea.x_row_bytes = a.x_row_bytes;
      ea.total_rows = a.skip_expand ? 0 : rows; ea.ws = a.ws;
      ea.zero = a.zero_words > 0 ? a.zero : nullptr;
      ea.zero_words = a.zero_words;
      // one warp per run of 32 * 4 (row, 16-byte chunk) pairs, 8 warps per block
      const int64_t pairs = ea.total_rows * (a.cin / 16);
      const unsigned blocks = pairs > 0 ? (unsigned)((pairs + 1023) / 1024) : 1u;
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(blocks);
      cfg.blockDim = dim3(256);
      cfg.stream = stream;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[0].val.programmaticStreamSerializationAllowed = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      cudaError_t e;
      if (fp4) {
        // nibble image: one thread per 16 output bytes, grid-strided
        const int64_t chunks = ea.total_rows * (a.cin / 32);
        const int64_t want = (chunks + 255) / 256;
        cfg.gridDim = dim3((unsigned)(want < 4096 ? (want > 0 ? want : 1) : 4096));
        e = cudaLaunchKernelEx(&cfg, expand_nib_kernel, ea);
      } else switch (a.x_bits) {
        case 2: e = cudaLaunchKernelEx(&cfg, expand_kernel<2>, ea); break;
        case 3: e = cudaLaunchKernelEx(&cfg, expand_kernel<3>, ea); break;
        case 4: e = cudaLaunchKernelEx(&cfg, expand_kernel<4>, ea); break;
        case 8: e = cudaLaunchKernelEx(&cfg, expand_kernel<8>, ea); break;
        default: *err = "conv_tc: activation bits must be 2, 3 or 4"; return 2;
      }
      if (e == cudaSuccess) e = cudaGetLastError();
      if (e != cudaSuccess) { *err = std::string("expand launch: ") + cudaGetErrorString(e); return 3; }
    }
    if (a.expand_only) return 0;
    // 2) tensor maps over the workspace (and, for chained layers in one launch, the second
    //    image) as [rows][cin] byte matrices with bk x 128 boxes
    // (a nibble image keeps the byte image's row stride: cin bytes, the first cin / 2 used)
    cuuint64_t gd[2] = {(cuuint64_t)img_row, (cuuint64_t)rows * (cuuint64_t)prm.a_planes};
    cuuint64_t gs[1] = {(cuuint64_t)a.cin};
    cuuint32_t bx[2] = {(cuuint32_t)bk, 128};
    for (int i = 0; i < (nlayers > 1 ? 2 : 1); ++i) {
      // (a nibble image row uses 128 of every 256 bytes: fetch 128-byte lines from DRAM)
      const CUresult r2 = enc(&maps.a[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, (void*)(i == 0 ? a.ws : a.ws2), gd, gs, bx,
                              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                              fp4 ? CU_TENSOR_MAP_L2_PROMOTION_L2_128B : CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r2 != CUDA_SUCCESS) {
        *err = "cuTensorMapEncodeTiled (activations) failed: " + std::to_string((int)r2);
        return 3;
      }
    }
    if (ostage) {  // int32 outputs, no skip, 128-byte chunks (see the smem plan)
      if (fp4)
        return pair ? launch_bits<2, true, true, true, false, false, 128, true, true>(prm, maps, grid, smem, stream, err)
                    : launch_bits<2, true, true, false, false, false, 128, true, true>(prm, maps, grid, smem, stream, err);
      return pair ? launch_bits<2, true, true, true, false, false, 128, false, true>(prm, maps, grid, smem, stream, err)
                  : launch_bits<2, true, true, false, false, false, 128, false, true>(prm, maps, grid, smem, stream, err);
    }
    if (fp4) {
      if (pair)
        return a.has_skip ? launch_bits<2, true, true, true, true, false, 128, true>(prm, maps, grid, smem, stream, err)
                          : launch_bits<2, true, true, true, false, false, 128, true>(prm, maps, grid, smem, stream, err);
      return a.has_skip ? launch_bits<2, true, true, false, true, false, 128, true>(prm, maps, grid, smem, stream, err)
                        : launch_bits<2, true, true, false, false, false, 128, true>(prm, maps, grid, smem, stream, err);
    }
    if (a.split_w) {  // (no skip: the API keeps skips off the split form)
      if (pair) return launch_bits<2, true, true, true, false, true>(prm, maps, grid, smem, stream, err);
      return launch_bits<2, true, true, false, false, true>(prm, maps, grid, smem, stream, err);
    }
    if (bk == 64) {
      if (pair)
        return a.has_skip ? launch_bits<2, true, true, true, true, false, 64>(prm, maps, grid, smem, stream, err)
                          : launch_bits<2, true, true, true, false, false, 64>(prm, maps, grid, smem, stream, err);
      return a.has_skip ? launch_bits<2, true, true, false, true, false, 64>(prm, maps, grid, smem, stream, err)
                        : launch_bits<2, true, true, false, false, false, 64>(prm, maps, grid, smem, stream, err);
    }
    if (pair)
      return a.has_skip ? launch_bits<2, true, true, true, true>(prm, maps, grid, smem, stream, err)
                        : launch_bits<2, true, true, true, false>(prm, maps, grid, smem, stream, err);
    return a.has_skip ? launch_bits<2, true, true, false, true>(prm, maps, grid, smem, stream, err)
                      : launch_bits<2, true, true, false, false>(prm, maps, grid, smem, stream, err);
  }
  // in-kernel unpacking; the instantiation without skip code keeps its registers for the
  // common case
#define AQD_INKERNEL(B)                                                                                  \
  if (a.has_skip)                                                                                          \
    return in_tap ? launch_bits<B, true, false, false, true>(prm, maps, grid, smem, stream, err) \
                  : launch_bits<B, false, false, false, true>(prm, maps, grid, smem, stream, err); \
  return in_tap ? launch_bits<B, true, false, false, false>(prm, maps, grid, smem, stream, err)   \
                : launch_bits<B, false, false, false, false>(prm, maps, grid, smem, stream, err);
  switch (a.x_bits) {
    case 2: { AQD_INKERNEL(2) }
    case 3: { AQD_INKERNEL(3) }
    case 4: { AQD_INKERNEL(4) }
    default: *err = "conv_tc: activation bits must be 2, 3 or 4"; return 2;
  }
#undef AQD_INKERNEL
}

}  // namespace aqd
