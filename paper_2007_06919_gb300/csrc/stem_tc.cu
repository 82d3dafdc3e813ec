// stem_tc.cu -- the network's first convolution (Eq. 4 on the 8-bit image codes, then the
// integer epilogue: Eq. 6 bias and Eq. 2 rescale + clip) on the tcgen05 tensor cores.
//
// The image has 3 channels of 8-bit codes (0..255) and the weights are signed integers
// |w| <= 127, so the implicit GEMM has K = 7 * 7 * 3 = 147 and codes too wide for the E4M3
// embedding of conv_tc.cu. Here both operands are F16 (kind::f16): integers up to 2048 are
// exact in F16, every product is an integer, and the FP32 accumulator is exact while
// K * 255 * max|w| < 2^24 (the host checks it; 147 * 255 * 128 < 2^23).
//
// Activation encoding: the F16 bit pattern 0x6400 | x is exactly 1024 + x for x in
// [0, 1023], so one byte permute (PRMT) turns two code bytes into two F16 values 1024 + x
// and one exact F16x2 subtraction of 1024 leaves x. Padding positions (outside the image)
// hold x = 0; K positions past the receptive field meet zero weights.
//
// K order: kernel row r, then the 21 contiguous bytes (7 columns x 3 channels) of that row
// of the receptive field, padded to 22 so that element pairs stay 4-byte aligned:
// kk = 22 r + j. 7 x 22 = 154 is padded to 160 = 10 MMAs of K = 16. Operands use the
// no-swizzle K-major layout of 8-row x 16-byte core matrices (K-adjacent core matrices 128 B
// apart, 8-row groups 2560 B apart).
//
// Per CTA (one per SM, persistent over tiles of 128 consecutive output pixels):
//   warps 0..3   epilogue: tcgen05.ld (warp w reads TMEM lanes 32w.., every 32-column
//                group in turn), Eq. 6 + Eq. 2, bit-pack, store
//   warp  4      TMEM allocation + one thread issuing tcgen05.mma (M=128, N=cout, K=16)
//   warps 5..12  im2col producers: two threads per tile row (kernel rows 0..3 / 4..6),
//                word loads of the receptive field, PRMT to F16, 16-byte stores
// The weights (cout x 160 F16) stay in shared memory for the whole launch. Every wait is
// bounded: on expiry the CTA latches kStatusTimeout and unwinds.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace aqd {
namespace stem {

using namespace aqd::tc;

constexpr int kKH = 7, kKW = 7, kC = 3;
constexpr int kSeg = kKW * kC;             // 21 bytes of one receptive-field row
constexpr int kLs = kSeg + (kSeg & 1);     // 22: K elements per kernel row
constexpr int kKUsed = kKH * kLs;          // 154
constexpr int kK = (kKUsed + 15) / 16 * 16;  // 160
constexpr int kKSteps = kK / 16;
constexpr int kLBO = 128;                  // K-adjacent core matrices
constexpr int kSBO = (kK / 8) * 128;       // 8-row groups
constexpr int kStageA = 128 * kK * 2;      // one tile's A operand
constexpr int kSplitR = 4;                 // producer half 0: kernel rows [0, 4); half 1: [4, 7)
static_assert((kSplitR * kLs) % 8 == 0, "the producer halves must meet on a core-matrix boundary");
static_assert(kLs <= 24, "a receptive-field row must fit six realigned words");
// 13 warps: at most 4 per SM sub-partition, so 128 registers per thread
constexpr int kEpiWarps = 4, kWarpMma = 4, kWarpProd0 = 5, kProdWarps = 8;
constexpr int kThreads = (kWarpProd0 + kProdWarps) * 32;
constexpr uint32_t kF16Pair1024 = 0x64006400u;

struct StemParams {
  const uint8_t* x;       // [n][h][w][3] 8-bit codes
  uint8_t* y;             // [n][ho][wo] rows of y_row_bytes
  int64_t x_bytes;        // bytes of x (bounds of the word loads)
  int32_t n, h, w, ho, wo, stride, pad;
  int32_t m_total, hw_out; // n * ho * wo (< 2^31, checked on the host), ho * wo
  int32_t cout, n_pad, out_bits, level, total_tiles, stages, tmem_cols;
  int64_t y_row_bytes;
  const int32_t* m0;
  const int8_t* shift;
  const int32_t* bias;
  const int16_t* w_i16;   // [cout][147], K order (r, s, c)
  uint32_t off_b, off_cst, off_bar;
  uint32_t* status;
};


__device__ __forceinline__ uint64_t sdesc_noswz(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)(kLBO >> 4) << 16;
  d |= (uint64_t)(kSBO >> 4) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version; swizzle field 0 = none
  return d;
}

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(acc) : "memory");
}

// Two code bytes (bytes 0-1 or 2-3 of u) -> two F16 values: 1024 + x by a byte permute,
// then 1024 subtracted (exact).
__device__ __forceinline__ uint32_t f16_pair(uint32_t u, bool high) {
  const uint32_t b = __byte_perm(u, 0x64646464u, high ? 0x4342u : 0x4140u);
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(b), "r"(kF16Pair1024));
  return r;
}

// One producer thread: tile row m's K elements of kernel rows [R0, R1) (plus the zero tail
// past 154 when kTail), written as core-matrix rows of 16 bytes. Kernel row r of the
// receptive field is 21 contiguous code bytes; inside the image they are read as seven
// aligned words and realigned with funnel shifts (the 22nd byte meets a zero weight), at the
// image border byte by byte with out-of-image columns and rows read as code 0.
template <int R0, int R1, bool kTail>
__device__ __forceinline__ void build_half(const StemParams& p, int mg, uint8_t* row_dst) {
  constexpr int kWordsRows = (R1 - R0) * kLs / 2;
  constexpr int kWords = kWordsRows + (kTail ? (kK - kKUsed) / 2 : 0);
  static_assert(kWords % 4 == 0, "whole core-matrix rows");
  uint32_t o[kWords];
  const bool valid = mg < p.m_total;
  int img = 0, ho = 0, wo = 0;
  if (valid) {
    img = mg / p.hw_out;
    const int rem = mg - img * p.hw_out;
    ho = rem / p.wo;
    wo = rem - ho * p.wo;
  }
  const int wi0 = wo * p.stride - p.pad;
  const int hi0 = ho * p.stride - p.pad;
  // byte offset of (img, hi0 + R0, wi0): one kernel row further is one image row further
  const int64_t a0 = (((int64_t)img * p.h + hi0 + R0) * p.w + wi0) * kC;
  const int64_t row_step = (int64_t)p.w * kC;
  const int64_t a4_last = (a0 + (R1 - 1 - R0) * row_step) & ~(int64_t)3;
  const bool interior = valid && hi0 + R0 >= 0 && hi0 + R1 <= p.h && wi0 >= 0 && wi0 + kKW <= p.w &&
                        a4_last + 28 <= p.x_bytes;
  if (interior) {
#pragma unroll
    for (int r = R0; r < R1; ++r) {
      const int64_t a = a0 + (r - R0) * row_step;
      const uint32_t* src = reinterpret_cast<const uint32_t*>(p.x + (a & ~(int64_t)3));
      const uint32_t shr = 8u * (uint32_t)(a & 3);
      uint32_t w[7];
#pragma unroll
      for (int i = 0; i < 7; ++i) w[i] = __ldg(src + i);
#pragma unroll
      for (int q = 0; q < kLs / 2; ++q)
        o[(r - R0) * (kLs / 2) + q] = f16_pair(__funnelshift_r(w[q / 2], w[q / 2 + 1], shr), q & 1);
    }
  } else {
#pragma unroll
    for (int r = R0; r < R1; ++r) {
      const int hi = hi0 + r;
      uint32_t u[6] = {0u, 0u, 0u, 0u, 0u, 0u};
      if (valid && hi >= 0 && hi < p.h) {
        const int64_t a = a0 + (r - R0) * row_step;
#pragma unroll
        for (int j = 0; j < kSeg; ++j) {
          const int wi = wi0 + j / kC;
          if (wi >= 0 && wi < p.w) u[j / 4] |= (uint32_t)__ldg(p.x + a + j) << (8 * (j % 4));
        }
      }
#pragma unroll
      for (int q = 0; q < kLs / 2; ++q) o[(r - R0) * (kLs / 2) + q] = f16_pair(u[q / 2], q & 1);
    }
  }
#pragma unroll
  for (int q = kWordsRows; q < kWords; ++q) o[q] = 0u;
#pragma unroll
  for (int c = 0; c < kWords / 4; ++c)
    *reinterpret_cast<uint4*>(row_dst + (R0 * kLs / 8 + c) * kLBO) = make_uint4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
}

// Packs 32 k-bit codes into one group (the layout of common.cuh) and stores it at dst.
template <int kOut>
__device__ __forceinline__ void store_codes(uint8_t* dst, const uint32_t (&gw)[8]) {
  uint32_t* d = reinterpret_cast<uint32_t*>(dst);
  if constexpr (kOut == 2) {
    *reinterpret_cast<uint2*>(d) = make_uint2(gw[0], gw[1]);
  } else if constexpr (kOut == 3) {
    d[0] = gw[0]; d[1] = gw[1]; d[2] = gw[2];
  } else if constexpr (kOut == 4) {
    *reinterpret_cast<uint4*>(d) = make_uint4(gw[0], gw[1], gw[2], gw[3]);
  } else {
    reinterpret_cast<uint4*>(d)[0] = make_uint4(gw[0], gw[1], gw[2], gw[3]);
    reinterpret_cast<uint4*>(d)[1] = make_uint4(gw[4], gw[5], gw[6], gw[7]);
  }
}
template <int kOut>
__device__ __forceinline__ void put_code(uint32_t (&gw)[8], int i, uint32_t y) {
  if constexpr (kOut == 3) {
    gw[i / 16] |= (y & 3u) << (8 * (i % 4) + 2 * ((i % 16) / 4));
    gw[2] |= (y >> 2) << (8 * (i % 4) + i / 4);
  } else {
    constexpr int q = 32 / kOut;
    gw[i / q] |= y << (8 * (i % 4) + kOut * ((i % q) / 4));
  }
}

// Epilogue of 32 accumulator columns [c0, c0 + ncols) of one tile row: Eq. 6 bias, Eq. 2
// rescale + clip, packed into the k-bit group at column c0 (int32 out: stored in fours).
// The 32-bit form (every R >= 33: rhu(u * M0, R) = (mulhi(u, M0) + 2^(R-33)) >> (R-32)) and
// the int64 form are separate loops, so the common one runs as straight-line code.
template <int kOut>
__device__ __forceinline__ void epi_unit(const uint32_t (&v)[32], const int4* cst4, const EpiChan* cste, int c0,
                                         int ncols, bool fast_req, int qmax, uint8_t* yrow, bool valid) {
  if constexpr (kOut == 32) {
    int32_t* y32 = reinterpret_cast<int32_t*>(yrow) + c0;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      int32_t o[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        o[k] = add_sat(__float2int_rn(__uint_as_float(v[4 * q + k])), cst4[c0 + 4 * q + k].x);
      if (!valid) continue;
      if (ncols == 32) {
        reinterpret_cast<int4*>(y32)[q] = make_int4(o[0], o[1], o[2], o[3]);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (4 * q + k < ncols) y32[4 * q + k] = o[k];
      }
    }
  } else {
    uint32_t gw[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
    if (fast_req) {
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int4 c = cst4[c0 + i];  // bias, M0, 2^(R-33), R-32
        const int32_t u = add_sat(__float2int_rn(__uint_as_float(v[i])), c.x);
        put_code<kOut>(gw, i, (uint32_t)__vimin_s32_relu((__mulhi(u, c.y) + c.z) >> c.w, qmax));
      }
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        put_code<kOut>(gw, i, (uint32_t)epilogue<false>((int64_t)__float2int_rn(__uint_as_float(v[i])), 0,
                                                         cste[c0 + i], 0, kOut));
    }
    if (valid) store_codes<kOut>(yrow + (c0 / 32) * 4 * kOut, gw);
  }
}

__global__ void __launch_bounds__(kThreads, 1) stem_kernel(const __grid_constant__ StemParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  const uint32_t s_a = smem_u32(smem);
  const uint32_t s_b = s_a + p.off_b;
  // per output channel of the launch's level: {bias, M0, 2^(R-33), R-32} and the int64 form
  int4* cst4 = reinterpret_cast<int4*>(smem + p.off_cst);
  EpiChan* cste = reinterpret_cast<EpiChan*>(smem + p.off_cst + 256 * sizeof(int4));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + p.off_bar);
  const int S = p.stages;
  const uint32_t b_full = smem_u32(bars);
  const uint32_t b_empty = b_full + 8 * S;
  const uint32_t b_tfull = b_empty + 8 * S;
  const uint32_t b_tempty = b_tfull + 16;
  const uint32_t b_final = b_tempty + 16;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* s_fast = reinterpret_cast<int*>(tmem_slot + 2);  // AND over channels of "R >= 33"
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(b_full + 8 * s, kProdWarps);
      mbar_init(b_empty + 8 * s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(b_tfull + 8 * b, 1);
      mbar_init(b_tempty + 8 * b, kEpiWarps);
    }
    mbar_init(b_final, 1);
    *abort_flag = 0;
    *s_fast = 1;
    fence_barrier_init();
  }
  if (warp == kWarpMma) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(smem_u32(tmem_slot)), "r"(p.tmem_cols) : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();
  if (threadIdx.x == 0) grid_dep_launch();

  // weights -> F16 B operand (n_pad rows x 160, core-matrix layout); per-channel constants
  for (int e = threadIdx.x; e < p.n_pad * (kK / 2); e += blockDim.x) {
    const int n = e / (kK / 2), kk = 2 * (e - n * (kK / 2));
    uint32_t pr = 0u;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int r = (kk + h) / kLs, j = (kk + h) - r * kLs;
      int16_t wv = 0;
      if (n < p.cout && r < kKH && j < kSeg) wv = p.w_i16[(int64_t)n * (kKH * kSeg) + r * kSeg + j];
      pr |= (uint32_t)__half_as_ushort(__short2half_rn(wv)) << (16 * h);
    }
    *reinterpret_cast<uint32_t*>(smem + p.off_b + (n / 8) * kSBO + (kk / 8) * kLBO + (n % 8) * 16 + (kk % 8) * 2) = pr;
  }
  int fast = 1;
  for (int n = threadIdx.x; n < p.n_pad; n += blockDim.x) {
    EpiChan ec{};
    int4 c4 = make_int4(0, 0, 0, 0);
    if (n < p.cout) {
      const int64_t idx = (int64_t)p.level * p.cout + n;
      ec.bias = p.bias ? p.bias[idx] : 0;
      c4.x = ec.bias;
      if (p.out_bits != 32) {
        ec.m0 = p.m0[idx];
        const int r = 31 + p.shift[idx];
        ec.r = (int8_t)r;
        if (r >= 33) c4 = make_int4(ec.bias, ec.m0, 1 << (r - 33), r - 32);
        else fast = 0;
      }
    }
    cst4[n] = c4;
    cste[n] = ec;
  }
  if (!fast) atomicAnd(s_fast, 0);
  fence_proxy_async();  // generic-proxy stores of B -> visible to the MMA
  __syncthreads();
  const bool fast_req = *s_fast != 0;

  const int first = blockIdx.x, stride_t = gridDim.x;
  if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_e4m3(p.n_pad);  // F16 has the same type code 0
      const uint64_t db0 = sdesc_noswz(s_b);
      uint32_t s = 0, ph = 0, lt = 0;
      bool ok = true;
      for (int t = first; t < p.total_tiles && ok; t += stride_t, ++lt) {
        const uint32_t buf = lt & 1;
        if (!mbar_poll(b_tempty + 8 * buf, ((lt >> 1) & 1) ^ 1, abort_flag)) { ok = false; break; }
        tc_fence_after();
        if (!mbar_poll(b_full + 8 * s, ph, abort_flag)) { ok = false; break; }
        const uint64_t da0 = sdesc_noswz(s_a + s * kStageA);
        const uint32_t d = tmem_base + buf * (uint32_t)p.n_pad;
#pragma unroll
        for (int i = 0; i < kKSteps; ++i)  // K = 16 = two core matrices per step
          mma_f16(d, da0 + (uint64_t)((2 * i * kLBO) >> 4), db0 + (uint64_t)((2 * i * kLBO) >> 4), idesc,
                  i > 0 ? 1u : 0u);
        mma_commit(b_empty + 8 * s);
        mma_commit(b_tfull + 8 * buf);
        if (++s == (uint32_t)S) { s = 0; ph ^= 1; }
      }
      if (!ok) fail(abort_flag, p.status);
      mma_commit(b_final);
      if (!mbar_wait(b_final, 0, abort_flag)) fail(abort_flag, p.status);
    }
  } else if (warp >= kWarpProd0) {
    // ------------------------------------------------------------ im2col producers
    const int pt = threadIdx.x - kWarpProd0 * 32;  // 0..255
    const int row = pt & 127, half = pt >> 7;
    uint32_t s = 0, ph = 0;
    bool ok = true;
    for (int t = first; t < p.total_tiles; t += stride_t) {
      if (!mbar_wait(b_empty + 8 * s, ph ^ 1, abort_flag)) { ok = false; break; }
      uint8_t* dst = smem + s * kStageA + (row / 8) * kSBO + (row % 8) * 16;
      const int mg = t * 128 + row;
      if (half == 0) build_half<0, kSplitR, false>(p, mg, dst);
      else build_half<kSplitR, kKH, true>(p, mg, dst);
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_full + 8 * s);
      if (++s == (uint32_t)S) { s = 0; ph ^= 1; }
    }
    if (!ok) fail(abort_flag, p.status);
  } else {
    // ------------------------------------------------------------ epilogue (warps 0..3)
    const int quarter = warp;
    const uint32_t lane_base = tmem_base + ((uint32_t)(quarter * 32) << 16);
    const int ngrp = (p.cout + 31) / 32;
    const int qmax = (1 << (p.out_bits & 15)) - 1;
    uint32_t lt = 0;
    bool ok = true;
    for (int t = first; t < p.total_tiles; t += stride_t, ++lt) {
      const uint32_t buf = lt & 1;
      if (!mbar_wait(b_tfull + 8 * buf, (lt >> 1) & 1, abort_flag)) { ok = false; break; }
      tc_fence_after();
      const int mg = t * 128 + quarter * 32 + lane;
      const bool valid = mg < p.m_total;
      uint8_t* yrow = p.y + (int64_t)(valid ? mg : 0) * p.y_row_bytes;
      for (int g = 0; g < ngrp; ++g) {
        const int c0 = g * 32;
        const int ncols = p.cout - c0 < 32 ? p.cout - c0 : 32;
        uint32_t v[32];
        __syncwarp();
        tmem_ld32(lane_base + buf * (uint32_t)p.n_pad + (uint32_t)c0, ncols == 32, v);
        tmem_wait_ld();
        reg_fence32(v);
        if (ncols < 32) {
#pragma unroll
          for (int i = 16; i < 32; ++i) v[i] = 0u;  // only 16 columns were loaded
        }
        switch (p.out_bits) {
          case 2: epi_unit<2>(v, cst4, cste, c0, ncols, fast_req, qmax, yrow, valid); break;
          case 3: epi_unit<3>(v, cst4, cste, c0, ncols, fast_req, qmax, yrow, valid); break;
          case 4: epi_unit<4>(v, cst4, cste, c0, ncols, fast_req, qmax, yrow, valid); break;
          case 8: epi_unit<8>(v, cst4, cste, c0, ncols, fast_req, qmax, yrow, valid); break;
          default: epi_unit<32>(v, cst4, cste, c0, ncols, fast_req, qmax, yrow, valid); break;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(b_tempty + 8 * buf);
    }
    if (!ok) fail(abort_flag, p.status);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(p.tmem_cols) : "memory");
  }
}

}  // namespace stem

bool stem_applicable(const ConvArgs& a) {
  return a.njobs == 1 && a.x_bits == 8 && a.cin == stem::kC && a.kh == stem::kKH && a.kw == stem::kKW &&
         !a.has_skip && a.cout % 16 == 0 && a.cout <= 256 && a.k_total == stem::kKH * stem::kSeg &&
         a.acc_bound < (1LL << 24);  // K * 255 * max|w|: the FP32 sum is exact
}

int launch_stem(const ConvArgs& a, cudaStream_t stream, std::string* err) {
  using namespace stem;
  const ConvJobDev& jb = a.jobs[0];
  StemParams p{};
  p.x = jb.x;
  p.y = jb.y;
  p.x_bytes = (int64_t)jb.n * jb.h * jb.w * kC;
  p.n = jb.n; p.h = jb.h; p.w = jb.w; p.ho = jb.ho; p.wo = jb.wo;
  p.stride = a.stride; p.pad = a.pad;
  p.cout = a.cout;
  p.n_pad = (a.cout + 15) / 16 * 16;
  p.out_bits = a.out_bits;
  p.level = jb.level;
  p.y_row_bytes = a.y_row_bytes;
  p.m0 = a.m0; p.shift = a.shift; p.bias = a.bias;
  p.w_i16 = a.w_i16;
  p.status = a.status;
  const int64_t m_total = (int64_t)jb.n * jb.ho * jb.wo;
  if (m_total + 128 >= (1LL << 31)) { *err = "stem conv: more than 2^31 output pixels"; return 2; }
  p.m_total = (int32_t)m_total;
  p.hw_out = jb.ho * jb.wo;
  p.total_tiles = (int32_t)((m_total + 127) / 128);
  if (p.total_tiles == 0) return 0;
  int cols = 32;
  while (cols < 2 * p.n_pad) cols *= 2;
  p.tmem_cols = cols;
  int dev = 0, sms = 0, max_smem = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const uint32_t b_bytes = (uint32_t)p.n_pad * kK * 2;
  const uint32_t cst_bytes = (uint32_t)(256 * (sizeof(int4) + sizeof(EpiChan)));
  int stages = 4;
  uint32_t total = 0;
  for (; stages >= 2; --stages) {
    p.off_b = (uint32_t)stages * kStageA;
    p.off_cst = p.off_b + b_bytes;
    p.off_bar = (p.off_cst + cst_bytes + 15) / 16 * 16;
    total = p.off_bar + 8 * (2 * stages + 5) + 16 + 1024;  // barriers, TMEM slot + 2 flags, alignment
    if ((int)total <= max_smem) break;
  }
  if (stages < 2) { *err = "stem conv: shared memory too small"; return 2; }
  p.stages = stages;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [&] {
    attr_err = cudaFuncSetAttribute(stem_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem);
  });
  if (attr_err != cudaSuccess) {
    *err = std::string("stem conv: shared-memory attribute: ") + cudaGetErrorString(attr_err);
    return 3;
  }
  const int grid = (int)(p.total_tiles < sms ? p.total_tiles : sms);
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = total;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, stem_kernel, p);
  if (e != cudaSuccess) {
    *err = std::string("stem conv launch: ") + cudaGetErrorString(e);
    return 3;
  }
  return 0;
}

}  // namespace aqd
