// conv_direct.cu -- AQD's integer convolution (Eq. 4) on CUDA cores with exact int32
// accumulation, plus the same fused epilogue (Eq. 6, Eq. 7/8, Eq. 2).
//
// Used for the shapes the tensor-core kernel does not take: 8-bit codes (the detector's
// 8-bit input and output layers, Sec. 4 "AQD"), input channel counts that are not a
// multiple of 32 (the 3-channel image), and products too large for the exact FP32
// accumulation bound. Each thread owns one output pixel and 32 output channels; the
// block's 32 weight rows are staged in shared memory K-chunk by K-chunk.
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"

namespace aqd {
namespace direct {

constexpr int kThreads = 128;
constexpr int kKC = 256;  // K elements staged per pass

template <bool kHasSkip>
__global__ void __launch_bounds__(kThreads)
conv_direct_kernel(const ConvArgs a, int job_index) {
  __shared__ __align__(16) int16_t wsm[kKC][32];
  __shared__ EpiChan epi[32];
  const ConvJobDev& jb = a.jobs[job_index];
  const int m = blockIdx.x * kThreads + threadIdx.x;
  const int co0 = blockIdx.y * 32;
  const bool valid = m < jb.m_total;
  const int mm = valid ? m : 0;
  const int hw = jb.ho * jb.wo;
  const int img = mm / hw;
  const int rem = mm - img * hw;
  const int ho = rem / jb.wo, wo = rem - (rem / jb.wo) * jb.wo;
  const int hb = ho * a.stride - a.pad, wb = wo * a.stride - a.pad;
  const uint8_t* ximg = jb.x + (int64_t)img * jb.h * jb.w * a.x_row_bytes;

  if (threadIdx.x < 32) {
    const int ch = co0 + threadIdx.x;
    EpiChan ec{};
    if (ch < a.cout) {
      const int64_t idx = (int64_t)jb.level * a.cout + ch;
      ec.bias = a.bias ? a.bias[idx] : 0;
      if (a.out_bits != 32) { ec.m0 = a.m0[idx]; ec.r = (int8_t)(31 + a.shift[idx]); }
      if (kHasSkip) { ec.c = a.skip_c[idx]; ec.d = a.skip_d[idx]; }
    }
    epi[threadIdx.x] = ec;
  }

  int32_t acc[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) acc[j] = 0;

  for (int k0 = 0; k0 < a.k_total; k0 += kKC) {
    const int kc = min(kKC, a.k_total - k0);
    __syncthreads();
    for (int i = threadIdx.x; i < kKC * 32; i += kThreads) {
      const int kk = i / 32, j = i % 32;
      const int co = co0 + j;
      wsm[kk][j] = (kk < kc && co < a.cout) ? a.w_i16[(int64_t)co * a.k_total + k0 + kk] : (int16_t)0;
    }
    __syncthreads();
    int tap = k0 / a.cin;
    int c = k0 - tap * a.cin;
    int r = tap / a.kw, s = tap - (tap / a.kw) * a.kw;
    for (int kk = 0; kk < kc; ++kk) {
      const int hi = hb + r, wi = wb + s;
      int32_t x = 0;
      if (valid && hi >= 0 && hi < jb.h && wi >= 0 && wi < jb.w)
        x = read_code(ximg + ((int64_t)hi * jb.w + wi) * a.x_row_bytes, c, a.x_bits, false);
      if (x != 0) {
        const int4* wr = reinterpret_cast<const int4*>(&wsm[kk][0]);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int4 w4 = wr[q];
          const int32_t ww[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
          for (int h = 0; h < 4; ++h) {
            acc[8 * q + 2 * h] += x * (int32_t)(int16_t)(ww[h] & 0xFFFF);
            acc[8 * q + 2 * h + 1] += x * (ww[h] >> 16);
          }
        }
      }
      if (++c == a.cin) { c = 0; if (++s == a.kw) { s = 0; ++r; } }
    }
  }
  if (!valid) return;

  int32_t sk[32];
  if (kHasSkip) {
    const int sh = ho / a.upsample, sw = wo / a.upsample;
    const uint8_t* srow = jb.skip + (((int64_t)img * jb.skip_h + sh) * jb.skip_w + sw) * a.skip_row_bytes;
#pragma unroll 4
    for (int j = 0; j < 32; ++j) sk[j] = (co0 + j < a.cout) ? read_code(srow, co0 + j, a.skip_bits, false) : 0;
  }
  int32_t out[32];
#pragma unroll
  for (int j = 0; j < 32; ++j)
    out[j] = epilogue<kHasSkip>(acc[j], kHasSkip ? sk[j] : 0, epi[j], a.scale_main, a.out_bits);
  uint8_t* yrow = jb.y + (int64_t)m * a.y_row_bytes;
  if (a.out_bits == 32) {
    int32_t* yr = reinterpret_cast<int32_t*>(yrow);
    for (int j = 0; j < 32; ++j)
      if (co0 + j < a.cout) yr[co0 + j] = out[j];
  } else if (a.out_bits == 8 && (a.cout % 32) != 0) {
    for (int j = 0; j < 32; ++j)
      if (co0 + j < a.cout) yrow[co0 + j] = (uint8_t)out[j];
  } else {
    uint32_t g[8];
    pack_group_vals(out, a.out_bits, g);
    store_group(yrow + (co0 >> 5) * group_bytes(a.out_bits), g, a.out_bits);
  }
}

}  // namespace direct

int launch_conv_direct(const ConvArgs& a, cudaStream_t stream, std::string* err) {
  for (int j = 0; j < a.njobs; ++j) {
    const int m = a.jobs[j].m_total;
    if (m == 0) continue;
    dim3 grid((m + direct::kThreads - 1) / direct::kThreads, (a.cout + 31) / 32);
    if (a.has_skip)
      direct::conv_direct_kernel<true><<<grid, direct::kThreads, 0, stream>>>(a, j);
    else
      direct::conv_direct_kernel<false><<<grid, direct::kThreads, 0, stream>>>(a, j);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) { *err = std::string("conv_direct launch: ") + cudaGetErrorString(e); return 3; }
  }
  return 0;
}

}  // namespace aqd
