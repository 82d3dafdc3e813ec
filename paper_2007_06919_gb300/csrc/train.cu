// train.cu -- the training-side steps of AQD (Sec. 3.1.2, Sec. 3.2.2) on the GPU:
//   * the quantizers with learnable intervals, Eq. 2 (activations, [0, nu]) and Eq. 3
//     (weights, [-nu, nu]): fake-quantized values and their integer codes;
//   * their backward under the Straight-Through Estimator: the input gradient and the
//     interval's gradient (a sum over the tensor);
//   * the per-level batch statistics of the multi-level batch normalization.
// All three stream their tensors once (HBM-bound). Every rounding decision is taken in float32
// with explicit round-to-nearest operations in the order the equations state (no fused
// multiply-adds), so a code is decided exactly as a float32 restatement decides it; sums run
// in float32 over short runs and in float64 beyond.
#include <cuda_runtime.h>

#include <cstdint>

#include "kernels.h"

namespace aqd {
namespace trn {

constexpr int kThreads = 256;

// One element of Eq. 2 / Eq. 3: the code eta and the fake-quantized value.
template <bool kWeight>
__device__ __forceinline__ float quant_one(float x, float nu, float q, float s, uint32_t& eta_out) {
  const float v = __fdiv_rn(x, nu);
  float eta, y;
  if constexpr (kWeight) {
    // eta = round((clip(w / nu, -1, 1) + 1) / 2 * Q), w_bar = (2 eta / Q - 1) nu
    const float c = fminf(fmaxf(v, -1.0f), 1.0f);
    eta = floorf(__fadd_rn(__fmul_rn(__fmul_rn(__fadd_rn(c, 1.0f), 0.5f), q), 0.5f));
    y = __fmul_rn(__fsub_rn(__fdiv_rn(__fmul_rn(eta, 2.0f), q), 1.0f), nu);
  } else {
    // eta = round(clip(x / nu, 0, 1) * Q), x_bar = eta * nu / Q (s = nu / Q)
    const float c = fminf(fmaxf(v, 0.0f), 1.0f);
    eta = floorf(__fadd_rn(__fmul_rn(c, q), 0.5f));
    y = __fmul_rn(eta, s);
  }
  eta_out = (uint32_t)eta;
  return y;
}

template <bool kWeight, int kVec>
__global__ void __launch_bounds__(kThreads) fake_quant_kernel(const float* __restrict__ x, int64_t n, float nu,
                                                              float q, float s, float* __restrict__ y,
                                                              uint8_t* __restrict__ codes) {
  const int64_t units = n / kVec;
  for (int64_t u = (int64_t)blockIdx.x * kThreads + threadIdx.x; u < units; u += (int64_t)gridDim.x * kThreads) {
    if constexpr (kVec == 4) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(x) + u);
      uint32_t e0, e1, e2, e3;
      const float4 o = make_float4(quant_one<kWeight>(v.x, nu, q, s, e0), quant_one<kWeight>(v.y, nu, q, s, e1),
                                   quant_one<kWeight>(v.z, nu, q, s, e2), quant_one<kWeight>(v.w, nu, q, s, e3));
      if (y) reinterpret_cast<float4*>(y)[u] = o;
      if (codes) reinterpret_cast<uint32_t*>(codes)[u] = e0 | (e1 << 8) | (e2 << 16) | (e3 << 24);
    } else {
      uint32_t e;
      const float o = quant_one<kWeight>(__ldg(x + u), nu, q, s, e);
      if (y) y[u] = o;
      if (codes) codes[u] = (uint8_t)e;
    }
  }
  // the tail past the last whole vector (kVec = 4: at most 3 elements), by block 0
  if (kVec > 1 && blockIdx.x == 0 && threadIdx.x < n - units * kVec) {
    const int64_t i = units * kVec + threadIdx.x;
    uint32_t e;
    const float o = quant_one<kWeight>(x[i], nu, q, s, e);
    if (y) y[i] = o;
    if (codes) codes[i] = (uint8_t)e;
  }
}

// One element of the STE backward: the input gradient and d y / d nu.
template <bool kWeight>
__device__ __forceinline__ float dquant_one(float x, float gy, float nu, float q, float& dnu) {
  const float v = __fdiv_rn(x, nu);
  if constexpr (kWeight) {
    if (v > -1.0f && v < 1.0f) {
      const float eta = floorf(__fadd_rn(__fmul_rn(__fmul_rn(__fadd_rn(v, 1.0f), 0.5f), q), 0.5f));
      dnu = __fsub_rn(__fsub_rn(__fdiv_rn(__fmul_rn(eta, 2.0f), q), 1.0f), v);  // 2 eta / Q - 1 - w / nu
      return gy;
    }
    dnu = v >= 1.0f ? 1.0f : -1.0f;
    return 0.0f;
  } else {
    if (v > 0.0f && v < 1.0f) {
      const float eta = floorf(__fadd_rn(__fmul_rn(v, q), 0.5f));
      dnu = __fsub_rn(__fdiv_rn(eta, q), v);  // eta / Q - x / nu
      return gy;
    }
    dnu = v >= 1.0f ? 1.0f : 0.0f;
    return 0.0f;
  }
}

// gx (STE) and one float64 partial of sum(gy * dy/dnu) per block: float32 within a thread,
// float64 across threads.
template <bool kWeight, int kVec>
__global__ void __launch_bounds__(kThreads) fake_quant_backward_kernel(const float* __restrict__ x,
                                                                       const float* __restrict__ gy, int64_t n,
                                                                       float nu, float q, float* __restrict__ gx,
                                                                       double* __restrict__ partial) {
  __shared__ double red[kThreads / 32];
  float acc = 0.0f;
  double accd = 0.0;
  int run = 0;
  const int64_t units = n / kVec;
  for (int64_t u = (int64_t)blockIdx.x * kThreads + threadIdx.x; u < units; u += (int64_t)gridDim.x * kThreads) {
    float d0;
    if constexpr (kVec == 4) {
      const float4 xv = __ldg(reinterpret_cast<const float4*>(x) + u);
      const float4 gv = __ldg(reinterpret_cast<const float4*>(gy) + u);
      float d1, d2, d3;
      const float4 o = make_float4(dquant_one<kWeight>(xv.x, gv.x, nu, q, d0), dquant_one<kWeight>(xv.y, gv.y, nu, q, d1),
                                   dquant_one<kWeight>(xv.z, gv.z, nu, q, d2), dquant_one<kWeight>(xv.w, gv.w, nu, q, d3));
      if (gx) reinterpret_cast<float4*>(gx)[u] = o;
      acc = __fadd_rn(acc, __fadd_rn(__fadd_rn(__fmul_rn(gv.x, d0), __fmul_rn(gv.y, d1)),
                                     __fadd_rn(__fmul_rn(gv.z, d2), __fmul_rn(gv.w, d3))));
    } else {
      const float g = __ldg(gy + u);
      const float o = dquant_one<kWeight>(__ldg(x + u), g, nu, q, d0);
      if (gx) gx[u] = o;
      acc = __fadd_rn(acc, __fmul_rn(g, d0));
    }
    if (++run == 16) { accd += (double)acc; acc = 0.0f; run = 0; }
  }
  if (kVec > 1 && blockIdx.x == 0 && threadIdx.x < n - units * kVec) {
    const int64_t i = units * kVec + threadIdx.x;
    float d;
    const float o = dquant_one<kWeight>(x[i], gy[i], nu, q, d);
    if (gx) gx[i] = o;
    accd += (double)__fmul_rn(gy[i], d);
  }
  accd += (double)acc;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) accd += __shfl_xor_sync(0xffffffffu, accd, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = accd;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < kThreads / 32; ++w) t += red[w];
    partial[blockIdx.x] = t;
  }
}

// the blocks' partials summed in a fixed order (deterministic)
__global__ void sum_partials_kernel(const double* __restrict__ partial, int nparts, double* __restrict__ out) {
  __shared__ double red[kThreads];
  double t = 0.0;
  for (int i = threadIdx.x; i < nparts; i += kThreads) t += partial[i];
  red[threadIdx.x] = t;
  __syncthreads();
  for (int w = kThreads / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = red[0];
}

// Per-level batch statistics: a 1D grid whose blocks are dealt to the levels in proportion to
// their pixels (at least one each); block b of level l (of B_l) takes pixels b, b + B_l, ...;
// thread t channels t, t + 256, ... (consecutive threads read consecutive channels of one
// pixel). Each channel's values are shifted by the level's first pixel
// (k = z[0][ch]) and summed as (z - k) and (z - k)^2: float32 over runs of 32 pixels, float64
// beyond, written as one float64 partial pair per (level, block, channel). A thread's loads for 8
// pixels are issued before they are summed.
struct StatsArgs {
  const float* z[kMaxJobs];
  int64_t pixels[kMaxJobs];
  int32_t nblk[kMaxJobs], blk0[kMaxJobs];  // blocks of level l: [blk0[l], blk0[l] + nblk[l])
  int32_t levels, c;
};

__global__ void __launch_bounds__(kThreads) bn_stats_partial_kernel(const StatsArgs a, double* __restrict__ s1,
                                                                    double* __restrict__ s2) {
  int l = 0;
  while (l + 1 < a.levels && (int)blockIdx.x >= a.blk0[l + 1]) ++l;
  const int b = (int)blockIdx.x - a.blk0[l], B = a.nblk[l];
  const float* z = a.z[l];
  const int64_t P = a.pixels[l];
  for (int ch = threadIdx.x; ch < a.c; ch += kThreads) {
    const float k = P > 0 ? __ldg(z + ch) : 0.0f;
    double d1 = 0.0, d2 = 0.0;
    float f1 = 0.0f, f2 = 0.0f;
    int run = 0;
    // 8 of this block's pixels per step, their loads issued together (pixels past the level
    // contribute d = 0)
    constexpr int kU = 8;
    for (int64_t p0 = b; p0 < P; p0 += (int64_t)B * kU) {
      float d[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int64_t p = p0 + (int64_t)u * B;
        d[u] = p < P ? __fsub_rn(__ldg(z + p * a.c + ch), k) : 0.0f;
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        f1 = __fadd_rn(f1, d[u]);
        f2 = __fadd_rn(f2, __fmul_rn(d[u], d[u]));
      }
      run += kU;
      if (run >= 32) { d1 += (double)f1; d2 += (double)f2; f1 = f2 = 0.0f; run = 0; }
    }
    d1 += (double)f1;
    d2 += (double)f2;
    const int64_t o = (int64_t)blockIdx.x * a.c + ch;
    s1[o] = d1;
    s2[o] = d2;
  }
}

// mean = k + S1 / N, var = S2 / N - (S1 / N)^2 (biased, as batch normalization's training
// statistics), in float64 from the blocks' partials summed in order
__global__ void __launch_bounds__(kThreads) bn_stats_final_kernel(const StatsArgs a, const double* __restrict__ s1,
                                                                  const double* __restrict__ s2,
                                                                  double* __restrict__ mean, double* __restrict__ var) {
  const int l = blockIdx.x;
  const int64_t P = a.pixels[l];
  for (int ch = threadIdx.x; ch < a.c; ch += kThreads) {
    double t1 = 0.0, t2 = 0.0;
    for (int b = 0; b < a.nblk[l]; ++b) {
      const int64_t o = ((int64_t)a.blk0[l] + b) * a.c + ch;
      t1 += s1[o];
      t2 += s2[o];
    }
    const double k = P > 0 ? (double)a.z[l][ch] : 0.0;
    const double m1 = P > 0 ? t1 / (double)P : 0.0;
    const double v = P > 0 ? t2 / (double)P - m1 * m1 : 0.0;
    mean[(int64_t)l * a.c + ch] = k + m1;
    var[(int64_t)l * a.c + ch] = v > 0.0 ? v : 0.0;
  }
}

inline unsigned grid_for(int64_t units, int cap) {
  const int64_t b = (units + kThreads - 1) / kThreads;
  return (unsigned)(b < 1 ? 1 : (b > cap ? cap : b));
}

}  // namespace trn

static int check_launch_t(const char* what, std::string* err) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { *err = std::string(what) + ": " + cudaGetErrorString(e); return 3; }
  return 0;
}

int launch_fake_quant(const float* x, int64_t n, float nu, int32_t bits, bool weight, float* y, uint8_t* codes,
                      cudaStream_t stream, std::string* err) {
  if (n == 0) return 0;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const float q = (float)((1 << bits) - 1);
  const float s = nu / q;
  const bool v4 = ((uintptr_t)x % 16 == 0) && ((uintptr_t)y % 16 == 0) && ((uintptr_t)codes % 4 == 0);
  const int cap = (sms > 0 ? sms : 152) * 8;
  if (v4) {
    const unsigned g = trn::grid_for(n / 4, cap);
    if (weight) trn::fake_quant_kernel<true, 4><<<g, trn::kThreads, 0, stream>>>(x, n, nu, q, s, y, codes);
    else trn::fake_quant_kernel<false, 4><<<g, trn::kThreads, 0, stream>>>(x, n, nu, q, s, y, codes);
  } else {
    const unsigned g = trn::grid_for(n, cap);
    if (weight) trn::fake_quant_kernel<true, 1><<<g, trn::kThreads, 0, stream>>>(x, n, nu, q, s, y, codes);
    else trn::fake_quant_kernel<false, 1><<<g, trn::kThreads, 0, stream>>>(x, n, nu, q, s, y, codes);
  }
  return check_launch_t("fake_quant launch", err);
}

int launch_fake_quant_backward(const float* x, const float* gy, int64_t n, float nu, int32_t bits, bool weight,
                               float* gx, double* gnu, double* partial, int32_t max_parts, cudaStream_t stream,
                               std::string* err) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const float q = (float)((1 << bits) - 1);
  const bool v4 = ((uintptr_t)x % 16 == 0) && ((uintptr_t)gy % 16 == 0) && ((uintptr_t)gx % 16 == 0);
  int cap = (sms > 0 ? sms : 152) * 6;
  if (cap > max_parts) cap = max_parts;
  const unsigned g = trn::grid_for(v4 ? n / 4 : n, cap);
  if (v4) {
    if (weight) trn::fake_quant_backward_kernel<true, 4><<<g, trn::kThreads, 0, stream>>>(x, gy, n, nu, q, gx, partial);
    else trn::fake_quant_backward_kernel<false, 4><<<g, trn::kThreads, 0, stream>>>(x, gy, n, nu, q, gx, partial);
  } else {
    if (weight) trn::fake_quant_backward_kernel<true, 1><<<g, trn::kThreads, 0, stream>>>(x, gy, n, nu, q, gx, partial);
    else trn::fake_quant_backward_kernel<false, 1><<<g, trn::kThreads, 0, stream>>>(x, gy, n, nu, q, gx, partial);
  }
  trn::sum_partials_kernel<<<1, trn::kThreads, 0, stream>>>(partial, (int)g, gnu);
  return check_launch_t("fake_quant_backward launch", err);
}

// blocks of the statistics pass over all levels together: about 4 per SM
int bn_stats_blocks(int32_t levels) { return 152 * 4 > levels ? 152 * 4 : levels; }

int launch_bn_level_stats(const float* const* z, const int64_t* pixels, int32_t levels, int32_t c, double* mean,
                          double* var, double* work, cudaStream_t stream, std::string* err) {
  trn::StatsArgs a{};
  int64_t ptot = 0;
  for (int l = 0; l < levels; ++l) { a.z[l] = z[l]; a.pixels[l] = pixels[l]; ptot += pixels[l]; }
  a.levels = levels; a.c = c;
  // one block per level, the rest in proportion to the pixels: the sum stays within the cap
  const int cap = bn_stats_blocks(levels);
  int total = 0;
  for (int l = 0; l < levels; ++l) {
    const int extra = ptot > 0 ? (int)((double)(cap - levels) * (double)pixels[l] / (double)ptot) : 0;
    a.nblk[l] = 1 + extra;
    a.blk0[l] = total;
    total += a.nblk[l];
  }
  double* s1 = work;
  double* s2 = work + (size_t)cap * c;
  trn::bn_stats_partial_kernel<<<(unsigned)total, trn::kThreads, 0, stream>>>(a, s1, s2);
  trn::bn_stats_final_kernel<<<(unsigned)levels, trn::kThreads, 0, stream>>>(a, s1, s2, mean, var);
  return check_launch_t("bn_level_stats launch", err);
}

}  // namespace aqd
