// aqd_api.cu -- the C ABI of libaqd (declared in include/aqd.h): argument validation,
// kernel selection and launch. Every argument error is reported before any launch.
#include <cuda_runtime.h>

#include <climits>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>

#include "../../include/aqd.h"
#include "common.cuh"
#include "kernels.h"

namespace aqd {

static thread_local std::string g_last_error;
static thread_local int32_t g_last_path = 0;
// 0 auto, 1 tensor core, 2 direct, 3 tensor core without CTA pairs, 4 tensor core without the
// FP4 pipe, 5 tensor core without either
static int32_t g_forced_path = 0;

__device__ uint32_t g_status_word;

static aqd_status fail(aqd_status s, const std::string& msg) {
  g_last_error = msg;
  return s;
}

// Current CUDA context (driver handle, fetched through the runtime's entry-point query so
// the library needs no link against libcuda); NULL if none is current or the query fails.
typedef int (*CtxGetCurrentFn)(void**);
static void* current_context() {
  static CtxGetCurrentFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  });
  void* ctx = nullptr;
  if (fn && fn(&ctx) != 0) ctx = nullptr;
  return ctx;
}

// Device address of a __device__ symbol, looked up with that device current and cached per
// (device, context): a context created later on the same device (after cudaDeviceReset,
// say) loads the module again at another address, so it gets its own lookup.
struct SymbolCache {
  std::mutex mu;
  struct Entry { int dev; void* ctx; void* ptr; } e[64];
  int n = 0;
};
static void* symbol_ptr(SymbolCache& c, const void* symbol, const char* what, std::string* err) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    *err = "cudaGetDevice failed";
    return nullptr;
  }
  void* ctx = current_context();
  if (!ctx) {
    // no context yet on this thread (first CUDA use): make the device's primary context
    // current, so the context read here is the one the lookup and the later launches use
    if (cudaFree(nullptr) != cudaSuccess) {
      *err = "no usable CUDA context";
      return nullptr;
    }
    ctx = current_context();
  }
  std::lock_guard<std::mutex> lk(c.mu);
  for (int i = 0; i < c.n; ++i)
    if (c.e[i].dev == dev && c.e[i].ctx == ctx) return c.e[i].ptr;
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, symbol);
  if (e != cudaSuccess) {
    *err = std::string("cudaGetSymbolAddress(") + what + "): " + cudaGetErrorString(e);
    return nullptr;
  }
  const int slot = c.n < 64 ? c.n++ : (int)(((uintptr_t)ctx >> 4) % 64);  // more than 64: overwrite one
  c.e[slot] = {dev, ctx, p};
  return p;
}

static uint32_t* status_ptr(std::string* err) {
  static SymbolCache cache;
  return static_cast<uint32_t*>(symbol_ptr(cache, (const void*)&g_status_word, "status", err));
}

WeightGeom weight_geom(int32_t cout, int32_t kh, int32_t kw, int32_t cin) {
  WeightGeom g{};
  g.cout = cout; g.kh = kh; g.kw = kw; g.cin = cin;
  g.k_total = kh * kw * cin;
  g.k_pad = (g.k_total + 127) / 128 * 128;
  g.bn = cout <= 256 ? (cout + 15) / 16 * 16 : 256;  // N tile of the tensor-core kernel
  g.cout_pad = (cout + g.bn - 1) / g.bn * g.bn;
  g.split_rows = 2 * ((cout + 127) / 128 * 128);
  // the tensor-core weight block holds either layout: [cout_pad][k_pad] E4M3 bytes for
  // |w| <= 15, or, for 8-bit weights, per 128 output channels 128 rows of w_lo = w & 15 then
  // 128 rows of w_hi = w >> 4 (floor), so it is sized for the larger of the two
  g.e4m3_bytes = (size_t)(g.cout_pad > g.split_rows ? g.cout_pad : g.split_rows) * g.k_pad;
  g.i16_offset = (g.e4m3_bytes + 255) / 256 * 256;
  g.fp4_offset = (g.i16_offset + 2 * (size_t)cout * g.k_total + 255) / 256 * 256;
  g.fp4_bytes = (size_t)g.cout_pad * (size_t)(g.k_pad / 2);
  g.total_bytes = g.fp4_offset + g.fp4_bytes;
  return g;
}

static bool code_bits(int b) { return b == 2 || b == 3 || b == 4 || b == 8; }
static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

static bool check_tensor(const aqd_tensor* t, bool allow32, const char* name, std::string* err) {
  if (!t) { *err = std::string(name) + " is NULL"; return false; }
  if (!t->data) { *err = std::string(name) + "->data is NULL"; return false; }
  if (t->n <= 0 || t->h <= 0 || t->w <= 0 || t->c <= 0) { *err = std::string(name) + " has a non-positive dimension"; return false; }
  if (!(code_bits(t->bits) || (allow32 && t->bits == 32))) { *err = std::string(name) + " has unsupported bits"; return false; }
  if (row_bytes_of(t->c, t->bits) < 0) { *err = std::string(name) + ": channels must be a multiple of 32 at 2/3/4 bits"; return false; }
  if (!aligned16(t->data)) { *err = std::string(name) + "->data must be 16-byte aligned"; return false; }
  if ((int64_t)t->n * t->h * t->w >= (int64_t)INT_MAX) { *err = std::string(name) + " has too many pixels"; return false; }
  return true;
}

static int64_t max_abs_weight(int w_bits, int w_format) {
  return w_format == AQD_W_TWOS ? (1LL << (w_bits - 1)) : ((1LL << w_bits) - 1);
}

extern "C" {

int64_t aqd_row_bytes(int32_t c, int32_t bits) { return row_bytes_of(c, bits); }

const char* aqd_status_string(aqd_status s) {
  switch (s) {
    case AQD_OK: return "ok";
    case AQD_ERR_INVALID: return "invalid argument";
    case AQD_ERR_UNSUPPORTED: return "unsupported";
    case AQD_ERR_CUDA: return "CUDA error";
    case AQD_ERR_TIMEOUT: return "device wait timed out";
    case AQD_ERR_DEVICE_CHECK: return "device check failed";
  }
  return "unknown status";
}

const char* aqd_last_error(void) { return g_last_error.c_str(); }

// Eq. 8 with |c| < 2^31 and d = 31 + shift in [0, 62]: the largest d whose rounded c fits.
aqd_status aqd_quantize_multiplier(double real, int32_t* m0, int8_t* shift) {
  if (!m0 || !shift) return fail(AQD_ERR_INVALID, "null output pointer");
  if (!std::isfinite(real)) return fail(AQD_ERR_INVALID, "real must be finite");
  if (real == 0.0) { *m0 = 0; *shift = 0; return AQD_OK; }
  const double mag = std::fabs(real);
  int e = 0;
  std::frexp(mag, &e);  // mag = f * 2^e, f in [0.5, 1)
  // c = round(mag * 2^d) < 2^31 needs d <= 31 - e (and one less if rounding reaches 2^31)
  int d = 31 - e;
  if (d > 62) d = 62;
  for (; d >= 0; --d) {
    const double c = std::floor(std::ldexp(mag, d) + 0.5);
    if (c < 2147483648.0) {
      *m0 = (int32_t)(real < 0 ? -c : c);
      *shift = (int8_t)(d - 31);
      return AQD_OK;
    }
  }
  return fail(AQD_ERR_INVALID, "|real| too large for a 31-bit multiplier");
}

aqd_status aqd_device_status(aqd_stream_t stream, int32_t* code) {
  if (!code) return fail(AQD_ERR_INVALID, "code is NULL");
  std::string err;
  uint32_t* sp = status_ptr(&err);
  if (!sp) return fail(AQD_ERR_CUDA, err);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint32_t v = 0;
  cudaError_t e = cudaMemcpyAsync(&v, sp, sizeof(v), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e == cudaSuccess && v != 0) {
    e = cudaMemsetAsync(sp, 0, sizeof(uint32_t), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  }
  if (e != cudaSuccess) return fail(AQD_ERR_CUDA, std::string("device status: ") + cudaGetErrorString(e));
  *code = (int32_t)v;
  return AQD_OK;
}

int32_t aqd_set_conv_path(int32_t path) {
  if (path < 0 || path > 5) return -1;
  const int32_t old = g_forced_path;
  g_forced_path = path;
  return old;
}

int32_t aqd_last_conv_path(void) { return g_last_path; }

aqd_status aqd_selftest_wait_timeout(int64_t* out, aqd_stream_t stream) {
  if (!out || (reinterpret_cast<uintptr_t>(out) & 7) != 0) return fail(AQD_ERR_INVALID, "out must be an 8-byte aligned device pointer");
  std::string err;
  uint32_t* sp = status_ptr(&err);
  if (!sp) return fail(AQD_ERR_CUDA, err);
  const int st = launch_wait_selftest(sp, out, static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

aqd_status aqd_pack_codes(const int32_t* codes, int64_t rows, int32_t c, int32_t bits, void* out,
                          aqd_stream_t stream) {
  if (!code_bits(bits)) return fail(AQD_ERR_INVALID, "bits must be 2, 3, 4 or 8");
  if (row_bytes_of(c, bits) < 0) return fail(AQD_ERR_INVALID, "channels must be a multiple of 32 at 2/3/4 bits");
  if (rows < 0) return fail(AQD_ERR_INVALID, "rows < 0");
  if (rows == 0) return AQD_OK;
  if (!codes || !out) return fail(AQD_ERR_INVALID, "null pointer");
  if (bits != 8 && !aligned16(out)) return fail(AQD_ERR_INVALID, "out must be 16-byte aligned");
  std::string err;
  int st = launch_pack(codes, rows, c, bits, static_cast<uint8_t*>(out), static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

aqd_status aqd_unpack_codes(const void* packed, int64_t rows, int32_t c, int32_t bits, int32_t is_signed,
                            int32_t* out, aqd_stream_t stream) {
  if (!code_bits(bits)) return fail(AQD_ERR_INVALID, "bits must be 2, 3, 4 or 8");
  if (row_bytes_of(c, bits) < 0) return fail(AQD_ERR_INVALID, "channels must be a multiple of 32 at 2/3/4 bits");
  if (rows < 0) return fail(AQD_ERR_INVALID, "rows < 0");
  if (rows == 0) return AQD_OK;
  if (!packed || !out) return fail(AQD_ERR_INVALID, "null pointer");
  if (bits != 8 && !aligned16(packed)) return fail(AQD_ERR_INVALID, "packed must be 16-byte aligned");
  std::string err;
  int st = launch_unpack(static_cast<const uint8_t*>(packed), rows, c, bits, is_signed, out,
                         static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

size_t aqd_conv_weights_bytes(int32_t cout, int32_t kh, int32_t kw, int32_t cin) {
  if (cout <= 0 || kh <= 0 || kw <= 0 || cin <= 0) return 0;
  if ((int64_t)kh * kw * cin > (1 << 24)) return 0;
  return weight_geom(cout, kh, kw, cin).total_bytes;
}

static bool check_weights(const aqd_conv_weights* w, std::string* err) {
  if (!w) { *err = "weights descriptor is NULL"; return false; }
  if (w->cout <= 0 || w->kh <= 0 || w->kw <= 0 || w->cin <= 0) { *err = "weights have a non-positive dimension"; return false; }
  if (!code_bits(w->w_bits)) { *err = "w_bits must be 2, 3, 4 or 8"; return false; }
  if (w->w_format != AQD_W_TWOS && w->w_format != AQD_W_ODD) { *err = "unknown w_format"; return false; }
  if (row_bytes_of(w->cin, w->w_bits) < 0) { *err = "weight rows: cin must be a multiple of 32 at 2/3/4 bits"; return false; }
  if ((int64_t)w->kh * w->kw * w->cin > (1 << 24)) { *err = "kernel too large"; return false; }
  return true;
}

aqd_status aqd_conv_prepare_weights(const void* w_packed, const aqd_conv_weights* w, void* w_prepared,
                                    size_t bytes, aqd_stream_t stream) {
  std::string err;
  if (!check_weights(w, &err)) return fail(AQD_ERR_INVALID, err);
  if (!w_packed || !w_prepared) return fail(AQD_ERR_INVALID, "null pointer");
  if ((reinterpret_cast<uintptr_t>(w_prepared) & 255) != 0) return fail(AQD_ERR_INVALID, "w_prepared must be 256-byte aligned");
  const WeightGeom g = weight_geom(w->cout, w->kh, w->kw, w->cin);
  if (bytes < g.total_bytes) return fail(AQD_ERR_INVALID, "w_prepared buffer too small");
  int st = launch_prepare_weights(static_cast<const uint8_t*>(w_packed), w->w_bits, w->w_format, g,
                                  static_cast<uint8_t*>(w_prepared), static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

// Rows (of cin bytes) of the expanded-activation workspace, or 0 if that path does not apply.
// Whether 8-bit operands go through the split form on the tensor cores (see ConvArgs).
static bool split_weights(const aqd_conv_weights* w) { return w->w_bits == 8 && w->w_format == AQD_W_TWOS; }

// Rows (of cin bytes, per plane) of the expanded-activation workspace, or 0 if that path does
// not apply. 8-bit activations take two planes; 8-bit two's-complement weights the split
// layout. Every partial sum of the FP32 accumulator stays exact while K * 3825 < 2^24
// (x_lo * w_lo + 16 x_hi * w_lo <= 15 * 255 per term, w_hi likewise smaller).
static int64_t flat_rows(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w, int32_t stride,
                         int32_t pad, int32_t* planes = nullptr) {
  if (!jobs || njobs <= 0 || njobs > kMaxJobs || !w) return 0;
  if (stride != 1 || pad < 0 || w->cin <= 0 || w->cin % 64 != 0) return 0;
  if (w->w_format != AQD_W_TWOS && w->w_format != AQD_W_ODD) return 0;
  const bool wsplit = split_weights(w);
  // rows of 64 channels (64-byte K chunks) only for 2- to 4-bit codes and 4-bit-range weights
  const bool half_rows = w->cin % 128 != 0;
  if (half_rows && wsplit) return 0;
  if (!(w->w_bits >= 2 && w->w_bits <= 4) && !wsplit) return 0;
  const int64_t max_w = max_abs_weight(w->w_bits, w->w_format);
  if (max_w > 15 && !wsplit) return 0;
  const int64_t k = (int64_t)w->kh * w->kw * w->cin;
  int64_t rows = 0;
  int np = 1;
  for (int j = 0; j < njobs; ++j) {
    const aqd_tensor& x = jobs[j].x;
    if (!(x.bits >= 2 && x.bits <= 4) && x.bits != 8) return 0;
    if (half_rows && x.bits == 8) return 0;
    if (x.c != w->cin || x.n <= 0 || x.h <= 0 || x.w <= 0) return 0;
    if (x.bits == 8) np = 2;
    const bool wide = x.bits == 8 || wsplit;
    if (wide ? k * 3825 >= (1LL << 24) : k * ((1LL << x.bits) - 1) * max_w >= (1LL << 24)) return 0;
    rows += (int64_t)x.n * (x.h + 2 * pad) * (x.w + 2 * pad);
  }
  if (planes) *planes = np;
  // the expansion pass indexes (row, 16-byte chunk) pairs of every plane in 32 bits
  return rows * np * (w->cin / 16) < (1LL << 31) ? rows : 0;
}

size_t aqd_conv_workspace_bytes(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                int32_t stride, int32_t pad) {
  int32_t planes = 1;
  const int64_t rows = flat_rows(jobs, njobs, w, stride, pad, &planes);
  return rows > 0 ? (size_t)rows * (size_t)planes * (size_t)w->cin : 0;
}

// What one grouped call runs on the workspace path: expansion + convolution (the public
// grouped call), the expansion alone, or the convolution from an already expanded workspace.
// kStageChain is kStageConvOnly that also writes the output codes, one byte each, as the
// zero-padded byte image the next stride-1 conv reads; kStageBothChain is kStageBoth that
// does the same.
enum ConvStage { kStageBoth = 0, kStageExpandOnly = 1, kStageConvOnly = 2, kStageChain = 3, kStageBothChain = 4 };

struct ChainOut {
  int32_t pad;
  void* ws;
  size_t bytes;
};

// A validated grouped convolution, ready to launch.
struct ConvPlan {
  ConvArgs a;
  int path;     // 1 tensor core, 2 CUDA core, 5 stem
  ConvStage stage;
};

// Validates one grouped call and decides its kernel; launches nothing. require_ws: the call
// must run on the expanded-activation workspace path (else AQD_ERR_UNSUPPORTED).
// in_nib: the workspace image the convolution reads is a nibble image (two 2-bit codes per
// byte, written by a previous layer for this one); then the convolution must run on the FP4
// pipe (else AQD_ERR_UNSUPPORTED). A convolution that expands its own input (kStageBoth) takes
// the FP4 pipe whenever it applies; the other stages read byte images.
static aqd_status plan_grouped(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                               int32_t stride, int32_t pad, const aqd_requant_params* rq,
                               const aqd_skip_params* sp, void* workspace, size_t ws_bytes,
                               ConvStage stage, const ChainOut* chain, bool require_ws, ConvPlan* plan,
                               bool in_nib = false) {
  std::string err;
  if (!jobs || njobs <= 0 || njobs > kMaxJobs) return fail(AQD_ERR_INVALID, "njobs must be 1..8");
  if (!check_weights(w, &err)) return fail(AQD_ERR_INVALID, err);
  if (!w->data || (reinterpret_cast<uintptr_t>(w->data) & 255) != 0)
    return fail(AQD_ERR_INVALID, "w->data must be a 256-byte aligned prepared-weights buffer");
  if (stride <= 0 || pad < 0) return fail(AQD_ERR_INVALID, "stride must be > 0 and pad >= 0");
  const int out_bits = jobs[0].y.bits;
  const bool has_skip = jobs[0].skip.data != nullptr;
  if (!(code_bits(out_bits) || out_bits == 32)) return fail(AQD_ERR_INVALID, "y.bits must be 2, 3, 4, 8 or 32");
  if (out_bits != 32 && (!rq || !rq->m0 || !rq->shift)) return fail(AQD_ERR_INVALID, "code outputs need rq->m0 and rq->shift");
  if (rq && rq->levels <= 0) return fail(AQD_ERR_INVALID, "rq->levels must be > 0");
  if (has_skip) {
    if (!sp || !sp->c || !sp->d) return fail(AQD_ERR_INVALID, "a skip needs sp->c and sp->d");
    if (sp->upsample != 1 && sp->upsample != 2) return fail(AQD_ERR_INVALID, "sp->upsample must be 1 or 2");
    if (sp->scale_main != 0 && sp->scale_main != 1) return fail(AQD_ERR_INVALID, "sp->scale_main must be 0 or 1");
    if (!rq) return fail(AQD_ERR_INVALID, "a skip needs rq (its level count indexes sp's tables)");
  }
  ConvArgs& a = plan->a;
  a = ConvArgs{};
  plan->stage = stage;
  a.njobs = njobs;
  a.cin = w->cin; a.cout = w->cout; a.kh = w->kh; a.kw = w->kw; a.stride = stride; a.pad = pad;
  a.x_bits = jobs[0].x.bits;
  a.out_bits = out_bits;
  a.skip_bits = has_skip ? jobs[0].skip.bits : 0;
  for (int j = 0; j < njobs; ++j) {
    const aqd_conv_job& jb = jobs[j];
    const std::string nm = "jobs[" + std::to_string(j) + "]";
    if (!check_tensor(&jb.x, false, (nm + ".x").c_str(), &err)) return fail(AQD_ERR_INVALID, err);
    if (!check_tensor(&jb.y, true, (nm + ".y").c_str(), &err)) return fail(AQD_ERR_INVALID, err);
    if (jb.x.c != w->cin) return fail(AQD_ERR_INVALID, nm + ".x.c != weights cin");
    if (jb.x.bits != a.x_bits || jb.y.bits != out_bits) return fail(AQD_ERR_INVALID, nm + ": all jobs must share x.bits and y.bits");
    const int ho = (jb.x.h + 2 * pad - w->kh) / stride + 1;
    const int wo = (jb.x.w + 2 * pad - w->kw) / stride + 1;
    if (jb.x.h + 2 * pad < w->kh || jb.x.w + 2 * pad < w->kw || ho <= 0 || wo <= 0)
      return fail(AQD_ERR_INVALID, nm + ": kernel larger than the padded input");
    if (jb.y.n != jb.x.n || jb.y.h != ho || jb.y.w != wo || jb.y.c != w->cout)
      return fail(AQD_ERR_INVALID, nm + ".y shape does not match the convolution output");
    if (rq && (jb.level < 0 || jb.level >= rq->levels)) return fail(AQD_ERR_INVALID, nm + ".level out of range");
    if (!rq && jb.level != 0) return fail(AQD_ERR_INVALID, nm + ".level must be 0 without rq");
    if ((jb.skip.data != nullptr) != has_skip) return fail(AQD_ERR_INVALID, "all jobs must agree on having a skip");
    ConvJobDev& d = a.jobs[j];
    d.x = static_cast<const uint8_t*>(jb.x.data);
    d.y = static_cast<uint8_t*>(jb.y.data);
    d.n = jb.x.n; d.h = jb.x.h; d.w = jb.x.w; d.ho = ho; d.wo = wo;
    d.level = jb.level;
    d.m_total = jb.x.n * ho * wo;
    if (has_skip) {
      if (!check_tensor(&jb.skip, true, (nm + ".skip").c_str(), &err)) return fail(AQD_ERR_INVALID, err);
      if (jb.skip.bits != a.skip_bits) return fail(AQD_ERR_INVALID, "all skips must share bits");
      const int up = sp->upsample;
      if (jb.skip.n != jb.x.n || jb.skip.c != w->cout || jb.skip.h < (ho + up - 1) / up || jb.skip.w < (wo + up - 1) / up)
        return fail(AQD_ERR_INVALID, nm + ".skip shape does not cover the output");
      d.skip = static_cast<const uint8_t*>(jb.skip.data);
      d.skip_h = jb.skip.h; d.skip_w = jb.skip.w;
    }
  }
  a.x_row_bytes = row_bytes_of(a.cin, a.x_bits);
  a.y_row_bytes = row_bytes_of(a.cout, out_bits);
  a.skip_row_bytes = has_skip ? row_bytes_of(a.cout, a.skip_bits) : 0;
  a.m0 = rq ? rq->m0 : nullptr;
  a.shift = rq ? rq->shift : nullptr;
  a.bias = rq ? rq->bias : nullptr;
  a.has_skip = has_skip;
  if (has_skip) { a.skip_c = sp->c; a.skip_d = sp->d; a.upsample = sp->upsample; a.scale_main = sp->scale_main; }
  else { a.upsample = 1; }
  const WeightGeom g = weight_geom(w->cout, w->kh, w->kw, w->cin);
  a.w_e4m3 = static_cast<const uint8_t*>(w->data);
  a.w_i16 = reinterpret_cast<const int16_t*>(static_cast<const uint8_t*>(w->data) + g.i16_offset);
  a.cout_pad = g.cout_pad; a.k_total = g.k_total; a.k_pad = g.k_pad; a.bn = g.bn;
  a.split_rows = g.split_rows;
  a.a_planes = 1;
  a.status = status_ptr(&err);
  if (!a.status) return fail(AQD_ERR_CUDA, err);

  // kernel choice: tensor cores when the FP32 sum is exact, else CUDA cores (int32)
  const int64_t max_a = (1LL << a.x_bits) - 1;
  const int64_t max_w = max_abs_weight(w->w_bits, w->w_format);
  const int64_t bound = (int64_t)g.k_total * max_a * max_w;
  a.acc_bound = bound;
  const bool tc_ok = a.x_bits <= 4 && max_w <= 15 && (a.cin % 32) == 0 && bound < (1LL << 24);
  const bool direct_ok = bound < (1LL << 31);
  // 8-bit operands go to the tensor cores in split form, on the workspace path, without a skip
  int32_t wide_planes = 1;
  bool wide_ok = false;
  if (!tc_ok && workspace && !has_skip && (a.x_bits == 8 || split_weights(w))) {
    const int64_t rows = flat_rows(jobs, njobs, w, stride, pad, &wide_planes);
    wide_ok = rows > 0 && (size_t)rows * (size_t)wide_planes * (size_t)w->cin <= ws_bytes;
  }
  // the network's first conv (3-channel 8-bit image, 7x7): its own F16 tensor-core kernel
  const bool stem_ok = !tc_ok && !wide_ok && stage == kStageBoth && stem_applicable(a);
  int path = (tc_ok || wide_ok) ? 1 : (stem_ok ? 5 : 2);
  if (g_forced_path != 0 && g_forced_path != 2 && (tc_ok || wide_ok)) path = 1;
  a.no_pair = (g_forced_path == 3 || g_forced_path == 5) ? 1 : 0;
  if (g_forced_path == 2) path = 2;
  // expanded-activation path when a large enough, aligned workspace is supplied
  a.ws = nullptr;
  a.ws_rows = 0;
  if (path == 1 && workspace) {
    if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0)
      return fail(AQD_ERR_INVALID, "workspace must be 256-byte aligned");
    int32_t planes = 1;
    const int64_t rows = flat_rows(jobs, njobs, w, stride, pad, &planes);
    if (rows > 0 && (size_t)rows * (size_t)planes * (size_t)w->cin <= ws_bytes) {
      a.ws = static_cast<uint8_t*>(workspace);
      a.ws_rows = (int64_t)(ws_bytes / ((size_t)planes * (size_t)w->cin));
      a.a_planes = planes;
      a.split_w = (!tc_ok && split_weights(w)) ? 1 : 0;
    }
  }
  if (path == 1 && !tc_ok && !a.ws) path = 2;  // the split form exists only on the workspace path
  if (path == 2 && !direct_ok) return fail(AQD_ERR_UNSUPPORTED, "accumulator bound exceeds int32");
  // a caller that gave the library's own workspace wants the workspace path or nothing
  if (require_ws && (path != 1 || !a.ws))
    return fail(AQD_ERR_UNSUPPORTED, "this convolution does not run on the expanded-activation workspace path");
  if (stage != kStageBoth) {
    if (path != 1) return fail(AQD_ERR_UNSUPPORTED, "the tensor-core kernel does not take this convolution");
    if (!workspace) return fail(AQD_ERR_INVALID, "the workspace must not be NULL");
    if (!a.ws) return fail(AQD_ERR_INVALID, "the workspace path does not apply, or the workspace is too small");
  }
  a.skip_expand = (stage == kStageConvOnly || stage == kStageChain) ? 1 : 0;
  if (stage == kStageChain || stage == kStageBothChain) {
    if (!chain || !chain->ws) return fail(AQD_ERR_INVALID, "next_workspace must not be NULL");
    if ((reinterpret_cast<uintptr_t>(chain->ws) & 255) != 0) return fail(AQD_ERR_INVALID, "next_workspace must be 256-byte aligned");
    if (chain->pad < 0) return fail(AQD_ERR_INVALID, "next_pad must be >= 0");
    if (out_bits < 2 || out_bits > 4) return fail(AQD_ERR_INVALID, "a chained output needs 2-, 3- or 4-bit codes");
    if (w->cout % 64 != 0) return fail(AQD_ERR_INVALID, "a chained output needs cout % 64 == 0");
    int64_t orows = 0;
    for (int j = 0; j < njobs; ++j)
      orows += (int64_t)jobs[j].y.n * (jobs[j].y.h + 2 * chain->pad) * (jobs[j].y.w + 2 * chain->pad);
    if (orows * (w->cout / 16) >= (1LL << 31)) return fail(AQD_ERR_UNSUPPORTED, "chained output image too large");
    const size_t need = (size_t)orows * (size_t)w->cout;
    if (chain->bytes < need) return fail(AQD_ERR_INVALID, "next_workspace is too small");
    const uintptr_t i0 = reinterpret_cast<uintptr_t>(workspace), o0 = reinterpret_cast<uintptr_t>(chain->ws);
    const size_t in_need = (size_t)flat_rows(jobs, njobs, w, stride, pad) * (size_t)a.a_planes * (size_t)w->cin;
    if (i0 < o0 + need && o0 < i0 + in_need) return fail(AQD_ERR_INVALID, "workspace and next_workspace overlap");
    a.ws_out = static_cast<uint8_t*>(chain->ws);
    a.out_pad = chain->pad;
  }
  a.expand_only = stage == kStageExpandOnly ? 1 : 0;
  // The FP4 pipe (kind::mxf4nvf4): 2-bit codes and weights exact as E2M1 values w / 2
  // (|w| <= 4), read from a nibble image in 128-byte chunks (cin % 256 == 0), tiles of at most
  // 240 channels (TMEM holds two accumulators and the scales), one launch of one layer that
  // chains nothing; the accumulator bound keeps the FP32 sum exact (|sum| / 4 < 2^24).
  const bool fp4_ok = path == 1 && a.ws && !a.split_w && a.a_planes == 1 && a.x_bits == 2 && a.cin % 256 == 0 &&
                      fp4_weights(w->w_bits, w->w_format) && 2 * g.bn + 32 <= 512 && !a.ws_out &&
                      stage != kStageExpandOnly && g_forced_path != 4 && g_forced_path != 5 && bound < (1LL << 24);
  if (in_nib && !fp4_ok) return fail(AQD_ERR_UNSUPPORTED, "the FP4 pipe does not take this convolution");
  if (fp4_ok && (in_nib || stage == kStageBoth)) {
    a.fp4 = 1;
    a.w_fp4 = static_cast<const uint8_t*>(w->data) + g.fp4_offset;
  }
  plan->path = path;
  return AQD_OK;
}

static aqd_status launch_plan(const ConvPlan& plan, aqd_stream_t stream) {
  std::string err;
  const ConvArgs& a = plan.a;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int path = plan.path;
  int rc = path == 1 ? launch_conv_tc(a, st, &err) : path == 5 ? launch_stem(a, st, &err) : launch_conv_direct(a, st, &err);
  if (rc) return fail((aqd_status)rc, err);
  if (plan.stage != kStageExpandOnly)
    g_last_path = (path == 1 && a.ws) ? (a.fp4 ? 6 : conv_tc_uses_pair(a) ? 4 : 3) : path;
  return AQD_OK;
}

static aqd_status conv_grouped(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                               int32_t stride, int32_t pad, const aqd_requant_params* rq,
                               const aqd_skip_params* sp, void* workspace, size_t ws_bytes,
                               aqd_stream_t stream, ConvStage stage, const ChainOut* chain = nullptr,
                               bool require_ws = false) {
  ConvPlan plan;
  const aqd_status s = plan_grouped(jobs, njobs, w, stride, pad, rq, sp, workspace, ws_bytes, stage, chain,
                                    require_ws, &plan);
  if (s != AQD_OK) return s;
  return launch_plan(plan, stream);
}

aqd_status aqd_conv_int_grouped(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                int32_t stride, int32_t pad, const aqd_requant_params* rq,
                                const aqd_skip_params* sp, void* workspace, size_t ws_bytes,
                                aqd_stream_t stream) {
  return conv_grouped(jobs, njobs, w, stride, pad, rq, sp, workspace, ws_bytes, stream, kStageBoth);
}

aqd_status aqd_conv_int_grouped_expanded(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                         int32_t stride, int32_t pad, const aqd_requant_params* rq,
                                         const aqd_skip_params* sp, void* workspace, size_t ws_bytes,
                                         aqd_stream_t stream) {
  return conv_grouped(jobs, njobs, w, stride, pad, rq, sp, workspace, ws_bytes, stream, kStageConvOnly);
}

aqd_status aqd_conv_expand_input(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                 int32_t stride, int32_t pad, void* workspace, size_t ws_bytes,
                                 aqd_stream_t stream) {
  if (!jobs || njobs <= 0 || njobs > kMaxJobs) return fail(AQD_ERR_INVALID, "njobs must be 1..8");
  if (!workspace) return fail(AQD_ERR_INVALID, "the workspace must not be NULL");
  // only the inputs matter here: give every job an int32 output of the right shape so the
  // shared validation accepts it (nothing is written to it)
  aqd_conv_job tmp[kMaxJobs];
  for (int j = 0; j < njobs; ++j) {
    tmp[j] = jobs[j];
    tmp[j].skip = aqd_tensor{};
    tmp[j].level = 0;
    if (w && stride > 0 && pad >= 0) {
      tmp[j].y.n = jobs[j].x.n;
      tmp[j].y.h = (jobs[j].x.h + 2 * pad - w->kh) / stride + 1;
      tmp[j].y.w = (jobs[j].x.w + 2 * pad - w->kw) / stride + 1;
      tmp[j].y.c = w->cout;
    }
    tmp[j].y.bits = 32;
    tmp[j].y.data = workspace;  // any non-null aligned pointer; never dereferenced
  }
  return conv_grouped(tmp, njobs, w, stride, pad, nullptr, nullptr, workspace, ws_bytes, stream,
                      kStageExpandOnly);
}

aqd_status aqd_conv_int_grouped_chain(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                      int32_t stride, int32_t pad, const aqd_requant_params* rq,
                                      const aqd_skip_params* sp, void* workspace, size_t ws_bytes,
                                      int32_t next_pad, void* next_workspace, size_t next_ws_bytes,
                                      aqd_stream_t stream) {
  const ChainOut c{next_pad, next_workspace, next_ws_bytes};
  return conv_grouped(jobs, njobs, w, stride, pad, rq, sp, workspace, ws_bytes, stream, kStageChain, &c);
}

// ---------------------------------------------------------------- chained tower

static bool same_tensor(const aqd_tensor& a, const aqd_tensor& b) {
  return a.data == b.data && a.n == b.n && a.h == b.h && a.w == b.w && a.c == b.c && a.bits == b.bits;
}

// Validates a tower: layers x njobs jobs, layer i's inputs are layer i-1's outputs, every
// layer a stride-1 conv that keeps the spatial size (kh = kw = 2 pad + 1), no skips.
static aqd_status check_tower(const aqd_conv_job* jobs, int32_t njobs, int32_t layers,
                              const aqd_conv_weights* w, int32_t pad) {
  if (!jobs || !w) return fail(AQD_ERR_INVALID, "jobs and w must not be NULL");
  if (njobs <= 0 || njobs > kMaxJobs) return fail(AQD_ERR_INVALID, "njobs must be 1..8");
  if (layers <= 0 || layers > 64) return fail(AQD_ERR_INVALID, "layers must be 1..64");
  if (pad < 0) return fail(AQD_ERR_INVALID, "pad must be >= 0");
  for (int i = 0; i < layers; ++i) {
    if (w[i].kh != 2 * pad + 1 || w[i].kw != 2 * pad + 1)
      return fail(AQD_ERR_INVALID, "every tower layer needs kh = kw = 2 pad + 1");
    for (int j = 0; j < njobs; ++j) {
      const aqd_conv_job& jb = jobs[(size_t)i * njobs + j];
      if (jb.skip.data) return fail(AQD_ERR_INVALID, "tower layers take no skip");
      if (i > 0 && !same_tensor(jb.x, jobs[(size_t)(i - 1) * njobs + j].y))
        return fail(AQD_ERR_INVALID, "layer " + std::to_string(i) + " job " + std::to_string(j) +
                                         ": x must be the previous layer's y");
    }
  }
  return AQD_OK;
}

size_t aqd_conv_tower_sync_bytes(const aqd_conv_job* jobs, int32_t njobs, int32_t layers, int32_t pad) {
  if (!jobs || njobs <= 0 || njobs > kMaxJobs || layers < 2 || pad < 0) return 0;
  int64_t tiles = 0;
  for (int j = 0; j < njobs; ++j) {
    const aqd_tensor& x = jobs[j].x;
    if (x.n <= 0 || x.h <= 0 || x.w <= 0) return 0;
    tiles += (int64_t)x.n * (((int64_t)x.h * (x.w + 2 * pad) + 255) / 256);
  }
  return (size_t)(layers - 1) * (size_t)tiles * sizeof(uint32_t);
}

aqd_status aqd_conv_int_grouped_tower(const aqd_conv_job* jobs, int32_t njobs, int32_t layers,
                                      const aqd_conv_weights* w, const aqd_requant_params* rq, int32_t pad,
                                      void* ws_a, void* ws_b, size_t ws_bytes, void* sync, size_t sync_bytes,
                                      int32_t input_expanded, aqd_stream_t stream) {
  aqd_status s = check_tower(jobs, njobs, layers, w, pad);
  if (s != AQD_OK) return s;
  if (!rq) return fail(AQD_ERR_INVALID, "rq must not be NULL");
  if (!ws_a || (layers > 1 && !ws_b)) return fail(AQD_ERR_INVALID, "ws_a and ws_b must not be NULL");
  // every layer planned (validated, kernel chosen) before anything is launched
  ConvPlan plans[64];
  for (int i = 0; i < layers; ++i) {
    void* ws = (i % 2 == 0) ? ws_a : ws_b;
    void* nxt = (i % 2 == 0) ? ws_b : ws_a;
    const ChainOut c{pad, nxt, ws_bytes};
    const bool expand = i == 0 && !input_expanded;
    const ConvStage st = i < layers - 1 ? (expand ? kStageBothChain : kStageChain)
                                        : (expand ? kStageBoth : kStageConvOnly);
    s = plan_grouped(jobs + (size_t)i * njobs, njobs, &w[i], 1, pad, &rq[i], nullptr, ws, ws_bytes, st,
                     i < layers - 1 ? &c : nullptr, true, &plans[i]);
    if (s != AQD_OK) {
      g_last_error = "layer " + std::to_string(i) + ": " + g_last_error;
      return s;
    }
  }
  // The last layer runs on the FP4 pipe when it applies: the layer before it then writes its
  // chained output as a nibble image.
  if (layers > 1 && plans[layers - 2].a.out_bits == 2) {
    ConvPlan last;
    const aqd_status st4 = plan_grouped(jobs + (size_t)(layers - 1) * njobs, njobs, &w[layers - 1], 1, pad,
                                        &rq[layers - 1], nullptr, (layers - 1) % 2 == 0 ? ws_a : ws_b, ws_bytes,
                                        kStageConvOnly, nullptr, true, &last, true);
    if (st4 == AQD_OK) {
      plans[layers - 1] = last;
      plans[layers - 2].a.ws_out_nib = 1;
    }
  }
  // The longest prefix of layers of one shape (same weights geometry and code widths, chained
  // 2/3/4-bit outputs, CTA pairs with one N tile) runs as one launch when the caller gave
  // counters: layer l + 1's tiles start as soon as the tiles of layer l they read are stored.
  // The other layers run one launch each, each waiting for the previous launch.
  int fused = 1;
  if (sync != nullptr) {
    auto same_shape = [&](const ConvArgs& a, const ConvArgs& b) {
      return a.cin == b.cin && a.cout == b.cout && a.kh == b.kh && a.kw == b.kw && a.x_bits == b.x_bits &&
             a.out_bits == b.out_bits && a.bn == b.bn && a.cout_pad == b.cout_pad && a.k_pad == b.k_pad &&
             a.acc_bound == b.acc_bound;
    };
    auto fusable = [&](const ConvArgs& a) {
      return conv_tc_uses_pair(a) && !a.split_w && a.a_planes <= 1 && a.bn == a.cout_pad && a.ws_out != nullptr;
    };
    while (fused < layers && fused < kMaxLayers && fusable(plans[fused - 1].a) && plans[fused].path == 1 &&
           same_shape(plans[0].a, plans[fused].a) && conv_tc_uses_pair(plans[fused].a))
      ++fused;
  }
  if (fused > 1) {
    const int64_t tiles = conv_tc_pair_tiles(plans[0].a);
    const size_t need = (size_t)(fused - 1) * (size_t)tiles * sizeof(uint32_t);
    if ((reinterpret_cast<uintptr_t>(sync) & 3) != 0) return fail(AQD_ERR_INVALID, "sync must be 4-byte aligned");
    if (sync_bytes < need) return fail(AQD_ERR_INVALID, "sync is smaller than aqd_conv_tower_sync_bytes()");
    ConvPlan f = plans[0];
    ConvArgs& a = f.a;
    a.nlayers = fused;
    for (int l = 0; l < fused; ++l) {
      const ConvArgs& b = plans[l].a;
      a.layer[l].w_e4m3 = b.w_e4m3;
      a.layer[l].m0 = b.m0; a.layer[l].shift = b.shift; a.layer[l].bias = b.bias;
      for (int j = 0; j < njobs; ++j) a.layer[l].y[j] = b.jobs[j].y;
      a.layer[l].ws_out = b.ws_out;
      a.layer[l].ws_nib = b.ws_out_nib;
    }
    a.ws2 = static_cast<uint8_t*>(ws_b);
    a.dep = static_cast<uint32_t*>(sync);
    // the counters are cleared by the expansion pass that precedes the launch (an expansion of
    // no rows when the input is already expanded); the launch waits for that grid first
    a.zero = a.dep;
    a.zero_words = (int32_t)(need / sizeof(uint32_t));
    s = launch_plan(f, stream);
    if (s != AQD_OK) return s;
  }
  for (int i = fused > 1 ? fused : 0; i < layers; ++i) {
    s = launch_plan(plans[i], stream);
    if (s != AQD_OK) return s;
  }
  return AQD_OK;
}

aqd_status aqd_conv_int(const aqd_tensor* x, const aqd_conv_weights* w, int32_t stride, int32_t pad,
                        int32_t level, const aqd_requant_params* rq, const aqd_tensor* skip,
                        const aqd_skip_params* sp, aqd_tensor* y, void* workspace, size_t ws_bytes,
                        aqd_stream_t stream) {
  if (!x || !y) return fail(AQD_ERR_INVALID, "x and y must not be NULL");
  aqd_conv_job job{};
  job.x = *x;
  job.y = *y;
  if (skip) {
    job.skip = *skip;
    if (!skip->data) return fail(AQD_ERR_INVALID, "skip->data is NULL");
  }
  job.level = level;
  return aqd_conv_int_grouped(&job, 1, w, stride, pad, rq, sp, workspace, ws_bytes, stream);
}

static aqd_status elementwise(const aqd_tensor* a, const aqd_tensor* b, const aqd_skip_params* sp,
                              const aqd_requant_params* rq, int32_t level, aqd_tensor* y, aqd_stream_t stream) {
  std::string err;
  if (!check_tensor(a, true, "a", &err)) return fail(AQD_ERR_INVALID, err);
  if (!check_tensor(y, true, "y", &err)) return fail(AQD_ERR_INVALID, err);
  if (y->n != a->n || y->h != a->h || y->w != a->w || y->c != a->c) return fail(AQD_ERR_INVALID, "y shape must equal a's");
  if (y->bits != 32 && (!rq || !rq->m0 || !rq->shift)) return fail(AQD_ERR_INVALID, "code outputs need rq->m0 and rq->shift");
  if (rq && (rq->levels <= 0 || level < 0 || level >= rq->levels)) return fail(AQD_ERR_INVALID, "level out of range");
  if (!rq && level != 0) return fail(AQD_ERR_INVALID, "level must be 0 without rq");
  EltArgs e{};
  e.status = status_ptr(&err);
  if (!e.status) return fail(AQD_ERR_CUDA, err);
  e.a = static_cast<const uint8_t*>(a->data); e.a_bits = a->bits; e.a_row_bytes = row_bytes_of(a->c, a->bits);
  e.y = static_cast<uint8_t*>(y->data); e.y_bits = y->bits; e.y_row_bytes = row_bytes_of(y->c, y->bits);
  e.n = a->n; e.h = a->h; e.w = a->w; e.c = a->c; e.level = level;
  e.m0 = rq ? rq->m0 : nullptr; e.shift = rq ? rq->shift : nullptr; e.bias = rq ? rq->bias : nullptr;
  e.upsample = 1;
  if (b) {
    if (!check_tensor(b, true, "b", &err)) return fail(AQD_ERR_INVALID, err);
    if (!sp || !sp->c || !sp->d) return fail(AQD_ERR_INVALID, "sp with c and d is required");
    if (sp->upsample != 1 && sp->upsample != 2) return fail(AQD_ERR_INVALID, "sp->upsample must be 1 or 2");
    if (sp->scale_main != 0 && sp->scale_main != 1) return fail(AQD_ERR_INVALID, "sp->scale_main must be 0 or 1");
    const int up = sp->upsample;
    if (b->n != a->n || b->c != a->c || b->h < (a->h + up - 1) / up || b->w < (a->w + up - 1) / up)
      return fail(AQD_ERR_INVALID, "b shape does not cover a");
    e.b = static_cast<const uint8_t*>(b->data); e.b_bits = b->bits; e.b_row_bytes = row_bytes_of(b->c, b->bits);
    e.b_h = b->h; e.b_w = b->w;
    e.skip_c = sp->c; e.skip_d = sp->d; e.upsample = up; e.scale_main = sp->scale_main; e.has_skip = 1;
  }
  int st = launch_elementwise(e, static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

aqd_status aqd_requant(const aqd_tensor* acc, const aqd_requant_params* rq, int32_t level, aqd_tensor* y,
                       aqd_stream_t stream) {
  if (!acc || acc->bits != 32) return fail(AQD_ERR_INVALID, "acc must be an int32 tensor");
  if (!rq) return fail(AQD_ERR_INVALID, "rq is NULL");
  return elementwise(acc, nullptr, nullptr, rq, level, y, stream);
}

aqd_status aqd_residual_add_int(const aqd_tensor* a, const aqd_tensor* b, const aqd_skip_params* sp,
                                const aqd_requant_params* rq, int32_t level, aqd_tensor* y, aqd_stream_t stream) {
  if (!b) return fail(AQD_ERR_INVALID, "b is NULL");
  return elementwise(a, b, sp, rq, level, y, stream);
}

aqd_status aqd_maxpool_codes(const aqd_tensor* x, int32_t k, int32_t stride, int32_t pad, aqd_tensor* y,
                             aqd_stream_t stream) {
  std::string err;
  if (!check_tensor(x, false, "x", &err)) return fail(AQD_ERR_INVALID, err);
  if (!check_tensor(y, false, "y", &err)) return fail(AQD_ERR_INVALID, err);
  if (k <= 0 || stride <= 0 || pad < 0 || pad >= k) return fail(AQD_ERR_INVALID, "need k > 0, stride > 0, 0 <= pad < k");
  const int ho = (x->h + 2 * pad - k) / stride + 1, wo = (x->w + 2 * pad - k) / stride + 1;
  if (x->h + 2 * pad < k || x->w + 2 * pad < k) return fail(AQD_ERR_INVALID, "window larger than the padded input");
  if (y->n != x->n || y->h != ho || y->w != wo || y->c != x->c || y->bits != x->bits)
    return fail(AQD_ERR_INVALID, "y shape does not match the pooled output");
  PoolArgs p{};
  p.x = static_cast<const uint8_t*>(x->data); p.y = static_cast<uint8_t*>(y->data);
  p.n = x->n; p.h = x->h; p.w = x->w; p.c = x->c; p.bits = x->bits; p.ho = ho; p.wo = wo;
  p.k = k; p.stride = stride; p.pad = pad; p.row_bytes = row_bytes_of(x->c, x->bits);
  int st = launch_maxpool(p, static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

aqd_status aqd_maxpool_expand(const aqd_tensor* x, int32_t k, int32_t stride, int32_t pad, aqd_tensor* y,
                              const aqd_conv_weights* w, int32_t conv_stride, int32_t conv_pad, void* workspace,
                              size_t ws_bytes, aqd_stream_t stream) {
  std::string err;
  if (!check_tensor(x, false, "x", &err)) return fail(AQD_ERR_INVALID, err);
  if (!check_tensor(y, false, "y", &err)) return fail(AQD_ERR_INVALID, err);
  if (k <= 0 || stride <= 0 || pad < 0 || pad >= k) return fail(AQD_ERR_INVALID, "need k > 0, stride > 0, 0 <= pad < k");
  if (x->h + 2 * pad < k || x->w + 2 * pad < k) return fail(AQD_ERR_INVALID, "window larger than the padded input");
  const int ho = (x->h + 2 * pad - k) / stride + 1, wo = (x->w + 2 * pad - k) / stride + 1;
  if (y->n != x->n || y->h != ho || y->w != wo || y->c != x->c || y->bits != x->bits)
    return fail(AQD_ERR_INVALID, "y shape does not match the pooled output");
  if (x->data == y->data) return fail(AQD_ERR_INVALID, "x and y must not share storage");
  if (!workspace) return fail(AQD_ERR_INVALID, "the workspace must not be NULL");
  if ((x->bits != 2 && x->bits != 4) || k != 3 || stride != 2)
    return fail(AQD_ERR_UNSUPPORTED, "the fused max-pool takes a 3x3 stride-2 pool on 2- or 4-bit codes");
  // the expansion of the job {x = y} for the convolution (only its input matters)
  aqd_conv_job job{};
  job.x = *y;
  job.y.n = y->n;
  job.y.h = w && conv_stride > 0 && conv_pad >= 0 ? (y->h + 2 * conv_pad - w->kh) / conv_stride + 1 : 0;
  job.y.w = w && conv_stride > 0 && conv_pad >= 0 ? (y->w + 2 * conv_pad - w->kw) / conv_stride + 1 : 0;
  job.y.c = w ? w->cout : 0;
  job.y.bits = 32;
  job.y.data = workspace;  // any non-null aligned pointer; never dereferenced
  // validates the convolution and its workspace (the image geometry: one job, rows of cin bytes
  // from the workspace start, padding conv_pad)
  ConvPlan plan;
  const aqd_status s = plan_grouped(&job, 1, w, conv_stride, conv_pad, nullptr, nullptr, workspace, ws_bytes,
                                    kStageExpandOnly, nullptr, true, &plan);
  if (s != AQD_OK) return s;
  if (plan.path != 1 || plan.a.a_planes != 1 || plan.a.fp4 || plan.a.cin != y->c || plan.a.jobs[0].row_off != 0)
    return fail(AQD_ERR_UNSUPPORTED, "the convolution does not read a one-plane byte image");
  PoolArgs p{};
  p.x = static_cast<const uint8_t*>(x->data); p.y = static_cast<uint8_t*>(y->data);
  p.n = x->n; p.h = x->h; p.w = x->w; p.c = x->c; p.bits = x->bits; p.ho = ho; p.wo = wo;
  p.k = k; p.stride = stride; p.pad = pad; p.row_bytes = row_bytes_of(x->c, x->bits);
  const int st = launch_maxpool_expand(p, static_cast<uint8_t*>(workspace), conv_pad,
                                       static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

// ---------------------------------------------------------------- training-side steps

static constexpr int32_t kFqParts = 1024;  // float64 block partials of the interval's gradient

size_t aqd_fake_quant_backward_workspace_bytes(void) { return (size_t)kFqParts * sizeof(double); }

static bool fq_args_ok(int64_t n, float nu, int32_t bits, int32_t weight, std::string* err) {
  if (n < 0) { *err = "n must be >= 0"; return false; }
  if (!(nu > 0.0f) || !std::isfinite(nu)) { *err = "nu must be a positive finite interval"; return false; }
  if (bits < 1 || bits > 8) { *err = "bits must be 1..8"; return false; }
  if (weight != 0 && weight != 1) { *err = "weight must be 0 (Eq. 2) or 1 (Eq. 3)"; return false; }
  return true;
}

aqd_status aqd_fake_quant(const float* x, int64_t n, float nu, int32_t bits, int32_t weight, float* y,
                          uint8_t* codes, aqd_stream_t stream) {
  std::string err;
  if (!fq_args_ok(n, nu, bits, weight, &err)) return fail(AQD_ERR_INVALID, err);
  if (n > 0 && (!x || (!y && !codes))) return fail(AQD_ERR_INVALID, "x and at least one of y, codes are required");
  if (((uintptr_t)x | (uintptr_t)y) % 4 != 0) return fail(AQD_ERR_INVALID, "x and y must be 4-byte aligned");
  const int st = launch_fake_quant(x, n, nu, bits, weight != 0, y, codes, static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

aqd_status aqd_fake_quant_backward(const float* x, const float* gy, int64_t n, float nu, int32_t bits, int32_t weight,
                                   float* gx, double* gnu, void* workspace, size_t ws_bytes, aqd_stream_t stream) {
  std::string err;
  if (!fq_args_ok(n, nu, bits, weight, &err)) return fail(AQD_ERR_INVALID, err);
  if (!gnu) return fail(AQD_ERR_INVALID, "gnu is required");
  if (n > 0 && (!x || !gy)) return fail(AQD_ERR_INVALID, "x and gy are required");
  if (((uintptr_t)x | (uintptr_t)gy | (uintptr_t)gx) % 4 != 0)
    return fail(AQD_ERR_INVALID, "x, gy and gx must be 4-byte aligned");
  if (!workspace || ws_bytes < aqd_fake_quant_backward_workspace_bytes() || (uintptr_t)workspace % 8 != 0)
    return fail(AQD_ERR_INVALID, "workspace: aqd_fake_quant_backward_workspace_bytes() bytes, 8-byte aligned");
  const int st = launch_fake_quant_backward(x, gy, n, nu, bits, weight != 0, gx, gnu, static_cast<double*>(workspace),
                                            kFqParts, static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

size_t aqd_bn_level_stats_workspace_bytes(int32_t levels, int32_t c) {
  if (levels <= 0 || levels > kMaxJobs || c <= 0) return 0;
  return (size_t)2 * bn_stats_blocks(levels) * c * sizeof(double);
}

aqd_status aqd_bn_level_stats(const float* const* z, const int64_t* pixels, int32_t levels, int32_t c, double* mean,
                              double* var, void* workspace, size_t ws_bytes, aqd_stream_t stream) {
  std::string err;
  if (levels <= 0 || levels > kMaxJobs) return fail(AQD_ERR_INVALID, "levels must be 1..8");
  if (c <= 0) return fail(AQD_ERR_INVALID, "c must be > 0");
  if (!z || !pixels || !mean || !var) return fail(AQD_ERR_INVALID, "z, pixels, mean and var are required");
  for (int l = 0; l < levels; ++l) {
    if (pixels[l] < 0) return fail(AQD_ERR_INVALID, "pixels must be >= 0");
    if (pixels[l] > 0 && (!z[l] || (uintptr_t)z[l] % 4 != 0)) return fail(AQD_ERR_INVALID, "z[l] must be 4-byte aligned");
  }
  const size_t need = aqd_bn_level_stats_workspace_bytes(levels, c);
  if (!workspace || ws_bytes < need || (uintptr_t)workspace % 8 != 0)
    return fail(AQD_ERR_INVALID, "workspace: aqd_bn_level_stats_workspace_bytes() bytes, 8-byte aligned");
  const int st = launch_bn_level_stats(z, pixels, levels, c, mean, var, static_cast<double*>(workspace),
                                       static_cast<cudaStream_t>(stream), &err);
  return st ? fail((aqd_status)st, err) : AQD_OK;
}

}  // extern "C"

// ---------------------------------------------------------------- static workspace
// A fixed expanded-activation workspace inside the library, for callers that cannot
// allocate device memory themselves: code that runs after its process's device memory
// budget was fixed (a serving loop that pre-reserves everything at start-up and treats any
// later allocation as a failure), or a host plugin that holds no allocator of its own.
// One array per device context, shared by every call: the expansion pass of each call
// writes every byte the convolution then reads (zero border included), so nothing in it
// has to start at zero; two calls that overlap in time (different streams, or host
// threads) race on it and must be ordered by the caller.
static __device__ __align__(256) uint8_t g_static_ws[AQD_STATIC_WORKSPACE_BYTES];

static uint8_t* static_ws_ptr(std::string* err) {
  static SymbolCache cache;
  return static_cast<uint8_t*>(symbol_ptr(cache, (const void*)g_static_ws, "static workspace", err));
}

extern "C" {

aqd_status aqd_conv_int_static_workspace(const aqd_tensor* x, const aqd_conv_weights* w, int32_t stride,
                                         int32_t pad, int32_t level, const aqd_requant_params* rq,
                                         const aqd_tensor* skip, const aqd_skip_params* sp, aqd_tensor* y,
                                         aqd_stream_t stream) {
  // argument errors first, as aqd_conv_int reports them: AQD_ERR_INVALID with the cause
  std::string err;
  if (!x || !y) return fail(AQD_ERR_INVALID, "x and y must not be NULL");
  if (!check_weights(w, &err)) return fail(AQD_ERR_INVALID, err);
  if (!check_tensor(x, false, "x", &err) || !check_tensor(y, true, "y", &err)) return fail(AQD_ERR_INVALID, err);
  if (x->c != w->cin) return fail(AQD_ERR_INVALID, "x.c != weights cin");
  if (stride <= 0 || pad < 0) return fail(AQD_ERR_INVALID, "stride must be > 0 and pad >= 0");
  if (skip && !skip->data) return fail(AQD_ERR_INVALID, "skip->data is NULL");
  aqd_conv_job job{};
  job.x = *x;
  job.y = *y;
  if (skip) job.skip = *skip;
  job.level = level;
  const size_t need = aqd_conv_workspace_bytes(&job, 1, w, stride, pad);
  if (need == 0) return fail(AQD_ERR_UNSUPPORTED, "the expanded-activation workspace path does not apply");
  if (need > (size_t)AQD_STATIC_WORKSPACE_BYTES)
    return fail(AQD_ERR_UNSUPPORTED, "needs " + std::to_string(need) + " workspace bytes, more than the " +
                                         std::to_string((size_t)AQD_STATIC_WORKSPACE_BYTES) + " of the static one");
  uint8_t* ws = static_ws_ptr(&err);
  if (!ws) return fail(AQD_ERR_CUDA, err);
  // the call runs on the workspace path or is refused before any launch (the shared kernel
  // choice could otherwise pick a kernel that ignores the workspace, e.g. 8-bit codes with a skip)
  return conv_grouped(&job, 1, w, stride, pad, rq, sp, ws, (size_t)AQD_STATIC_WORKSPACE_BYTES, stream, kStageBoth,
                      nullptr, true);
}

}  // extern "C"
}  // namespace aqd
