// kernels.h -- internal interface between the C-ABI layer (aqd_api.cu) and the kernels.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>
#include <string>

namespace aqd {

constexpr int kMaxJobs = 8;
constexpr int kMaxLayers = 4;  // chained layers of one shape in one tensor-core launch

struct ConvJobDev {
  const uint8_t* x;
  uint8_t* y;
  const uint8_t* skip;
  int32_t n, h, w;        // input
  int32_t ho, wo;         // output
  int32_t skip_h, skip_w;
  int32_t level;
  int32_t m_total;        // n * ho * wo
  int32_t tile_begin;     // first global tile index of this job
  // expanded-activation ("flat") path: zero-padded byte image of this job in the workspace
  int32_t row_off;        // first workspace row (one row = cin bytes) of image 0
  int32_t hp, wp;         // padded height / width (h + 2 pad, w + 2 pad)
  int32_t vimg;           // virtual output rows per image: ho * wp (columns >= wo are junk)
  int32_t tpi;            // tiles per image
  // chained output (ws_out): zero-padded byte image of this job's output for the next conv
  int32_t orow_off;       // first ws_out row (one row = cout bytes) of image 0
  int32_t ohp, owp;       // padded output height / width (ho + 2 out_pad, wo + 2 out_pad)
};

struct ConvArgs {
  ConvJobDev jobs[kMaxJobs];
  int32_t njobs;
  int32_t cin, cout, kh, kw, stride, pad;
  int32_t x_bits, out_bits, skip_bits;
  int64_t x_row_bytes, y_row_bytes, skip_row_bytes;
  const int32_t* m0;
  const int8_t* shift;
  const int32_t* bias;
  const int32_t* skip_c;
  const int8_t* skip_d;
  int32_t upsample, scale_main, has_skip;
  // prepared weights
  const uint8_t* w_e4m3;  // [cout_pad][k_pad] E4M3 sign-magnitude bytes (|w| <= 15)
  const int16_t* w_i16;   // [cout][k_total] signed integers
  int32_t cout_pad, k_total, k_pad, bn;
  int64_t acc_bound;      // K * max|x| * max|w|: bound on |accumulator|
  uint8_t* ws;            // expanded-activation workspace (NULL: in-kernel unpacking)
  int64_t ws_rows;        // rows of cin bytes available in the workspace
  int32_t skip_expand;    // workspace already holds the expansion: launch only the conv
  int32_t expand_only;    // launch only the expansion into the workspace
  int32_t no_pair;        // workspace path: use the one-CTA kernel even for 256-wide N tiles
  // 8-bit operands on the tensor cores (workspace path): activations as two planes of
  // 4-bit halves (x_lo, 16 x_hi) over which K runs twice; weights, when wider than 15, as
  // two row blocks per 128 output channels (w_lo, w_hi) whose accumulators combine as D1 + 16 D2
  int32_t a_planes;       // 1, or 2 for 8-bit activation codes
  int32_t split_w;        // weights in the split layout
  int32_t split_rows;     // weight rows of that layout (2 * round_up(cout, 128))
  uint8_t* ws_out;        // chained output: also write the output codes as the next conv's byte image
  int32_t out_pad;        // padding of that next conv
  uint32_t* status;       // device status word
  uint32_t* zero;         // words cleared by the expansion pass before the conv (NULL: none)
  int32_t zero_words;
  // Several chained layers of this shape in one launch (workspace path, CTA pairs, one N
  // tile): layer l reads ws for even l and ws2 for odd l, and writes layer[l].ws_out (the
  // other image); its tiles wait on the per-tile counters dep of layer l - 1 (see conv_tc.cu).
  // nlayers <= 1: one layer, described by the fields above.
  int32_t nlayers;
  struct Layer {
    const uint8_t* w_e4m3;
    const int32_t* m0;
    const int8_t* shift;
    const int32_t* bias;
    uint8_t* y[kMaxJobs];
    uint8_t* ws_out;
    int32_t ws_nib;
  } layer[kMaxLayers];
  uint8_t* ws2;
  uint32_t* dep;
  // The FP4 pipe (2-bit codes, |w| <= 4, cin % 256 == 0): the workspace holds a nibble image
  // (two codes per byte) and the weights come from the E2M1 block w_fp4.
  int32_t fp4;
  const uint8_t* w_fp4;
  int32_t ws_out_nib;     // the chained output image holds two codes per byte (its reader is FP4)
};
// Tiles of one layer of a grouped workspace-path launch on CTA pairs with one N tile (the
// per-layer length of a chained launch's counter array).
int64_t conv_tc_pair_tiles(const ConvArgs& a);

// Prepared-weight geometry shared by the API and the weight-prep kernel.
struct WeightGeom {
  int32_t cout, kh, kw, cin;
  int32_t k_total, k_pad, bn, cout_pad;
  int32_t split_rows;     // 2 * round_up(cout, 128): rows of the split (8-bit) weight layout
  size_t e4m3_bytes, i16_offset;
  // [cout_pad][k_pad / 2] E2M1 nibbles (weight w as the value w / 2, |w| <= 4; weight k of a
  // row in the low nibble of byte k / 2 for even k): the FP4 tensor-core B operand
  size_t fp4_offset, fp4_bytes;
  size_t total_bytes;
};
// Whether weights of this width and format are exact as E2M1 values w / 2 (|w| <= 4).
inline bool fp4_weights(int32_t w_bits, int32_t w_format) {
  const int max_abs = w_format == 0 ? (1 << (w_bits - 1)) : ((1 << w_bits) - 1);
  return max_abs <= 4;
}
WeightGeom weight_geom(int32_t cout, int32_t kh, int32_t kw, int32_t cin);

// 0 on success, else an aqd_status value; *err gets a message.
int launch_conv_tc(const ConvArgs& a, cudaStream_t stream, std::string* err);
// whether launch_conv_tc runs these arguments on CTA pairs (cta_group::2)
bool conv_tc_uses_pair(const ConvArgs& a);
int launch_conv_direct(const ConvArgs& a, cudaStream_t stream, std::string* err);
// the first conv of the network (3-channel 8-bit image, 7x7 kernel) on F16 tensor cores
bool stem_applicable(const ConvArgs& a);
int launch_stem(const ConvArgs& a, cudaStream_t stream, std::string* err);
int launch_prepare_weights(const uint8_t* w_packed, int32_t w_bits, int32_t w_format,
                           const WeightGeom& g, uint8_t* out, cudaStream_t stream,
                           std::string* err);
int launch_pack(const int32_t* codes, int64_t rows, int32_t c, int32_t bits, uint8_t* out,
                cudaStream_t stream, std::string* err);
int launch_unpack(const uint8_t* packed, int64_t rows, int32_t c, int32_t bits,
                  int32_t is_signed, int32_t* out, cudaStream_t stream, std::string* err);

struct EltArgs {
  const uint8_t* a;
  int32_t a_bits;
  int64_t a_row_bytes;
  const uint8_t* b;       // skip (may be null)
  int32_t b_bits;
  int64_t b_row_bytes;
  int32_t b_h, b_w;
  uint8_t* y;
  int32_t y_bits;
  int64_t y_row_bytes;
  int32_t n, h, w, c;
  const int32_t* m0;
  const int8_t* shift;
  const int32_t* bias;
  const int32_t* skip_c;
  const int8_t* skip_d;
  int32_t upsample, scale_main, has_skip, level;
  uint32_t* status;       // device status word (bounded waits of the staged kernel)
};
int launch_elementwise(const EltArgs& a, cudaStream_t stream, std::string* err);

struct PoolArgs {
  const uint8_t* x;
  uint8_t* y;
  int32_t n, h, w, c, bits, ho, wo, k, stride, pad;
  int64_t row_bytes;
};
int launch_maxpool(const PoolArgs& a, cudaStream_t stream, std::string* err);
// 3x3 stride-2 max-pool on 2-/4-bit codes fused with the zero-padded byte image (padding
// cpad, rows of a.c bytes, one image after another from ws) of its output
int launch_maxpool_expand(const PoolArgs& a, uint8_t* ws, int32_t cpad, cudaStream_t stream, std::string* err);

// training-side steps (train.cu): Eq. 2 / Eq. 3 fake quantization (weight: Eq. 3), its STE
// backward (gnu: one float64, the interval's gradient; partial: max_parts float64), and the
// per-level batch statistics (work: bn_stats_work_doubles(levels, c) float64)
int launch_fake_quant(const float* x, int64_t n, float nu, int32_t bits, bool weight, float* y, uint8_t* codes,
                      cudaStream_t stream, std::string* err);
int launch_fake_quant_backward(const float* x, const float* gy, int64_t n, float nu, int32_t bits, bool weight,
                               float* gx, double* gnu, double* partial, int32_t max_parts, cudaStream_t stream,
                               std::string* err);
int bn_stats_blocks(int32_t levels);
int launch_bn_level_stats(const float* const* z, const int64_t* pixels, int32_t levels, int32_t c, double* mean,
                          double* var, double* work, cudaStream_t stream, std::string* err);

// the bounded-wait self-test (selftest.cu): out receives 5 int64 values
int launch_wait_selftest(uint32_t* status, int64_t* out, cudaStream_t stream, std::string* err);

}  // namespace aqd
