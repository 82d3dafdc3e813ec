/*
 * aqd.h -- C ABI of libaqd: integer-only quantized convolution for GB300 (sm_103a).
 *
 * Implements the inference path of AQD (Chen et al., "AQD: Towards Accurate Quantized
 * Object Detection", arXiv 2007.06919, Sec. 3.2): convolution on low-bit integer codes
 * (Eq. 4) followed by a fused integer epilogue -- the folded batch-norm bias (Eq. 6,
 * optionally one parameter set per FPN level for multi-level BN, Sec. 3.2.2 / Fig. 3),
 * the dyadically rescaled skip add (Eq. 7 with F of Eq. 8), and the fixed-point rescale,
 * round and clip that produce the next layer's k-bit codes (Eq. 2). No floating point
 * value crosses a layer boundary.
 *
 * Conventions for every entry point
 *   - Pointers inside aqd_tensor / parameter structs are DEVICE pointers owned by the
 *     caller; the structs themselves live in host memory and are read before return.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream). Work is enqueued on it;
 *     no entry point synchronizes except aqd_device_status.
 *   - The library allocates no device memory. Errors come back as aqd_status; argument
 *     errors are detected before any launch and launch nothing. C++ exceptions never
 *     cross this boundary. aqd_last_error() gives a message for the calling thread.
 *   - Device-side failures (a bounded wait that timed out, a failed device check) are
 *     latched in a device status word that aqd_device_status() reads and clears.
 *
 * Tensor layout (NHWC, one "row" = the C channels of one pixel)
 *   bits 2, 4, 8 (unsigned codes, Eq. 2 range [0, 2^k - 1]):
 *     a row is a run of 32-bit little-endian words; word w holds channels [w*q, (w+1)*q)
 *     with q = 32/bits, and channel i of its word sits at bit 8*(i%4) + bits*(i/4).
 *     bits 8 is plain bytes. bits 2 and 4 need C % 32 == 0.
 *   bits 3: each group of 32 channels takes 12 bytes = 3 words; words 0 and 1 hold the
 *     low 2 bits of channels 0..15 and 16..31 in the 2-bit layout, word 2 holds bit 2 of
 *     channel i at bit 8*(i%4) + i/4. Needs C % 32 == 0.
 *   bits 32: one int32 per channel (accumulator-domain values, e.g. detection-head
 *     outputs whose scale is passed on to the next stage, Sec. 3.2.1).
 *   Rows are contiguous: pixel (n, h, w) starts at byte ((n*H + h)*W + w) * row_bytes.
 *   Code tensors must be 16-byte aligned.
 *
 * Arithmetic of one output element (all integer; rhu(v, R) = floor((v + 2^(R-1)) / 2^R),
 * rhu(v, 0) = v; sat32 saturates to int32):
 *   acc = sum_{r,s,c} x[n, ho*S - P + r, wo*S - P + s, c] * w[co, r, s, c]   (Eq. 4;
 *         taps outside the image read code 0, the zero point of Eq. 2)
 *   t   = acc + bias[l][co]                                                   (Eq. 6)
 *   with a skip tensor s (Eq. 7, F(m, n) = c / 2^d of Eq. 8):
 *     scale_main = 0 (skip coarser): t = t + rhu(s * c[l][co], d[l][co])
 *     scale_main = 1 (main coarser): t = rhu(sat32(t) * c[l][co], d[l][co]) + s
 *   u   = sat32(t)
 *   out = u                                            for 32-bit outputs
 *   out = min(max(rhu(u * M0[l][co], 31 + shift[l][co]), 0), 2^k - 1)   for k-bit codes
 *         (Eq. 2 applied to the BN output; the clip at 0 is the ReLU)
 * Weights: signed integers w, either k-bit two's complement (AQD_W_TWOS) or Eq. 3's
 * unsigned eta_w standing for 2*eta_w - (2^k - 1) (AQD_W_ODD, the odd grid of Eq. 4).
 */
#ifndef AQD_H
#define AQD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void* aqd_stream_t; /* a cudaStream_t */

typedef enum {
  AQD_OK = 0,
  AQD_ERR_INVALID = 1,      /* bad argument; nothing launched */
  AQD_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels implement */
  AQD_ERR_CUDA = 3,         /* a CUDA runtime call failed */
  AQD_ERR_TIMEOUT = 4,      /* a bounded device-side wait expired (device status) */
  AQD_ERR_DEVICE_CHECK = 5  /* a device-side consistency check failed (device status) */
} aqd_status;

enum { AQD_W_TWOS = 0, AQD_W_ODD = 1 };

typedef struct {
  int32_t n, h, w, c; /* logical NHWC shape */
  int32_t bits;       /* 2, 3, 4, 8: packed unsigned codes; 32: int32 values */
  void* data;         /* device pointer, layout above */
} aqd_tensor;

/* Per-(level, output channel) requant tables, each [levels][cout] row-major (Eq. 6, the
 * multi-level BN of Sec. 3.2.2 keeps one row per FPN level over shared weights).
 * m0/shift may be NULL when the output is 32-bit; bias may be NULL (all zero).
 * shift must lie in [-31, 31] (total right shift 31 + shift in [0, 62]). */
typedef struct {
  const int32_t* m0;
  const int8_t* shift;
  const int32_t* bias;
  int32_t levels;
} aqd_requant_params;

/* Skip-add rescale of Eq. 7/8, tables [levels][cout]: c any int32, d in [0, 62].
 * upsample = 2 reads the skip at (h/2, w/2): the nearest 2x interpolation of the FPN
 * top-down path (Sec. 3.2.3 occasion 3 with Sec. 3.2.4). */
typedef struct {
  const int32_t* c;
  const int8_t* d;
  int32_t upsample;   /* 1 or 2 */
  int32_t scale_main; /* 0: the skip is rescaled; 1: the main branch is rescaled */
} aqd_skip_params;

/* Prepared weights: written once by aqd_conv_prepare_weights, read by every conv call. */
typedef struct {
  const void* data; /* device buffer of aqd_conv_weights_bytes() bytes, 256-byte aligned */
  int32_t cout, kh, kw, cin;
  int32_t w_bits;   /* 2, 3, 4 or 8 */
  int32_t w_format; /* AQD_W_TWOS or AQD_W_ODD */
} aqd_conv_weights;

/* One image group of a grouped convolution (e.g. one FPN level). */
typedef struct {
  aqd_tensor x;    /* input codes */
  aqd_tensor y;    /* output: codes or int32 */
  aqd_tensor skip; /* skip operand; skip.data == NULL means no skip for this job */
  int32_t level;   /* row of the requant / skip tables */
} aqd_conv_job;

/* ---- host helpers ---------------------------------------------------------------- */

/* Bytes of one packed row of c channels at `bits`, or -1 if the layout does not exist. */
int64_t aqd_row_bytes(int32_t c, int32_t bits);

/* Eq. 8: the dyadic approximation m0 * 2^-(31 + shift) of `real` with |m0| < 2^31 and
 * 31 + shift in [0, 62] that minimizes the absolute error (largest shift whose
 * round-half-up m0 still fits). real = 0 gives (0, 0). Host only; no device work. */
aqd_status aqd_quantize_multiplier(double real, int32_t* m0, int8_t* shift);

const char* aqd_status_string(aqd_status s);
const char* aqd_last_error(void);

/* Reads and clears the device status word of the current device (synchronizes the
 * stream). *code receives AQD_OK or the first latched AQD_ERR_TIMEOUT /
 * AQD_ERR_DEVICE_CHECK. */
aqd_status aqd_device_status(aqd_stream_t stream, int32_t* code);

/* Diagnostics: force the convolution kernel (0 = automatic choice, 1 = tensor-core
 * kernel when the shape allows it, 2 = CUDA-core kernel, 3 = as 1 but never on CTA
 * pairs, 4 = as 1 but never on the FP4 pipe, 5 = as 1 but on neither); returns the previous
 * setting, or -1 for an unknown value. aqd_last_conv_path() reports the kernel the calling thread's last
 * successful conv call used (1 tensor core unpacking in-kernel, 2 CUDA core, 3 tensor core
 * fed from the expanded workspace, 4 the same on CTA pairs sharing each weight tile, 5 the
 * F16 tensor-core kernel of a network's first conv on a 3-channel 8-bit image with a 7x7
 * kernel, 6 the FP4 tensor-core pipe for 2-bit codes, 0 none yet). Forcing 2 also turns
 * paths 5 and 6 off.
 *
 * The FP4 pipe (path 6, kind::mxf4nvf4 with unit block scales) takes 2-bit activation codes
 * with weights |w| <= 4 (2-bit two's complement or Eq. 3's odd grid, 3-bit two's complement),
 * cin % 256 == 0 and at most 240 output channels per tile, on the workspace path, in
 * aqd_conv_int / aqd_conv_int_grouped (which expand their own input) and for the last layer
 * of aqd_conv_int_grouped_tower; each code and weight is the E2M1 value n / 2, w / 2, so
 * every product is exact and the FP32 sum is 1/4 of the integer sum, as exact as the E4M3
 * embedding. The split calls (expand / expanded / chain) always use byte images. */
int32_t aqd_set_conv_path(int32_t path);
int32_t aqd_last_conv_path(void);

/* Diagnostics (the paper has no counterpart): exercises the device-side failure path that
 * every tensor-core kernel uses, without faulting anything. One thread waits, with the
 * kernels' bounded mbarrier wait shortened to 2 ms, on a barrier that nobody arrives at; the
 * wait expires and latches AQD_ERR_TIMEOUT in the device status word; a second thread,
 * waiting the kernels' full 1 s limit on another such barrier, leaves through the kernel's
 * shared abort flag. out: 5 int64 in device memory, written by the kernel:
 * [0] 1 if the short wait expired, [1] its duration in ns, [2] 1 if the second wait
 * returned without its phase, [3] its duration in ns, [4] 1 if a control barrier whose
 * phase completed was seen as complete. The next aqd_device_status() returns
 * AQD_ERR_TIMEOUT once and clears it. */
aqd_status aqd_selftest_wait_timeout(int64_t* out, aqd_stream_t stream);

/* ---- codes <-> int32 ----------------------------------------------------------- */

/* Packs rows x c int32 codes (device) into the k-bit layout (low k bits of each value;
 * signed weights therefore pack as two's complement). bits 2/3/4/8. */
aqd_status aqd_pack_codes(const int32_t* codes, int64_t rows, int32_t c, int32_t bits,
                          void* out, aqd_stream_t stream);
/* Inverse of aqd_pack_codes; is_signed sign-extends two's-complement fields. */
aqd_status aqd_unpack_codes(const void* packed, int64_t rows, int32_t c, int32_t bits,
                            int32_t is_signed, int32_t* out, aqd_stream_t stream);

/* ---- convolution (Eq. 4 + fused epilogue) ----------------------------------------- */

/* Size of the prepared-weights buffer for a [cout][kh][kw][cin] kernel. */
size_t aqd_conv_weights_bytes(int32_t cout, int32_t kh, int32_t kw, int32_t cin);

/* Converts packed signed weights [cout][kh][kw][cin] (rows packed along cin in the
 * w_bits layout) into the prepared layout at w->data (the struct's shape fields must be
 * filled in). Done once per model load; conv calls then read the prepared form. */
aqd_status aqd_conv_prepare_weights(const void* w_packed, const aqd_conv_weights* w,
                                    void* w_prepared, size_t bytes, aqd_stream_t stream);

/* One convolution y = epilogue(conv(x, w)) at the given level of the tables.
 * skip may be NULL (no skip; sp ignored). y->bits selects the output: 2/3/4/8 codes or
 * 32 (int32, rq->m0/shift unused). rq may be NULL only for 32-bit outputs (no bias).
 * workspace (device, 256-byte aligned, owned by the caller, contents not preserved) may be
 * NULL; see aqd_conv_workspace_bytes. Results are identical with and without it. */
aqd_status aqd_conv_int(const aqd_tensor* x, const aqd_conv_weights* w, int32_t stride,
                        int32_t pad, int32_t level, const aqd_requant_params* rq,
                        const aqd_tensor* skip, const aqd_skip_params* sp, aqd_tensor* y,
                        void* workspace, size_t ws_bytes, aqd_stream_t stream);

/* The same convolution over up to 8 jobs with shared weights in ONE launch: the shared
 * detector head applied to every FPN level, each with its own level's BN row. All jobs
 * share x->c, y->bits, skip presence and the weights; spatial sizes and batch differ. */
aqd_status aqd_conv_int_grouped(const aqd_conv_job* jobs, int32_t njobs,
                                const aqd_conv_weights* w, int32_t stride, int32_t pad,
                                const aqd_requant_params* rq, const aqd_skip_params* sp,
                                void* workspace, size_t ws_bytes, aqd_stream_t stream);

/* Workspace that lets a convolution expand its packed input codes once into a zero-padded
 * byte image (one byte per code: sum over jobs of n*(h+2*pad)*(w+2*pad)*cin bytes) and feed
 * the tensor cores from it with TMA tile loads, instead of unpacking every code once per
 * kernel tap inside the convolution. Returns 0 when this path does not apply (stride != 1,
 * cin % 64 != 0, codes or weights wider than 4 bits with cin % 128 != 0, K * 3825 >= 2^24
 * with 8-bit codes or weights); a NULL or smaller workspace passed
 * to the conv calls then selects the in-kernel unpacking path. */
size_t aqd_conv_workspace_bytes(const aqd_conv_job* jobs, int32_t njobs,
                                const aqd_conv_weights* w, int32_t stride, int32_t pad);

/* The two steps of the workspace path as separate calls, for callers that expand an input
 * once and convolve it more than once (e.g. two heads over one feature map) or time the
 * steps apart. aqd_conv_expand_input writes the byte image of the jobs' inputs (only x of
 * each job is read; y, skip and level are ignored). aqd_conv_int_grouped_expanded is
 * aqd_conv_int_grouped reading that image: `workspace` must hold the expansion of exactly
 * these jobs' inputs, for the same weights' geometry, stride and pad, written by an
 * earlier aqd_conv_expand_input on this stream. Both need the workspace path to apply
 * (aqd_conv_workspace_bytes > 0) and a large enough workspace: otherwise AQD_ERR_INVALID,
 * or AQD_ERR_UNSUPPORTED when the tensor-core kernel does not take the convolution. */
aqd_status aqd_conv_expand_input(const aqd_conv_job* jobs, int32_t njobs, const aqd_conv_weights* w,
                                 int32_t stride, int32_t pad, void* workspace, size_t ws_bytes,
                                 aqd_stream_t stream);
aqd_status aqd_conv_int_grouped_expanded(const aqd_conv_job* jobs, int32_t njobs,
                                         const aqd_conv_weights* w, int32_t stride, int32_t pad,
                                         const aqd_requant_params* rq, const aqd_skip_params* sp,
                                         void* workspace, size_t ws_bytes, aqd_stream_t stream);

/* Layer chaining on the workspace path: aqd_conv_int_grouped_expanded that, besides the
 * packed k-bit outputs y (k = 2, 3 or 4), writes the same codes one byte each into
 * `next_workspace` as the zero-padded byte image that a following stride-1 convolution
 * with padding `next_pad` over these outputs reads (the layout aqd_conv_expand_input
 * writes for inputs of the outputs' shape, jobs in the same order), so that convolution
 * can be called with aqd_conv_int_grouped_expanded (or this function) without an
 * expansion pass. Only the interior of the image is written: its border must already hold
 * zeros (fill next_workspace with zeros once, or expand an input of the same shape into it
 * once; no call writes the border afterwards). Needs cout % 64 == 0, a next_workspace of
 * at least sum(n * (ho + 2 next_pad) * (wo + 2 next_pad)) * cout bytes, 256-byte aligned
 * and not overlapping `workspace`; otherwise AQD_ERR_INVALID. The paper's layers pass
 * k-bit codes from one layer to the next (Eq. 2, Fig. 1); this is the same codes stored one
 * per byte for the tensor cores. */
aqd_status aqd_conv_int_grouped_chain(const aqd_conv_job* jobs, int32_t njobs,
                                      const aqd_conv_weights* w, int32_t stride, int32_t pad,
                                      const aqd_requant_params* rq, const aqd_skip_params* sp,
                                      void* workspace, size_t ws_bytes, int32_t next_pad,
                                      void* next_workspace, size_t next_ws_bytes, aqd_stream_t stream);

/* ---- a chained tower, layers overlapped tile by tile -------------------------------- */

/* Bytes of per-tile counters that aqd_conv_int_grouped_tower needs to overlap its layers:
 * 4 x (layers - 1) x the tiles of one layer (256 output positions of the padded-width grid
 * per tile). 0 for invalid arguments or a single layer. */
size_t aqd_conv_tower_sync_bytes(const aqd_conv_job* jobs, int32_t njobs, int32_t layers, int32_t pad);

/* Runs `layers` grouped stride-1 convolutions in a chain, as the shared detector head applies
 * its tower to every FPN level (Sec. 3.2.2, Fig. 3: one weight set per layer, one parameter
 * row per level): layer i is Eq. 4 -> Eq. 6 -> Eq. 2 (no skip) of w[i] and rq[i] on layer
 * i-1's output codes.
 *   jobs: layers x njobs, row-major: jobs[i * njobs + j] is job j of layer i; its x must be
 *     jobs[(i-1) * njobs + j].y (same data pointer and shape) for i > 0; skip must be empty.
 *     Every layer keeps the spatial size: w[i].kh = w[i].kw = 2 pad + 1.
 *   Layers 0 .. layers-2 write 2/3/4-bit codes (their packed y, and, in the same epilogue,
 *     the next layer's zero-padded byte image); the last layer any output (int32 heads).
 *   ws_a, ws_b: two expanded-activation workspaces of ws_bytes each (256-byte aligned, each
 *     at least aqd_conv_workspace_bytes of every layer); layer i reads ws_a for even i, ws_b
 *     for odd i. input_expanded == 0: the call expands layer 0's input into ws_a first
 *     (aqd_conv_expand_input); nonzero: ws_a already holds it (written by that call, or by a
 *     chained previous layer). The call never writes ws_b's zero border: zero ws_b once
 *     before its first use.
 *   sync: device counters of aqd_conv_tower_sync_bytes() bytes (4-byte aligned), cleared on
 *     `stream` by the call's first kernel. With sync given, the longest leading run of
 *     layers of one shape (same weight geometry and code widths, at most 4, each running on
 *     CTA pairs with one output-channel tile, cout <= 256) runs as ONE persistent launch in
 *     layer-major tile order: each tile waits (a bounded wait, AQD_ERR_TIMEOUT on expiry)
 *     only for the tiles of the previous layer whose rows it reads. The remaining layers,
 *     and every layer when sync is NULL, run one launch each, each waiting for the whole
 *     previous launch. Calls that share sync or the workspaces must not overlap in time.
 * Every layer is validated before anything is launched; an error names the layer. */
aqd_status aqd_conv_int_grouped_tower(const aqd_conv_job* jobs, int32_t njobs, int32_t layers,
                                      const aqd_conv_weights* w, const aqd_requant_params* rq, int32_t pad,
                                      void* ws_a, void* ws_b, size_t ws_bytes, void* sync, size_t sync_bytes,
                                      int32_t input_expanded, aqd_stream_t stream);

/* ---- convolution without a caller workspace ---------------------------------------- */

/* Size of the library's own expanded-activation workspace (16 MiB per device context). */
#define AQD_STATIC_WORKSPACE_BYTES (16u << 20)

/* aqd_conv_int on the expanded-activation workspace path, with the workspace taken from a
 * fixed array inside the library instead of from the caller; it allocates nothing. The
 * paper has no counterpart: this exists for callers that cannot allocate device memory
 * (a serving loop whose device memory was all reserved at start-up, a host plugin without
 * an allocator of its own). Results are the same bytes as aqd_conv_int with a workspace.
 * The first call on a device looks the array up (cudaGetSymbolAddress); make it before any
 * stream capture. Every call on a device shares the one array: calls that overlap in time
 * (other streams, other host threads) race on it and must be ordered by the caller;
 * nothing in it needs to start at zero (each call writes every byte it reads).
 * The array's address is looked up once per (device, context): a context created later on
 * the same device (after cudaDeviceReset) gets its own lookup on its first call.
 * Argument errors return AQD_ERR_INVALID as aqd_conv_int does. Returns AQD_ERR_UNSUPPORTED,
 * launching nothing, whenever the call would not run on the workspace path: the path does
 * not apply (aqd_conv_workspace_bytes would be 0), the kernel choice would take a kernel
 * that reads no workspace (8-bit codes with a skip, or a forced CUDA-core path), or the
 * problem needs more than AQD_STATIC_WORKSPACE_BYTES. */
aqd_status aqd_conv_int_static_workspace(const aqd_tensor* x, const aqd_conv_weights* w, int32_t stride,
                                         int32_t pad, int32_t level, const aqd_requant_params* rq,
                                         const aqd_tensor* skip, const aqd_skip_params* sp, aqd_tensor* y,
                                         aqd_stream_t stream);

/* ---- training side (Sec. 3.1.2, Sec. 3.2.2) --------------------------------------- */

/* The quantizers with learnable intervals. weight = 0: Eq. 2 on activations,
 *   eta = round(clip(x / nu, 0, 1) (2^b - 1)), y = eta nu / (2^b - 1);
 * weight = 1: Eq. 3 on weights,
 *   eta = round((clip(w / nu, -1, 1) + 1) / 2 (2^b - 1)), y = (2 eta / (2^b - 1) - 1) nu.
 * "round" is half-up. Every code is decided in float32 in that order (one correctly rounded
 * division x / nu, the clip, the products, floor(v + 0.5); no fused multiply-add), so a float32
 * restatement of the equations gives the same codes and values. x, y: n float32 (device,
 * 4-byte aligned; 16-byte alignment takes vector loads); codes: n uint8 codes eta or NULL;
 * y may be NULL when codes is given. bits 1..8, nu > 0. */
aqd_status aqd_fake_quant(const float* x, int64_t n, float nu, int32_t bits, int32_t weight, float* y,
                          uint8_t* codes, aqd_stream_t stream);

/* The Straight-Through Estimator backward of aqd_fake_quant (the rounding's derivative taken
 * as 1). gx = gy where the value lies inside the clip range (0 < x / nu < 1 for Eq. 2,
 * -1 < w / nu < 1 for Eq. 3), else 0 (gx may be NULL). *gnu (one device float64) =
 * sum of gy * d y / d nu with d y / d nu = eta / Q - x / nu inside, 1 above, 0 below (Eq. 2) and
 * 2 eta / Q - 1 - w / nu inside, 1 above, -1 below (Eq. 3), Q = 2^b - 1: float32 within runs of
 * a thread, float64 across threads, a fixed order across blocks (deterministic).
 * workspace: aqd_fake_quant_backward_workspace_bytes() bytes, 8-byte aligned. */
size_t aqd_fake_quant_backward_workspace_bytes(void);
aqd_status aqd_fake_quant_backward(const float* x, const float* gy, int64_t n, float nu, int32_t bits, int32_t weight,
                                   float* gx, double* gnu, void* workspace, size_t ws_bytes, aqd_stream_t stream);

/* Batch statistics of the multi-level BN (Sec. 3.2.2, Fig. 3: one BN per FPN level over a
 * shared head) during training: for level l, the per-channel mean and biased variance of the
 * float32 tensor z[l] ([pixels[l]][c], channels last, device) over all its pixels, written as
 * float64 mean[l][c], var[l][c] (device). z and pixels are host arrays of `levels` (1..8)
 * entries. Sums are shifted by the level's first pixel, float32 over runs of 32 pixels and
 * float64 beyond. workspace: aqd_bn_level_stats_workspace_bytes(levels, c) bytes (0 for
 * invalid arguments), 8-byte aligned. */
size_t aqd_bn_level_stats_workspace_bytes(int32_t levels, int32_t c);
aqd_status aqd_bn_level_stats(const float* const* z, const int64_t* pixels, int32_t levels, int32_t c, double* mean,
                              double* var, void* workspace, size_t ws_bytes, aqd_stream_t stream);

/* ---- elementwise ------------------------------------------------------------------ */

/* y = requant(sat32(acc + bias)) per channel at `level`: Eq. 6 + Eq. 2 on an int32
 * accumulator tensor. y->bits 2/3/4/8 (or 32: sat32(acc + bias)). */
aqd_status aqd_requant(const aqd_tensor* acc, const aqd_requant_params* rq, int32_t level,
                       aqd_tensor* y, aqd_stream_t stream);

/* Eq. 7 on two tensors: a plays the accumulator (codes or int32), b the skip (codes or
 * int32, half size when sp->upsample == 2). rq NULL: 32-bit output sat32(result) with no
 * bias; otherwise bias is added to a first and y->bits selects the output as above. */
aqd_status aqd_residual_add_int(const aqd_tensor* a, const aqd_tensor* b,
                                const aqd_skip_params* sp, const aqd_requant_params* rq,
                                int32_t level, aqd_tensor* y, aqd_stream_t stream);

/* Sec. 3.2.4: k x k max-pooling (stride, zero-or-more padding < k) directly on codes;
 * padded taps are ignored. y has x's bits. */
aqd_status aqd_maxpool_codes(const aqd_tensor* x, int32_t k, int32_t stride, int32_t pad,
                             aqd_tensor* y, aqd_stream_t stream);

/* Sec. 3.2.4's max-pool fused with the first step of the workspace path of the convolution
 * that reads its output (the stem's 3x3 stride-2 pool feeding the first residual stage):
 * y = aqd_maxpool_codes(x, k, stride, pad) is written as packed codes (for any other reader,
 * e.g. a skip), and in the same pass `workspace` receives the zero-padded byte image that
 * aqd_conv_expand_input would write for the single job {x = y} of weights w with conv_stride
 * and conv_pad. A following aqd_conv_int_grouped_expanded of that job then reads it, so the
 * pooled map is never read back for its expansion and no separate pooling launch runs.
 * The pool must be 3x3 with stride 2 on 2- or 4-bit codes (else AQD_ERR_UNSUPPORTED);
 * x and y: same n, c and bits, y the pooled shape, distinct storage. The workspace path must apply to that convolution and the workspace
 * hold aqd_conv_workspace_bytes of it: otherwise AQD_ERR_UNSUPPORTED (AQD_ERR_INVALID for a
 * NULL workspace or bad shapes). Results are the bytes the two separate calls produce. */
aqd_status aqd_maxpool_expand(const aqd_tensor* x, int32_t k, int32_t stride, int32_t pad, aqd_tensor* y,
                              const aqd_conv_weights* w, int32_t conv_stride, int32_t conv_pad,
                              void* workspace, size_t ws_bytes, aqd_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* AQD_H */
