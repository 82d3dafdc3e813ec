/*
 * aqd_ref.h -- declarations of the CPU oracle for AQD's integer-only inference path.
 *
 * TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and the CPU-baseline
 * leg of bench.py may load this library. The product library (include/aqd.h) shares
 * no code, header, table or helper with it.
 *
 * Every pointer here is a HOST pointer. All arithmetic is exact integer arithmetic
 * in int64; there is no floating point anywhere in the oracle except the double
 * argument of aqd_ref_quantize_multiplier (Eq. 8's real ratio).
 *
 * Packed code layout (the oracle's own restatement of the format it checks):
 *   bits 2, 4, 8: a pixel row of C codes is a run of 32-bit little-endian words;
 *     word w holds codes [w*q, (w+1)*q) with q = 32/bits; the code with index i
 *     inside its word sits at bit 8*(i%4) + bits*(i/4).  (bits 8: plain bytes.)
 *   bits 3: groups of 32 codes take 12 bytes = 3 words; words 0 and 1 hold the low
 *     two bits of codes 0..15 and 16..31 in the 2-bit layout; word 2 holds bit 2 of
 *     code i (0..31) at bit 8*(i%4) + i/4.
 *   bits 32: plain int32 per channel.
 *   C must be a multiple of 32 for bits 2, 3 and 4.
 */
#ifndef AQD_REF_H
#define AQD_REF_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { AQD_REF_OK = 0, AQD_REF_ERR_INVALID = 1 };
enum { AQD_REF_W_TWOS = 0, AQD_REF_W_ODD = 1 };

typedef struct {
  int32_t n, h, w, c;
  int32_t bits;  /* 2, 3, 4, 8: packed unsigned codes; 32: int32 values */
  void* data;
} aqd_ref_tensor;

/* Per-(level, channel) tables, each [levels][cout] row-major. bias may be NULL (0). */
typedef struct {
  const int32_t* m0;
  const int8_t* shift;  /* total right shift R = 31 + shift, R in [0, 62] */
  const int32_t* bias;
  int32_t levels;
} aqd_ref_requant;

typedef struct {
  const aqd_ref_tensor* skip;  /* codes (unsigned) or int32 */
  const int32_t* c;            /* [levels][cout] */
  const int8_t* d;             /* [levels][cout], 0..62 */
  int32_t upsample;            /* 1, or 2 = nearest 2x read skip[h/2][w/2] */
  int32_t scale_main;          /* 0: t + rhu(s*c, d); 1: rhu(sat32(t)*c, d) + s */
} aqd_ref_residual;

int64_t aqd_ref_row_bytes(int32_t c, int32_t bits);
int aqd_ref_pack(const int32_t* codes, int64_t rows, int32_t c, int32_t bits, uint8_t* out);
int aqd_ref_unpack(const uint8_t* packed, int64_t rows, int32_t c, int32_t bits,
                   int32_t is_signed, int32_t* out);

int aqd_ref_quantize_multiplier(double real, int32_t* m0, int8_t* shift);

int aqd_ref_conv_int(const aqd_ref_tensor* x, const uint8_t* w_packed, int32_t w_bits,
                     int32_t w_format, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                     int32_t cout, int32_t level, const aqd_ref_requant* rq,
                     const aqd_ref_residual* res, int32_t out_bits, aqd_ref_tensor* y);

/* Same computation for a list of output pixels only (flattened n*Ho*Wo + ho*Wo + wo);
 * writes out[npix][cout] unpacked (codes or int32). Used at full sizes. */
int aqd_ref_conv_int_pixels(const aqd_ref_tensor* x, const uint8_t* w_packed,
                            int32_t w_bits, int32_t w_format, int32_t kh, int32_t kw,
                            int32_t stride, int32_t pad, int32_t cout, int32_t level,
                            const aqd_ref_requant* rq, const aqd_ref_residual* res,
                            int32_t out_bits, int32_t out_h, int32_t out_w,
                            const int64_t* pix, int64_t npix, int32_t* out);

int aqd_ref_requant_tensor(const aqd_ref_tensor* acc, const aqd_ref_requant* rq,
                           int32_t level, int32_t out_bits, aqd_ref_tensor* y);

int aqd_ref_residual_add_int(const aqd_ref_tensor* a, const aqd_ref_tensor* b,
                             const int32_t* c, const int8_t* d, int32_t upsample,
                             int32_t scale_a, const aqd_ref_requant* rq, int32_t level,
                             int32_t out_bits, aqd_ref_tensor* y);

int aqd_ref_maxpool_codes(const aqd_ref_tensor* x, int32_t k, int32_t stride, int32_t pad,
                          aqd_ref_tensor* y);

#ifdef __cplusplus
}
#endif
#endif
