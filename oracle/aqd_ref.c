/*
 * aqd_ref.c -- CPU oracle for AQD's integer-only quantized convolution
 * (Chen et al., "AQD: Towards Accurate Quantized Object Detection", arXiv 2007.06919).
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE. Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py load this library. It shares no code, header, helper or
 * table with the CUDA path, and it never calls it.
 *
 * What it computes, step by step, in the paper's order (Fig. 1: conv -> BN -> skip ->
 * ReLU/quantize), all in exact int64 arithmetic:
 *   1. Eq. 4 (Sec. 3.2.1): eta_conv[m, n] = sum_{r,s,c} eta_x[...] * w_int[n, r, s, c]
 *      as a direct convolution; a tap outside the image reads code 0 (the zero point of
 *      Eq. 2 is 0, so zero padding of real values is code 0).
 *      w_int is the signed weight integer: a k-bit two's-complement code, or, for the
 *      Eq. 3 format, 2*eta_w - (2^k - 1) (the odd grid of Eq. 4's second line).
 *   2. Eq. 6 (Sec. 3.2.2): eta_z = eta_conv + round(s); round(s) is the int32 `bias`,
 *      per channel, and per FPN level for the shared head (multi-level BN, Fig. 3).
 *   3. Eq. 7 (Sec. 3.2.3): the skip add with Eq. 8's F = c / 2^d applied to the coarser
 *      operand: t + rhu(eta_s * c, d) (skip is coarser), or rhu(sat32(t) * c, d) + eta_s
 *      (main branch is coarser).
 *   4. Eq. 2 (Sec. 3.1.2) applied to the BN output: the fixed-point rescale by
 *      M0 * 2^-(31+shift) (Eq. 8's dyadic form), rounded to nearest, then clipped to
 *      [0, 2^k - 1]; the clip at 0 is the ReLU. int32 outputs stop after sat32.
 *   rhu(v, R) = floor((v + 2^(R-1)) / 2^R) for R >= 1, v for R = 0 (round half up;
 *   the paper's "nearest integer" has no tie rule, and for values clipped at 0
 *   half-up equals half-away-from-zero).
 *   Sec. 3.2.4: max-pooling acts on codes directly (scale unchanged).
 */
#include "aqd_ref.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#define I64(x) ((int64_t)(x))

/* ---------------------------------------------------------------- integer helpers */

/* floor(a / 2^r) for r in [0, 62], written as a plain floor division */
static int64_t floor_div_pow2(int64_t a, int r) {
  int64_t d = I64(1) << r;
  int64_t q = a / d; /* C truncates toward zero */
  if ((a % d) != 0 && a < 0) q -= 1;
  return q;
}

/* round half up of v / 2^r */
static int64_t rhu(int64_t v, int r) {
  if (r == 0) return v;
  return floor_div_pow2(v + (I64(1) << (r - 1)), r);
}

static int64_t sat32(int64_t v) {
  if (v > I64(2147483647)) return I64(2147483647);
  if (v < -I64(2147483648)) return -I64(2147483648);
  return v;
}

static int64_t clamp64(int64_t v, int64_t lo, int64_t hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

/* ---------------------------------------------------------------- packed layout */

static int valid_code_bits(int bits) { return bits == 2 || bits == 3 || bits == 4 || bits == 8; }

int64_t aqd_ref_row_bytes(int32_t c, int32_t bits) {
  if (c <= 0) return -1;
  if (bits == 32) return I64(4) * c;
  if (bits == 8) return c;
  if (bits == 2 || bits == 3 || bits == 4) {
    if (c % 32 != 0) return -1;
    return I64(c / 32) * (bits * 4); /* 32 codes take 4*bits bytes */
  }
  return -1;
}

/* bit offset, within the row, of code ch's lowest bit for bits 2/4/8 */
static int64_t pos_plain(int64_t ch, int bits) {
  int64_t q = 32 / bits;
  int64_t word = ch / q;
  int64_t i = ch % q;
  return word * 32 + 8 * (i % 4) + bits * (i / 4);
}

static uint32_t get_bits(const uint8_t* row, int64_t bitpos, int nbits) {
  uint32_t v = 0;
  for (int b = 0; b < nbits; ++b) {
    int64_t p = bitpos + b;
    v |= (uint32_t)((row[p >> 3] >> (p & 7)) & 1u) << b;
  }
  return v;
}

static void put_bits(uint8_t* row, int64_t bitpos, int nbits, uint32_t v) {
  for (int b = 0; b < nbits; ++b) {
    int64_t p = bitpos + b;
    uint8_t m = (uint8_t)(1u << (p & 7));
    if ((v >> b) & 1u) row[p >> 3] |= m; else row[p >> 3] &= (uint8_t)~m;
  }
}

/* raw k-bit field of channel ch in a packed row */
static uint32_t read_code(const uint8_t* row, int64_t ch, int bits) {
  if (bits == 3) {
    int64_t g = ch / 32, i = ch % 32;
    const uint8_t* grp = row + g * 12;
    uint32_t lo = get_bits(grp, pos_plain(i, 2), 2);
    uint32_t hi = get_bits(grp + 8, 8 * (i % 4) + (i / 4), 1);
    return lo | (hi << 2);
  }
  return get_bits(row, pos_plain(ch, bits), bits);
}

static void write_code(uint8_t* row, int64_t ch, int bits, uint32_t v) {
  if (bits == 3) {
    int64_t g = ch / 32, i = ch % 32;
    uint8_t* grp = row + g * 12;
    put_bits(grp, pos_plain(i, 2), 2, v & 3u);
    put_bits(grp + 8, 8 * (i % 4) + (i / 4), 1, (v >> 2) & 1u);
    return;
  }
  put_bits(row, pos_plain(ch, bits), bits, v);
}

int aqd_ref_pack(const int32_t* codes, int64_t rows, int32_t c, int32_t bits, uint8_t* out) {
  int64_t rb = aqd_ref_row_bytes(c, bits);
  if (rb < 0 || rows < 0 || (!codes && rows) || (!out && rows)) return AQD_REF_ERR_INVALID;
  if (bits == 32) {
    memcpy(out, codes, (size_t)(rows * rb));
    return AQD_REF_OK;
  }
  uint32_t mask = (1u << bits) - 1u;
  for (int64_t r = 0; r < rows; ++r) {
    uint8_t* row = out + r * rb;
    memset(row, 0, (size_t)rb);
    for (int64_t ch = 0; ch < c; ++ch) write_code(row, ch, bits, (uint32_t)codes[r * c + ch] & mask);
  }
  return AQD_REF_OK;
}

int aqd_ref_unpack(const uint8_t* packed, int64_t rows, int32_t c, int32_t bits,
                   int32_t is_signed, int32_t* out) {
  int64_t rb = aqd_ref_row_bytes(c, bits);
  if (rb < 0 || rows < 0 || (!packed && rows) || (!out && rows)) return AQD_REF_ERR_INVALID;
  if (bits == 32) {
    memcpy(out, packed, (size_t)(rows * rb));
    return AQD_REF_OK;
  }
  for (int64_t r = 0; r < rows; ++r) {
    const uint8_t* row = packed + r * rb;
    for (int64_t ch = 0; ch < c; ++ch) {
      int64_t v = read_code(row, ch, bits);
      if (is_signed && (v >> (bits - 1)) & 1) v -= (I64(1) << bits); /* two's complement */
      out[r * c + ch] = (int32_t)v;
    }
  }
  return AQD_REF_OK;
}

/* ---------------------------------------------------------------- Eq. 8: F(m, n) */

/*
 * Eq. 8 approximates a real ratio by c / 2^d. With c held in a signed 32-bit integer
 * (|c| < 2^31) and d = 31 + shift in [0, 62], the error |real - c/2^d| is at most
 * 2^-(d+1) when c = round(real * 2^d), so the argmin is the largest d whose rounded c
 * still fits; this returns that (c, d) as (m0, shift = d - 31).
 */
int aqd_ref_quantize_multiplier(double real, int32_t* m0, int8_t* shift) {
  if (!m0 || !shift || !isfinite(real)) return AQD_REF_ERR_INVALID;
  if (real == 0.0) { *m0 = 0; *shift = 0; return AQD_REF_OK; }
  double a = fabs(real);
  for (int d = 62; d >= 0; --d) {
    double scaled = ldexp(a, d);          /* exact: scaling by a power of two */
    double c = floor(scaled + 0.5);       /* round half up (scaled > 0) */
    if (c < 2147483648.0) {
      *m0 = (int32_t)(real < 0 ? -c : c);
      *shift = (int8_t)(d - 31);
      return AQD_REF_OK;
    }
  }
  return AQD_REF_ERR_INVALID; /* |real| >= 2^31 - 0.5: no representable c */
}

/* ---------------------------------------------------------------- epilogue */

typedef struct {
  int has_rq;
  int64_t bias, m0;
  int r;
  int has_skip, scale_main;
  int64_t c;
  int d;
} chan_params;

static int check_rq(const aqd_ref_requant* rq, int32_t level, int32_t cout, int out_bits) {
  if (!rq) return out_bits == 32 ? AQD_REF_OK : AQD_REF_ERR_INVALID;
  if (rq->levels <= 0 || level < 0 || level >= rq->levels) return AQD_REF_ERR_INVALID;
  if (out_bits != 32) {
    if (!rq->m0 || !rq->shift) return AQD_REF_ERR_INVALID;
    for (int64_t n = 0; n < cout; ++n) {
      int s = rq->shift[I64(level) * cout + n];
      if (s < -31 || s > 31) return AQD_REF_ERR_INVALID;
    }
  }
  return AQD_REF_OK;
}

static chan_params channel(const aqd_ref_requant* rq, const int32_t* c, const int8_t* d,
                           int has_skip, int scale_main, int32_t level, int32_t cout,
                           int64_t n, int out_bits) {
  chan_params p;
  int64_t idx = I64(level) * cout + n;
  p.has_rq = rq != 0;
  p.bias = (rq && rq->bias) ? rq->bias[idx] : 0;
  p.m0 = (rq && out_bits != 32) ? rq->m0[idx] : 0;
  p.r = (rq && out_bits != 32) ? 31 + rq->shift[idx] : 0;
  p.has_skip = has_skip;
  p.scale_main = scale_main;
  p.c = has_skip ? c[idx] : 0;
  p.d = has_skip ? d[idx] : 0;
  return p;
}

/* Eq. 6 -> Eq. 7 -> Eq. 2 on one accumulator value */
static int64_t epilogue(int64_t acc, int64_t skip_val, const chan_params* p, int out_bits) {
  int64_t t = acc + p->bias; /* Eq. 6: eta_conv + round(s) */
  int64_t t2 = t;
  if (p->has_skip) {         /* Eq. 7 with F = c / 2^d (Eq. 8) */
    if (p->scale_main == 0) t2 = t + rhu(skip_val * p->c, p->d);
    else t2 = rhu(sat32(t) * p->c, p->d) + skip_val;
  }
  int64_t u = sat32(t2);
  if (out_bits == 32) return u;
  int64_t v = rhu(u * p->m0, p->r); /* fixed-point rescale M0 * 2^-R */
  return clamp64(v, 0, (I64(1) << out_bits) - 1); /* Eq. 2 clip: ReLU + k-bit range */
}

/* ---------------------------------------------------------------- conv (Eq. 4) */

typedef struct {
  int32_t n, h, w, cin, kh, kw, stride, pad, cout, ho, wo;
  const int32_t* xu;  /* unpacked input  [n][h][w][cin] */
  const int32_t* wv;  /* signed weights  [cout][kh][kw][cin] */
} conv_geom;

static int64_t conv_acc(const conv_geom* g, int64_t img, int64_t ho, int64_t wo, int64_t co) {
  int64_t acc = 0;
  for (int64_t r = 0; r < g->kh; ++r) {
    int64_t hi = ho * g->stride - g->pad + r;
    if (hi < 0 || hi >= g->h) continue; /* zero padding: code 0 */
    for (int64_t s = 0; s < g->kw; ++s) {
      int64_t wi = wo * g->stride - g->pad + s;
      if (wi < 0 || wi >= g->w) continue;
      const int32_t* xp = g->xu + ((img * g->h + hi) * g->w + wi) * g->cin;
      const int32_t* wp = g->wv + ((co * g->kh + r) * g->kw + s) * g->cin;
      for (int64_t ci = 0; ci < g->cin; ++ci) acc += I64(xp[ci]) * I64(wp[ci]);
    }
  }
  return acc;
}

static int skip_value(const aqd_ref_tensor* sk, const int32_t* su, int32_t up, int64_t img,
                      int64_t ho, int64_t wo, int64_t ch, int64_t* out) {
  int64_t sh = ho / up, sw = wo / up;
  if (sh >= sk->h || sw >= sk->w) return 0;
  *out = su[((img * sk->h + sh) * sk->w + sw) * sk->c + ch];
  return 1;
}

static int32_t* unpack_tensor(const aqd_ref_tensor* t, int is_signed) {
  int64_t rows = I64(t->n) * t->h * t->w;
  int32_t* u = (int32_t*)malloc((size_t)(rows * t->c) * sizeof(int32_t) + 4);
  if (!u) return 0;
  if (aqd_ref_unpack((const uint8_t*)t->data, rows, t->c, t->bits, is_signed, u) != AQD_REF_OK) {
    free(u);
    return 0;
  }
  return u;
}

static int check_tensor(const aqd_ref_tensor* t) {
  if (!t || !t->data) return 0;
  if (t->n <= 0 || t->h <= 0 || t->w <= 0 || t->c <= 0) return 0;
  return aqd_ref_row_bytes(t->c, t->bits) > 0;
}

/* shared by the full and the sampled conv; writes out[npix][cout] unpacked */
static int conv_core(const aqd_ref_tensor* x, const uint8_t* w_packed, int32_t w_bits,
                     int32_t w_format, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                     int32_t cout, int32_t level, const aqd_ref_requant* rq,
                     const aqd_ref_residual* res, int32_t out_bits, int32_t ho_n, int32_t wo_n,
                     const int64_t* pix, int64_t npix, int32_t* out) {
  if (!check_tensor(x) || !valid_code_bits(x->bits) || !w_packed) return AQD_REF_ERR_INVALID;
  if (!valid_code_bits(w_bits) || (w_format != AQD_REF_W_TWOS && w_format != AQD_REF_W_ODD))
    return AQD_REF_ERR_INVALID;
  if (kh <= 0 || kw <= 0 || stride <= 0 || pad < 0 || cout <= 0) return AQD_REF_ERR_INVALID;
  if (!(valid_code_bits(out_bits) || out_bits == 32)) return AQD_REF_ERR_INVALID;
  if (check_rq(rq, level, cout, out_bits) != AQD_REF_OK) return AQD_REF_ERR_INVALID;
  int32_t ho_expect = (x->h + 2 * pad - kh) / stride + 1;
  int32_t wo_expect = (x->w + 2 * pad - kw) / stride + 1;
  if (ho_expect <= 0 || wo_expect <= 0 || ho_n != ho_expect || wo_n != wo_expect)
    return AQD_REF_ERR_INVALID;
  if (aqd_ref_row_bytes(x->c, w_bits) < 0) return AQD_REF_ERR_INVALID;
  int has_skip = res && res->skip;
  if (has_skip) {
    const aqd_ref_tensor* sk = res->skip;
    int32_t up = res->upsample;
    if (!check_tensor(sk) || !res->c || !res->d || (up != 1 && up != 2)) return AQD_REF_ERR_INVALID;
    if (sk->n != x->n || sk->c != cout) return AQD_REF_ERR_INVALID;
    if ((ho_n + up - 1) / up > sk->h || (wo_n + up - 1) / up > sk->w) return AQD_REF_ERR_INVALID;
    if (rq == 0 || level >= rq->levels) return AQD_REF_ERR_INVALID;
    for (int64_t n = 0; n < cout; ++n) {
      int dd = res->d[I64(level) * cout + n];
      if (dd < 0 || dd > 62) return AQD_REF_ERR_INVALID;
    }
  }

  int32_t* xu = unpack_tensor(x, 0);
  if (!xu) return AQD_REF_ERR_INVALID;
  int64_t kelems = I64(kh) * kw * x->c;
  int32_t* wv = (int32_t*)malloc((size_t)(cout * kelems) * sizeof(int32_t));
  int32_t* su = has_skip ? unpack_tensor(res->skip, res->skip->bits == 32) : 0;
  if (!wv || (has_skip && !su)) { free(xu); free(wv); free(su); return AQD_REF_ERR_INVALID; }
  /* weights: rows of [kh][kw][cin] per output channel, packed along cin */
  aqd_ref_unpack(w_packed, I64(cout) * kh * kw, x->c, w_bits, w_format == AQD_REF_W_TWOS, wv);
  if (w_format == AQD_REF_W_ODD) /* Eq. 3/4: eta_w -> 2*eta_w - (2^k - 1) */
    for (int64_t i = 0; i < cout * kelems; ++i) wv[i] = 2 * wv[i] - ((1 << w_bits) - 1);

  conv_geom g = {x->n, x->h, x->w, x->c, kh, kw, stride, pad, cout, ho_n, wo_n, xu, wv};
  int32_t up = has_skip ? res->upsample : 1;
  int scale_main = has_skip ? res->scale_main : 0;
  const int32_t* sc = has_skip ? res->c : 0;
  const int8_t* sd = has_skip ? res->d : 0;
  int bad = 0;

#pragma omp parallel for schedule(dynamic, 16)
  for (int64_t i = 0; i < npix; ++i) {
    int64_t p = pix ? pix[i] : i;
    int64_t img = p / (I64(ho_n) * wo_n);
    int64_t rem = p % (I64(ho_n) * wo_n);
    int64_t ho = rem / wo_n, wo = rem % wo_n;
    if (p < 0 || img >= x->n) { bad = 1; continue; }
    for (int64_t co = 0; co < cout; ++co) {
      chan_params cp = channel(rq, sc, sd, has_skip, scale_main, level, cout, co, out_bits);
      int64_t acc = conv_acc(&g, img, ho, wo, co);
      int64_t sv = 0;
      if (has_skip && !skip_value(res->skip, su, up, img, ho, wo, co, &sv)) bad = 1;
      out[i * cout + co] = (int32_t)epilogue(acc, sv, &cp, out_bits);
    }
  }
  free(xu); free(wv); free(su);
  return bad ? AQD_REF_ERR_INVALID : AQD_REF_OK;
}

int aqd_ref_conv_int(const aqd_ref_tensor* x, const uint8_t* w_packed, int32_t w_bits,
                     int32_t w_format, int32_t kh, int32_t kw, int32_t stride, int32_t pad,
                     int32_t cout, int32_t level, const aqd_ref_requant* rq,
                     const aqd_ref_residual* res, int32_t out_bits, aqd_ref_tensor* y) {
  if (!check_tensor(x) || !y || !y->data) return AQD_REF_ERR_INVALID;
  if (y->n != x->n || y->c != cout || y->bits != out_bits) return AQD_REF_ERR_INVALID;
  int64_t npix = I64(y->n) * y->h * y->w;
  int32_t* tmp = (int32_t*)malloc((size_t)(npix * cout) * sizeof(int32_t) + 4);
  if (!tmp) return AQD_REF_ERR_INVALID;
  int st = conv_core(x, w_packed, w_bits, w_format, kh, kw, stride, pad, cout, level, rq, res,
                     out_bits, y->h, y->w, 0, npix, tmp);
  if (st == AQD_REF_OK) st = aqd_ref_pack(tmp, npix, cout, out_bits, (uint8_t*)y->data);
  free(tmp);
  return st;
}

int aqd_ref_conv_int_pixels(const aqd_ref_tensor* x, const uint8_t* w_packed,
                            int32_t w_bits, int32_t w_format, int32_t kh, int32_t kw,
                            int32_t stride, int32_t pad, int32_t cout, int32_t level,
                            const aqd_ref_requant* rq, const aqd_ref_residual* res,
                            int32_t out_bits, int32_t out_h, int32_t out_w,
                            const int64_t* pix, int64_t npix, int32_t* out) {
  if (!pix || !out || npix < 0) return AQD_REF_ERR_INVALID;
  return conv_core(x, w_packed, w_bits, w_format, kh, kw, stride, pad, cout, level, rq, res,
                   out_bits, out_h, out_w, pix, npix, out);
}

/* ---------------------------------------------------------------- elementwise ops */

int aqd_ref_requant_tensor(const aqd_ref_tensor* acc, const aqd_ref_requant* rq,
                           int32_t level, int32_t out_bits, aqd_ref_tensor* y) {
  if (!check_tensor(acc) || acc->bits != 32 || !y || !y->data) return AQD_REF_ERR_INVALID;
  if (y->n != acc->n || y->h != acc->h || y->w != acc->w || y->c != acc->c || y->bits != out_bits)
    return AQD_REF_ERR_INVALID;
  if (!(valid_code_bits(out_bits) || out_bits == 32) || !rq) return AQD_REF_ERR_INVALID;
  if (check_rq(rq, level, acc->c, out_bits) != AQD_REF_OK) return AQD_REF_ERR_INVALID;
  int64_t rows = I64(acc->n) * acc->h * acc->w;
  const int32_t* a = (const int32_t*)acc->data;
  int32_t* tmp = (int32_t*)malloc((size_t)(rows * acc->c) * sizeof(int32_t) + 4);
  if (!tmp) return AQD_REF_ERR_INVALID;
  for (int64_t i = 0; i < rows; ++i)
    for (int64_t ch = 0; ch < acc->c; ++ch) {
      chan_params cp = channel(rq, 0, 0, 0, 0, level, acc->c, ch, out_bits);
      tmp[i * acc->c + ch] = (int32_t)epilogue(a[i * acc->c + ch], 0, &cp, out_bits);
    }
  int st = aqd_ref_pack(tmp, rows, acc->c, out_bits, (uint8_t*)y->data);
  free(tmp);
  return st;
}

int aqd_ref_residual_add_int(const aqd_ref_tensor* a, const aqd_ref_tensor* b,
                             const int32_t* c, const int8_t* d, int32_t upsample,
                             int32_t scale_a, const aqd_ref_requant* rq, int32_t level,
                             int32_t out_bits, aqd_ref_tensor* y) {
  if (!check_tensor(a) || !check_tensor(b) || !c || !d || !y || !y->data) return AQD_REF_ERR_INVALID;
  if (upsample != 1 && upsample != 2) return AQD_REF_ERR_INVALID;
  if (b->n != a->n || b->c != a->c) return AQD_REF_ERR_INVALID;
  if ((a->h + upsample - 1) / upsample > b->h || (a->w + upsample - 1) / upsample > b->w)
    return AQD_REF_ERR_INVALID;
  if (y->n != a->n || y->h != a->h || y->w != a->w || y->c != a->c || y->bits != out_bits)
    return AQD_REF_ERR_INVALID;
  if (!(valid_code_bits(out_bits) || out_bits == 32)) return AQD_REF_ERR_INVALID;
  if (check_rq(rq, level, a->c, out_bits) != AQD_REF_OK) return AQD_REF_ERR_INVALID;
  int32_t lv = rq ? level : 0;
  if (level < 0 || (!rq && level != 0)) return AQD_REF_ERR_INVALID;
  for (int64_t n = 0; n < a->c; ++n)
    if (d[I64(lv) * a->c + n] < 0 || d[I64(lv) * a->c + n] > 62) return AQD_REF_ERR_INVALID;
  int32_t* au = unpack_tensor(a, a->bits == 32);
  int32_t* bu = unpack_tensor(b, b->bits == 32);
  int64_t rows = I64(a->n) * a->h * a->w;
  int32_t* tmp = (int32_t*)malloc((size_t)(rows * a->c) * sizeof(int32_t) + 4);
  if (!au || !bu || !tmp) { free(au); free(bu); free(tmp); return AQD_REF_ERR_INVALID; }
  for (int64_t p = 0; p < rows; ++p) {
    int64_t img = p / (I64(a->h) * a->w), rem = p % (I64(a->h) * a->w);
    int64_t hh = rem / a->w, ww = rem % a->w;
    for (int64_t ch = 0; ch < a->c; ++ch) {
      chan_params cp = channel(rq, c, d, 1, scale_a, lv, a->c, ch, out_bits);
      int64_t sv = 0;
      skip_value(b, bu, upsample, img, hh, ww, ch, &sv);
      tmp[p * a->c + ch] = (int32_t)epilogue(au[p * a->c + ch], sv, &cp, out_bits);
    }
  }
  int st = aqd_ref_pack(tmp, rows, a->c, out_bits, (uint8_t*)y->data);
  free(au); free(bu); free(tmp);
  return st;
}

/* Sec. 3.2.4: max-pooling needs no rescale; it acts on the codes (all >= 0) */
int aqd_ref_maxpool_codes(const aqd_ref_tensor* x, int32_t k, int32_t stride, int32_t pad,
                          aqd_ref_tensor* y) {
  if (!check_tensor(x) || !valid_code_bits(x->bits) || !y || !y->data) return AQD_REF_ERR_INVALID;
  if (k <= 0 || stride <= 0 || pad < 0 || pad >= k) return AQD_REF_ERR_INVALID;
  int32_t ho = (x->h + 2 * pad - k) / stride + 1, wo = (x->w + 2 * pad - k) / stride + 1;
  if (y->n != x->n || y->h != ho || y->w != wo || y->c != x->c || y->bits != x->bits)
    return AQD_REF_ERR_INVALID;
  int32_t* xu = unpack_tensor(x, 0);
  int64_t rows = I64(y->n) * ho * wo;
  int32_t* tmp = (int32_t*)malloc((size_t)(rows * x->c) * sizeof(int32_t) + 4);
  if (!xu || !tmp) { free(xu); free(tmp); return AQD_REF_ERR_INVALID; }
  for (int64_t p = 0; p < rows; ++p) {
    int64_t img = p / (I64(ho) * wo), rem = p % (I64(ho) * wo);
    int64_t oh = rem / wo, ow = rem % wo;
    for (int64_t ch = 0; ch < x->c; ++ch) {
      int64_t best = -1;
      for (int64_t r = 0; r < k; ++r)
        for (int64_t s = 0; s < k; ++s) {
          int64_t hi = oh * stride - pad + r, wi = ow * stride - pad + s;
          if (hi < 0 || hi >= x->h || wi < 0 || wi >= x->w) continue;
          int64_t v = xu[((img * x->h + hi) * x->w + wi) * x->c + ch];
          if (v > best) best = v;
        }
      tmp[p * x->c + ch] = (int32_t)(best < 0 ? 0 : best);
    }
  }
  int st = aqd_ref_pack(tmp, rows, x->c, x->bits, (uint8_t*)y->data);
  free(xu); free(tmp);
  return st;
}
