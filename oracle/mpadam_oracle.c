/*
 * mpadam_oracle.c -- plain, slow, single-threaded CPU oracle of the M+Adam
 * optimizer step (arxiv 2607.10611).
 *
 * TEST INFRASTRUCTURE ONLY: it exists to check the CUDA library, and only the
 * tests, the smoke check and the benchmark's CPU-baseline leg may call it.
 * It shares no code with the CUDA path.
 *
 * What it follows:
 *   - Algorithm 1 (Sec. 4.1, "M+Adam: additive-multiplicative update"):
 *     Adam moments with bias correction, the exponent gradient
 *     g_e = (ln 2) w g, its second moment, the proposal
 *     u~ = -eta_m g_e / (sqrt(v_e-hat) + eps), rho = max(|w|, tau),
 *     u_m = u~ / rho and the combination w + w u_m + u_a.
 *   - Sec. 4.1: u_m = clip(u~ / rho).
 *   - Algorithm 2 (Appendix A): the optional clamp of the normalised exponent
 *     gradient at g_max, the relative bounds [-(0.75 - eps0), 0.75], the
 *     optional cap |log2(1 + u_m)| <= d_mult,max, the optional weight clip
 *     w_max and the optional additive (decoupled) weight decay; bias
 *     correction switched off reproduces Algorithm 2's raw moments.
 *   - Eq. for AdamW in Sec. 3: the decoupled decay term eta * lambda * w.
 *   - Appendix B, "bf16 round trip": each step is computed in FP32 and the
 *     parameter is rounded into its storage format right away.
 *
 * Readings where the paper leaves the arithmetic open (each also listed in
 * the design notes of the repository):
 *   - bias correction is folded into two per-step scalars: eta_a u-hat =
 *     eta_a mu / (1 - beta1^t) and sqrt(v-hat) = sqrt(v) / sqrt(1 - beta2^t);
 *   - the log2 / exp2 round trip of the step cap is the equivalent clamp of
 *     u_m to [2^-d - 1, 2^d - 1] (log2(1+u) is increasing), merged with the
 *     0.75 bounds; bounds are rounded towards zero into binary32;
 *   - clamp_a(x) = max(-a, min(x, a)) uses IEEE minNum/maxNum (C fminf and
 *     fmaxf); optional clips are skipped entirely when switched off;
 *   - fused multiply-adds: mu, nu and nu_e updates, the two denominators and
 *     w + w u_m are each one fmaf();
 *   - stochastic rounding keys a Philox4x32-10 stream by (seed, step, global
 *     element index); the global index of a tensor's first element is the
 *     previous tensor's end rounded up to a multiple of 8;
 *   - FP8 storage is OCP E4M3 (bias 7, max 448, no infinities, NaN 0x7F)
 *     with a per-tensor power-of-two scale chosen from the previous step's
 *     largest |w| (delayed scaling), saturating encode;
 *   - NaN stores as 0x7FFF in BF16 and 0x7F in E4M3.
 */
#include "mpadam_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

static float f_from_bits(uint32_t b) { float f; memcpy(&f, &b, sizeof f); return f; }
static uint32_t bits_from_f(float f) { uint32_t b; memcpy(&b, &f, sizeof b); return b; }

/* 2^k as binary32 for -126 <= k <= 127 (exact). */
static float pow2_int(int32_t k) { return f_from_bits((uint32_t)(k + 127) << 23); }

/* ------------------------------------------------------------------------ */
/* Philox4x32-10: J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw,        */
/* "Parallel random numbers: as easy as 1, 2, 3", SC'11.  Ten rounds of the  */
/* four-word Philox S-box; each round multiplies words 0 and 2 by the two    */
/* round multipliers, swaps the products' halves across the block and mixes  */
/* the high halves with words 1 and 3 and the round key.  The key advances   */
/* by the two Weyl constants after every round.                              */
/* ------------------------------------------------------------------------ */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  const uint32_t mult0 = 0xD2511F53u, mult1 = 0xCD9E8D57u;
  const uint32_t weyl0 = 0x9E3779B9u, weyl1 = 0xBB67AE85u;
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    uint64_t prod0 = (uint64_t)mult0 * (uint64_t)x0;
    uint64_t prod1 = (uint64_t)mult1 * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    k0 += weyl0;
    k1 += weyl1;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

uint32_t orc_rng_lane(uint64_t seed, uint64_t t, uint64_t i, int32_t storage) {
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  if (storage == ORC_BF16) {
    /* 8 lanes of 16 bits per block: lane L is half (L mod 2) of word L/2. */
    uint64_t block = i / 8;
    uint32_t lane = (uint32_t)(i % 8);
    uint32_t ctr[4] = {(uint32_t)block, (uint32_t)(block >> 32), (uint32_t)t, (uint32_t)(t >> 32)};
    orc_philox4x32_10(ctr, key, out);
    uint32_t word = out[lane / 2];
    return (lane % 2 == 0) ? (word & 0xFFFFu) : (word >> 16);
  }
  /* 4 lanes of 32 bits per block. */
  uint64_t block = i / 4;
  uint32_t lane = (uint32_t)(i % 4);
  uint32_t ctr[4] = {(uint32_t)block, (uint32_t)(block >> 32), (uint32_t)t, (uint32_t)(t >> 32)};
  orc_philox4x32_10(ctr, key, out);
  return out[lane];
}

/* ------------------------------------------------------------------------ */
/* BF16: the upper 16 bits of a binary32.                                    */
/* ------------------------------------------------------------------------ */
float orc_bf16_decode(uint16_t h) { return f_from_bits((uint32_t)h << 16); }

uint16_t orc_bf16_rne(float x) {
  if (isnan(x)) return 0x7FFFu;
  uint32_t b = bits_from_f(x);
  uint32_t upper = b >> 16;
  uint32_t lower = b & 0xFFFFu;
  /* nearest; ties to the even upper half.  A carry out of the mantissa moves
   * to the next binade, and past the largest finite value to infinity. */
  if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u))) upper += 1;
  return (uint16_t)upper;
}

uint16_t orc_bf16_sr(float x, uint32_t r16) {
  if (isnan(x)) return 0x7FFFu;
  uint32_t b = bits_from_f(x);
  uint32_t upper = b >> 16;           /* the neighbour towards zero */
  uint32_t lower = b & 0xFFFFu;       /* distance to it, in 2^-16 of a bf16 ulp */
  /* away from zero with probability lower / 2^16: exactly unbiased. */
  if ((r16 & 0xFFFFu) < lower) upper += 1;
  return (uint16_t)upper;
}

/* ------------------------------------------------------------------------ */
/* E4M3 (OCP FP8, "fn" variant): 1 sign, 4 exponent (bias 7), 3 mantissa     */
/* bits; largest finite 448 (0x7E); 0x7F / 0xFF are NaN; subnormal step 2^-9 */
/* ------------------------------------------------------------------------ */
float orc_e4m3_decode(uint8_t q) {
  uint32_t mag = q & 0x7Fu;
  if (mag == 0x7Fu) return NAN;
  uint32_t e = mag >> 3, f = mag & 7u;
  double val = (e == 0) ? ldexp((double)f, -9) : ldexp((double)(8u + f), (int)e - 10);
  return (float)((q & 0x80u) ? -val : val);
}

/* |x| (finite, below 448) = (code + rem / 2^shift) * ulp, ulp the E4M3
 * spacing at |x|, code the E4M3 magnitude code truncated towards zero. */
static void e4m3_split(uint32_t abits, uint32_t* code, uint64_t* rem, int32_t* shift) {
  uint32_t ef = abits >> 23, mant = abits & 0x7FFFFFu;
  uint64_t sig; int32_t e;
  if (ef == 0) { sig = mant; e = -126; }       /* binary32 subnormal */
  else { sig = mant | 0x800000u; e = (int32_t)ef - 127; }
  /* |x| = sig * 2^(e - 23) */
  if (e >= -6) {                               /* E4M3 normal: ulp = 2^(e-3) */
    *shift = 20;
    *code = (uint32_t)(((e + 7) << 3) + (int32_t)(sig >> 20) - 8);
    *rem = sig & 0xFFFFFu;
  } else {                                     /* E4M3 subnormal: ulp = 2^-9 */
    *shift = 14 - e;                           /* |x| / 2^-9 = sig * 2^(e - 14) */
    if (*shift >= 64) { *code = 0; *rem = sig; }
    else { *code = (uint32_t)(sig >> *shift); *rem = sig & ((1ull << *shift) - 1ull); }
  }
}

uint8_t orc_e4m3_rne(float x) {
  if (isnan(x)) return 0x7Fu;
  uint32_t b = bits_from_f(x);
  uint32_t sign = (b >> 24) & 0x80u;
  uint32_t abits = b & 0x7FFFFFFFu;
  if (abits >= bits_from_f(448.0f)) return (uint8_t)(sign | 0x7Eu);   /* saturate */
  uint32_t code; uint64_t rem; int32_t shift;
  e4m3_split(abits, &code, &rem, &shift);
  if (shift <= 40) {  /* for larger shifts rem < 2^24 is far below one half */
    uint64_t half = 1ull << (shift - 1);
    if (rem > half || (rem == half && (code & 1u))) code += 1;
  }
  if (code > 0x7Eu) code = 0x7Eu;
  return (uint8_t)(sign | code);
}

uint8_t orc_e4m3_sr(float x, uint32_t r32) {
  if (isnan(x)) return 0x7Fu;
  uint32_t b = bits_from_f(x);
  uint32_t sign = (b >> 24) & 0x80u;
  uint32_t abits = b & 0x7FFFFFFFu;
  if (abits >= bits_from_f(448.0f)) return (uint8_t)(sign | 0x7Eu);
  uint32_t code; uint64_t rem; int32_t shift;
  e4m3_split(abits, &code, &rem, &shift);
  /* threshold = floor(fraction * 2^32); away from zero iff r < threshold */
  uint64_t thr;
  if (shift <= 32) thr = rem << (32 - shift);
  else if (shift - 32 >= 64) thr = 0;
  else thr = rem >> (shift - 32);
  if ((uint64_t)r32 < thr) code += 1;
  if (code > 0x7Eu) code = 0x7Eu;
  return (uint8_t)(sign | code);
}

int32_t orc_fp8_next_exponent(float amax, int32_t e_cur) {
  if (!(amax > 0.0f) || isinf(amax)) return e_cur;   /* nothing to fit: keep */
  int x;
  float f = frexpf(amax, &x);                        /* amax = f 2^x, f in [0.5, 1) */
  /* smallest k with amax <= 448 2^k = 0.875 2^(9+k) */
  int32_t k = (f <= 0.875f) ? x - 9 : x - 8;
  if (k < -100) k = -100;
  if (k > 100) k = 100;
  return k;
}

float orc_e4m3_amax(int64_t n, const uint8_t* q, int32_t e) {
  float amax = 0.0f;
  float scale = pow2_int(e);
  for (int64_t k = 0; k < n; ++k) {
    float val = orc_e4m3_decode(q[k]);
    if (isnan(val)) continue;
    float a = fabsf(val * scale);
    if (a > amax) amax = a;
  }
  return amax;
}

/* ------------------------------------------------------------------------ */
/* Per-step scalars                                                          */
/* ------------------------------------------------------------------------ */
static float to_f32_toward_zero(double x) {
  float f = (float)x;
  if (x > 0.0 && (double)f > x) f = nextafterf(f, 0.0f);
  if (x < 0.0 && (double)f < x) f = nextafterf(f, 0.0f);
  return f;
}

static int finite_pos(float x) { return isfinite(x) && x > 0.0f; }

int32_t orc_scalars_for_step(const orc_hparams* hp, int64_t t, orc_scalars* s) {
  if (t < 1) return -1;
  if (!(isfinite(hp->lr_add) && hp->lr_add >= 0.0f)) return -1;
  if (!(isfinite(hp->lr_mul) && hp->lr_mul >= 0.0f)) return -1;
  if (!(hp->beta1 >= 0.0f && hp->beta1 < 1.0f)) return -1;
  if (!(hp->beta2 >= 0.0f && hp->beta2 < 1.0f)) return -1;
  if (!finite_pos(hp->eps) || !finite_pos(hp->tau)) return -1;
  if (!finite_pos(hp->rmax_pos)) return -1;
  if (!(finite_pos(hp->rmax_neg) && hp->rmax_neg < 1.0f)) return -1;
  if (!(hp->g_max > 0.0f) || !(hp->dmult_max > 0.0f) || !(hp->w_max > 0.0f)) return -1;
  if (!(isfinite(hp->wd_add) && hp->wd_add >= 0.0f)) return -1;

  double b1 = hp->beta1, b2 = hp->beta2;
  double bc1 = 1.0, bc2 = 1.0;
  if (hp->bias_correction) {
    bc1 = 1.0 - pow(b1, (double)t);
    bc2 = 1.0 - pow(b2, (double)t);
  }
  s->b1 = hp->beta1;
  s->b2 = hp->beta2;
  s->omb1 = (float)(1.0 - b1);
  s->omb2 = (float)(1.0 - b2);
  s->ka = (float)(-(double)hp->lr_add / bc1);
  s->c2 = (float)(1.0 / sqrt(bc2));
  s->km = -hp->lr_mul;
  s->ln2 = (float)0.69314718055994530942;
  s->eps = hp->eps;
  s->tau = hp->tau;
  double d = hp->dmult_max;
  double hi = fmin((double)hp->rmax_pos, exp2(d) - 1.0);
  double lo = fmax(-(double)hp->rmax_neg, exp2(-d) - 1.0);
  s->hi = to_f32_toward_zero(hi);
  s->lo = to_f32_toward_zero(lo);
  s->gmax_on = isfinite(hp->g_max) ? 1 : 0;
  s->gmax = s->gmax_on ? hp->g_max : 0.0f;
  s->wmax_on = isfinite(hp->w_max) ? 1 : 0;
  s->wmax = s->wmax_on ? hp->w_max : 0.0f;
  s->wd_on = hp->wd_add != 0.0f ? 1 : 0;
  s->kwd = (float)((double)hp->lr_add * (double)hp->wd_add);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* The canonical per-element update (Algorithm 1 + Algorithm 2 options)      */
/* ------------------------------------------------------------------------ */
void orc_update_element(const orc_scalars* s, float w, float g, float m, float v, float ve,
                        float* wn_out, float* m_out, float* v_out, float* ve_out) {
  /* additive branch: Adam moments */
  float m1 = fmaf(s->b1, m, s->omb1 * g);                 /* mu <- b1 mu + (1-b1) g */
  float v1 = fmaf(s->b2, v, s->omb2 * (g * g));           /* nu <- b2 nu + (1-b2) g^2 */
  /* u_a = -eta_a mu-hat / (sqrt(nu-hat) + eps) */
  float den_a = fmaf(sqrtf(v1), s->c2, s->eps);
  float ua = (s->ka * m1) / den_a;
  if (s->wd_on) ua = ua - s->kwd * w;                     /* decoupled additive decay */

  /* multiplicative branch */
  float ge = (s->ln2 * w) * g;                            /* g_e = (ln 2) w g */
  float ve1 = fmaf(s->b2, ve, s->omb2 * (ge * ge));       /* nu_e <- b2 nu_e + (1-b2) g_e^2 */
  float den_e = fmaf(sqrtf(ve1), s->c2, s->eps);
  float n = ge / den_e;                                   /* normalised exponent gradient */
  if (s->gmax_on) n = fmaxf(-s->gmax, fminf(n, s->gmax));
  float rho = fmaxf(fabsf(w), s->tau);                    /* rho = max(|w|, tau) */
  float um = (s->km * n) / rho;                           /* u_m = u~ / rho, u~ = -eta_m n */
  um = fmaxf(s->lo, fminf(um, s->hi));                    /* relative bounds and step cap */

  /* combine: w + w u_m + u_a */
  float wn = fmaf(w, um, w) + ua;
  if (s->wmax_on) wn = fmaxf(-s->wmax, fminf(wn, s->wmax));

  *wn_out = wn; *m_out = m1; *v_out = v1; *ve_out = ve1;
}

/* ------------------------------------------------------------------------ */
/* One step over a run of elements                                           */
/* ------------------------------------------------------------------------ */
static float load_elem(const void* p, int64_t k, int32_t dt) {
  if (dt == ORC_F32) return ((const float*)p)[k];
  if (dt == ORC_BF16) return orc_bf16_decode(((const uint16_t*)p)[k]);
  return orc_e4m3_decode(((const uint8_t*)p)[k]);
}

static void store_moment(void* p, int64_t k, int32_t dt, float x) {
  if (dt == ORC_F32) ((float*)p)[k] = x;
  else ((uint16_t*)p)[k] = orc_bf16_rne(x);
}

int32_t orc_step_elements(int64_t n, const int64_t* gidx, int64_t gidx0,
                          int32_t wdt, int32_t gdt, int32_t mdt,
                          void* w, const void* g, void* m, void* v, void* ve,
                          const orc_hparams* hp, int64_t t,
                          int32_t e_cur, int32_t e_next, float* amax) {
  if (wdt != ORC_F32 && wdt != ORC_BF16 && wdt != ORC_E4M3) return -1;
  if (gdt != ORC_F32 && gdt != ORC_BF16) return -1;
  if (mdt != ORC_F32 && mdt != ORC_BF16) return -1;
  if (e_cur < -100 || e_cur > 100 || e_next < -100 || e_next > 100) return -1;
  orc_scalars s;
  if (orc_scalars_for_step(hp, t, &s) != 0) return -1;
  float dec_scale = pow2_int(e_cur);
  float enc_scale = pow2_int(-e_next);

  for (int64_t k = 0; k < n; ++k) {
    uint64_t i = (uint64_t)(gidx ? gidx[k] : gidx0 + k);
    float wk = load_elem(w, k, wdt);
    if (wdt == ORC_E4M3) wk = wk * dec_scale;
    float gk = load_elem(g, k, gdt);
    float mk = load_elem(m, k, mdt);
    float vk = load_elem(v, k, mdt);
    float vek = load_elem(ve, k, mdt);

    float wn, m1, v1, ve1;
    orc_update_element(&s, wk, gk, mk, vk, vek, &wn, &m1, &v1, &ve1);

    if (wdt == ORC_F32) {
      ((float*)w)[k] = wn;
    } else if (wdt == ORC_BF16) {
      uint16_t h = hp->stochastic ? orc_bf16_sr(wn, orc_rng_lane(hp->seed, (uint64_t)t, i, ORC_BF16))
                                  : orc_bf16_rne(wn);
      ((uint16_t*)w)[k] = h;
    } else {
      if (isfinite(wn) && fabsf(wn) > *amax) *amax = fabsf(wn);
      float x = wn * enc_scale;
      uint8_t q = hp->stochastic ? orc_e4m3_sr(x, orc_rng_lane(hp->seed, (uint64_t)t, i, ORC_E4M3))
                                 : orc_e4m3_rne(x);
      ((uint8_t*)w)[k] = q;
    }
    store_moment(m, k, mdt, m1);
    store_moment(v, k, mdt, v1);
    store_moment(ve, k, mdt, ve1);
  }
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Block-scaled E4M3 (reading of Sec. 5.2 and the FP8-master figure: FP8     */
/* weights "quantized in blocks with FP16 scales"; block size and scale rule */
/* are not given).  Blocks are 32 consecutive elements of a tensor; a scale  */
/* is a power of two (a subset of FP16, so scaling is exact), chosen from    */
/* the block's own updated weights at each step.                             */
/* ------------------------------------------------------------------------ */
uint16_t orc_fp16_pow2(int32_t k) {
  if (k < -24) k = -24;
  if (k > 15) k = 15;
  if (k >= -14) return (uint16_t)((k + 15) << 10);      /* normal: exponent field k + 15 */
  return (uint16_t)(1u << (k + 24));                     /* subnormal: 2^-24 units */
}

float orc_fp16_decode(uint16_t h) {
  uint32_t e = (h >> 10) & 0x1Fu, f = h & 0x3FFu;
  double val;
  if (e == 0) val = ldexp((double)f, -24);
  else if (e == 31) val = f ? NAN : INFINITY;
  else val = ldexp((double)(1024u + f), (int)e - 25);
  return (float)((h & 0x8000u) ? -val : val);
}

int32_t orc_block_exponent(float amax, int32_t k_old) {
  if (!(amax > 0.0f) || isinf(amax)) return k_old;
  int x;
  float f = frexpf(amax, &x);                 /* amax = f 2^x, f in [0.5, 1) */
  int32_t k = (f <= 0.875f) ? x - 9 : x - 8;  /* smallest k with amax <= 0.875 2^(9+k) */
  if (k < -24) k = -24;
  if (k > 15) k = 15;
  return k;
}

static int32_t fp16_pow2_exponent(uint16_t h) {
  uint32_t e = (h >> 10) & 0x1Fu;
  if (e != 0) return (int32_t)e - 15;
  int32_t k = -24;
  for (uint32_t f = h & 0x3FFu; f > 1u; f >>= 1) ++k;
  return k;
}

int32_t orc_step_block_e4m3(int64_t n, int64_t gidx0, int32_t gdt, int32_t mdt,
                            uint8_t* q, uint16_t* bscale, const void* g, void* m, void* v, void* ve,
                            const orc_hparams* hp, int64_t t) {
  if (gdt != ORC_F32 && gdt != ORC_BF16) return -1;
  if (mdt != ORC_F32 && mdt != ORC_BF16) return -1;
  orc_scalars s;
  if (orc_scalars_for_step(hp, t, &s) != 0) return -1;
  for (int64_t b0 = 0; b0 < n; b0 += ORC_BLOCK) {
    const int64_t bn = (n - b0 < ORC_BLOCK) ? n - b0 : ORC_BLOCK;
    const int64_t blk = b0 / ORC_BLOCK;
    const float dec = orc_fp16_decode(bscale[blk]);
    float wn[ORC_BLOCK];
    float amax = 0.0f;
    for (int64_t j = 0; j < bn; ++j) {
      const int64_t k = b0 + j;
      float wk = orc_e4m3_decode(q[k]) * dec;
      float gk = load_elem(g, k, gdt), mk = load_elem(m, k, mdt), vk = load_elem(v, k, mdt);
      float vek = load_elem(ve, k, mdt);
      float m1, v1, ve1;
      orc_update_element(&s, wk, gk, mk, vk, vek, &wn[j], &m1, &v1, &ve1);
      if (isfinite(wn[j]) && fabsf(wn[j]) > amax) amax = fabsf(wn[j]);
      store_moment(m, k, mdt, m1);
      store_moment(v, k, mdt, v1);
      store_moment(ve, k, mdt, ve1);
    }
    /* current scaling: the block's new scale fits its largest updated |w| */
    const int32_t k_new = orc_block_exponent(amax, fp16_pow2_exponent(bscale[blk]));
    bscale[blk] = orc_fp16_pow2(k_new);
    const float enc = ldexpf(1.0f, -k_new);
    for (int64_t j = 0; j < bn; ++j) {
      const int64_t k = b0 + j;
      const float x = wn[j] * enc;
      q[k] = hp->stochastic ? orc_e4m3_sr(x, orc_rng_lane(hp->seed, (uint64_t)t, (uint64_t)(gidx0 + k), ORC_E4M3))
                            : orc_e4m3_rne(x);
    }
  }
  return 0;
}

void orc_dequant_bf16(int64_t n, const uint8_t* q, int32_t e, const uint16_t* bscale, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) {
    const float scale = bscale ? orc_fp16_decode(bscale[k / ORC_BLOCK]) : ldexpf(1.0f, e);
    out[k] = orc_bf16_rne(orc_e4m3_decode(q[k]) * scale);
  }
}

/* ------------------------------------------------------------------------ */
/* NVFP4: E2M1 payload, E4M3 block scales (16 elements), binary32 tensor     */
/* scale.  The paper stores master weights in NVFP4 (Sec. 5.2, the results   */
/* table's NVFP4/FP8 rows) and writes a block's weights as payload times     */
/* block scale (the FP4 block-scale paragraph of the ablation appendix).     */
/* ------------------------------------------------------------------------ */
static const float e2m1_grid[8] = {0.0f, 0.5f, 1.0f, 1.5f, 2.0f, 3.0f, 4.0f, 6.0f};

float orc_e2m1_decode(uint8_t c) {
  float v = e2m1_grid[c & 7u];
  return (c & 8u) ? -v : v;
}

/* Magnitude index of the grid point at or below a (a in [0, 6)), and the
 * fraction of the way to the next grid point, in binary64 (exact). */
static uint32_t e2m1_floor(float a, double* frac) {
  uint32_t i = 0;
  while (i < 6 && (double)e2m1_grid[i + 1] <= (double)a) ++i;
  *frac = ((double)a - (double)e2m1_grid[i]) / ((double)e2m1_grid[i + 1] - (double)e2m1_grid[i]);
  return i;
}

uint8_t orc_e2m1_rne(float x) {
  if (isnan(x)) return 0;
  uint32_t sign = signbit(x) ? 8u : 0u;
  float a = fabsf(x);
  if (a >= 6.0f) return (uint8_t)(sign | 7u);
  double frac;
  uint32_t i = e2m1_floor(a, &frac);
  if (frac > 0.5 || (frac == 0.5 && (i & 1u))) i += 1;   /* ties to the even code (mantissa 0) */
  return (uint8_t)(sign | i);
}

uint8_t orc_e2m1_sr(float x, uint32_t r32) {
  if (isnan(x)) return 0;
  uint32_t sign = signbit(x) ? 8u : 0u;
  float a = fabsf(x);
  if (a >= 6.0f) return (uint8_t)(sign | 7u);
  double frac;
  uint32_t i = e2m1_floor(a, &frac);
  double thr = floor(frac * 4294967296.0);                /* exact: frac has few bits */
  if ((double)r32 < thr) i += 1;
  return (uint8_t)(sign | i);
}

int32_t orc_nvfp4_scale_code(float amax, float G, int32_t c_old) {
  if (!(amax > 0.0f)) return c_old;
  for (int32_t c = 1; c <= 126; ++c) {
    float d = orc_e4m3_decode((uint8_t)c) * G;
    float top = 6.0f * d;
    if (top >= amax) return c;
  }
  return 126;
}

static uint8_t nvfp4_get(const uint8_t* q, int64_t k) {
  return (uint8_t)((k & 1) ? (q[k >> 1] >> 4) : (q[k >> 1] & 0x0Fu));
}

static void nvfp4_put(uint8_t* q, int64_t k, uint8_t c) {
  if (k & 1) q[k >> 1] = (uint8_t)((q[k >> 1] & 0x0Fu) | (c << 4));
  else q[k >> 1] = (uint8_t)((q[k >> 1] & 0xF0u) | (c & 0x0Fu));
}

int32_t orc_step_nvfp4(int64_t n, int64_t gidx0, int32_t gdt, int32_t mdt, uint8_t* q, uint8_t* bscale,
                       float G, const void* g, void* m, void* v, void* ve, const orc_hparams* hp, int64_t t) {
  if (gdt != ORC_F32 && gdt != ORC_BF16) return -1;
  if (mdt != ORC_F32 && mdt != ORC_BF16) return -1;
  if (!(G > 0.0f) || isinf(G)) return -1;
  orc_scalars s;
  if (orc_scalars_for_step(hp, t, &s) != 0) return -1;
  for (int64_t b0 = 0; b0 < n; b0 += ORC_FP4_BLOCK) {
    const int64_t bn = (n - b0 < ORC_FP4_BLOCK) ? n - b0 : ORC_FP4_BLOCK;
    const int64_t blk = b0 / ORC_FP4_BLOCK;
    const float d_old = orc_e4m3_decode(bscale[blk]) * G;
    float wn[ORC_FP4_BLOCK];
    float amax = 0.0f;
    for (int64_t j = 0; j < bn; ++j) {
      const int64_t k = b0 + j;
      float wk = orc_e2m1_decode(nvfp4_get(q, k)) * d_old;
      float gk = load_elem(g, k, gdt), mk = load_elem(m, k, mdt), vk = load_elem(v, k, mdt);
      float vek = load_elem(ve, k, mdt);
      float m1, v1, ve1;
      orc_update_element(&s, wk, gk, mk, vk, vek, &wn[j], &m1, &v1, &ve1);
      if (isfinite(wn[j]) && fabsf(wn[j]) > amax) amax = fabsf(wn[j]);
      store_moment(m, k, mdt, m1);
      store_moment(v, k, mdt, v1);
      store_moment(ve, k, mdt, ve1);
    }
    /* current scaling: the block's new scale covers its largest updated |w| */
    const int32_t c_new = orc_nvfp4_scale_code(amax, G, bscale[blk]);
    bscale[blk] = (uint8_t)c_new;
    const float d_new = orc_e4m3_decode((uint8_t)c_new) * G;
    for (int64_t j = 0; j < bn; ++j) {
      const int64_t k = b0 + j;
      const float x = wn[j] / d_new;
      const uint8_t c = hp->stochastic
          ? orc_e2m1_sr(x, orc_rng_lane(hp->seed, (uint64_t)t, (uint64_t)(gidx0 + k), ORC_E4M3))
          : orc_e2m1_rne(x);
      nvfp4_put(q, k, c);
    }
  }
  return 0;
}

void orc_dequant_nvfp4_bf16(int64_t n, const uint8_t* q, const uint8_t* bscale, float G, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) {
    const float d = orc_e4m3_decode(bscale[k / ORC_FP4_BLOCK]) * G;
    out[k] = orc_bf16_rne(orc_e2m1_decode(nvfp4_get(q, k)) * d);
  }
}

/* ------------------------------------------------------------------------ */
/* BF16-stored matrix fitting (the toy diagnostic of Sec. 5.1; its appendix  */
/* gives the loss c ||W - W*||^4 estimated on sampled entries, the three     */
/* update rules without moments, r_max = 0.75, tau = 1e-8, and the regimes). */
/* ------------------------------------------------------------------------ */
double orc_tree_sum(int64_t n, const double* x) {
  double* v = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  if (!v) return NAN;
  memcpy(v, x, sizeof(double) * (size_t)n);
  for (int64_t len = n; len > 1; len /= 2)
    for (int64_t i = 0; i < len / 2; ++i) v[i] = v[2 * i] + v[2 * i + 1];
  double r = n > 0 ? v[0] : 0.0;
  free(v);
  return r;
}

static int is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

double orc_toy_step(const orc_toy_config* c, int64_t n, uint16_t* w, const float* wstar, int64_t t) {
  if (!c || !w || !wstar || !is_pow2(n) || !is_pow2(c->batch) || c->batch < 64) return NAN;
  if (c->mode < 0 || c->mode > 2 || (c->split != 0 && c->split != 1)) return NAN;
  if (c->split && n < 2) return NAN;
  const int64_t B = c->batch, halves = c->split ? 2 : 1, Bh = B / halves, range = n / halves;
  int64_t* idx = (int64_t*)malloc(sizeof(int64_t) * (size_t)B);
  float* r = (float*)malloc(sizeof(float) * (size_t)B);
  double* sq = (double*)malloc(sizeof(double) * (size_t)Bh);
  int32_t* cnt = (int32_t*)calloc((size_t)n, sizeof(int32_t));
  int64_t* first = (int64_t*)calloc((size_t)n, sizeof(int64_t));   /* first sample + 1, 0 = none */
  if (!idx || !r || !sq || !cnt || !first) { free(idx); free(r); free(sq); free(cnt); free(first); return NAN; }

  /* sample with replacement; residuals of the stored weights */
  for (int64_t s = 0; s < B; ++s) {
    const int64_t h = c->split ? s / Bh : 0;
    const uint32_t lane = orc_rng_lane(c->seed, (uint64_t)t, (uint64_t)s, ORC_E4M3);
    idx[s] = h * range + (int64_t)((uint64_t)lane & (uint64_t)(range - 1));
    r[s] = orc_bf16_decode(w[idx[s]]) - wstar[idx[s]];
  }
  /* loss and gradient scale per half: M = mean r^2, L = c M^2, dL/dr_s = 4 c M r_s / B_h */
  double loss = 0.0;
  float alpha[2] = {0.0f, 0.0f};
  for (int64_t h = 0; h < halves; ++h) {
    for (int64_t i = 0; i < Bh; ++i) sq[i] = (double)r[h * Bh + i] * (double)r[h * Bh + i];
    const double M = orc_tree_sum(Bh, sq) / (double)Bh;
    const double ch = (double)(h == 0 ? c->c_lo : c->c_hi);
    loss += ch * M * M;
    alpha[h] = (float)(((4.0 * ch) * M) / (double)Bh);
  }
  /* hits per entry; the first sample of an entry applies its update */
  for (int64_t s = 0; s < B; ++s) {
    cnt[idx[s]] += 1;
    if (first[idx[s]] == 0) first[idx[s]] = s + 1;
  }
  const float ln2 = (float)0.693147180559945309417232121458;
  for (int64_t s = 0; s < B; ++s) {
    const int64_t j = idx[s];
    if (first[j] != s + 1) continue;
    const int64_t h = c->split ? s / Bh : 0;
    const float x = alpha[h] * r[s];
    float g = x;
    for (int32_t k = 1; k < cnt[j]; ++k) g = g + x;
    const float wf = orc_bf16_decode(w[j]);
    const float ua = -c->lr_add * g;
    const float ge = (ln2 * wf) * g;
    const float ut = -c->lr_mul * ge;
    const float rho = fabsf(wf) > c->tau ? fabsf(wf) : c->tau;
    float um = ut / rho;
    if (um > c->rmax) um = c->rmax;
    if (um < -c->rmax) um = -c->rmax;
    float wn;
    if (c->mode == 0) wn = wf + ua;
    else if (c->mode == 1) wn = fmaf(wf, um, wf);
    else wn = fmaf(wf, um, wf) + ua;
    w[j] = orc_bf16_rne(wn);
  }
  free(idx); free(r); free(sq); free(cnt); free(first);
  return loss;
}

/* ------------------------------------------------------------------------ */
/* Array helpers for the tests: plain loops over the scalar functions above. */
/* ------------------------------------------------------------------------ */
void orc_bf16_rne_n(int64_t n, const float* x, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_bf16_rne(x[k]);
}
void orc_bf16_sr_n(int64_t n, const float* x, const uint32_t* r16, uint16_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_bf16_sr(x[k], r16[k]);
}
void orc_e4m3_rne_n(int64_t n, const float* x, uint8_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_e4m3_rne(x[k]);
}
void orc_e4m3_sr_n(int64_t n, const float* x, const uint32_t* r32, uint8_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_e4m3_sr(x[k], r32[k]);
}
void orc_e4m3_decode_n(int64_t n, const uint8_t* q, float* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_e4m3_decode(q[k]);
}
void orc_rng_lanes_n(uint64_t seed, uint64_t t, int32_t storage, int64_t n,
                     const uint64_t* idx, uint32_t* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = orc_rng_lane(seed, t, idx[k], storage);
}
void orc_philox_n(int64_t n, const uint32_t* ctr, const uint32_t* key, uint32_t* out) {
  for (int64_t k = 0; k < n; ++k) orc_philox4x32_10(ctr + 4 * k, key, out + 4 * k);
}
int32_t orc_update_elements_n(const orc_hparams* hp, int64_t t, int64_t n,
                              const float* w, const float* g, const float* m,
                              const float* v, const float* ve,
                              float* wn, float* m1, float* v1, float* ve1) {
  orc_scalars s;
  if (orc_scalars_for_step(hp, t, &s) != 0) return -1;
  for (int64_t k = 0; k < n; ++k)
    orc_update_element(&s, w[k], g[k], m[k], v[k], ve[k], wn + k, m1 + k, v1 + k, ve1 + k);
  return 0;
}
