/*
 * mpadam_oracle.h -- plain single-threaded CPU oracle of the M+Adam optimizer
 * step (arxiv 2607.10611, Algorithm 1 with the options of Algorithm 2,
 * Appendix A).
 *
 * TEST INFRASTRUCTURE ONLY. Only the test suite, the smoke check and the CPU
 * baseline leg of the benchmark may load this library. The product library
 * (include/mpadam.h, the CUDA kernels) shares no code, header, table or
 * helper with this file, and neither side includes or links the other.
 *
 * Arithmetic model: every per-element operation is an IEEE-754 binary32
 * operation with round-to-nearest-even (the paper's toy diagnostic, Sec. 5.1
 * and Appendix B, computes each step in FP32 and rounds the parameter
 * immediately).  Fused multiply-adds appear only where written as fmaf().
 * Build with -ffp-contract=off so the compiler adds no others.
 */
#ifndef MPADAM_ORACLE_H
#define MPADAM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element formats.  ORC_E4M3_B32: E4M3 codes with one power-of-two scale
 * per 32 consecutive elements, stored as FP16 bits.  ORC_NVFP4: E2M1 codes
 * (two per byte, the even element in the low nibble) with one E4M3 scale per
 * 16 consecutive elements and one binary32 scale per tensor. */
enum { ORC_F32 = 0, ORC_BF16 = 1, ORC_E4M3 = 2, ORC_E4M3_B32 = 3, ORC_NVFP4 = 4 };
enum { ORC_BLOCK = 32, ORC_FP4_BLOCK = 16 };

/* Hyper-parameters (Algorithm 1 inputs; Algorithm 2 optional clips). */
typedef struct {
  float lr_add;          /* eta_a */
  float lr_mul;          /* eta_m */
  float beta1, beta2;    /* moment decay rates */
  float eps;             /* stabiliser, > 0 */
  float tau;             /* threshold of rho = max(|w|, tau), > 0 */
  float rmax_pos;        /* upper bound of u_m (0.75 in Algorithm 2) */
  float rmax_neg;        /* magnitude of the lower bound, 0.75 - eps0 */
  float g_max;           /* clamp of the normalised exponent gradient; +inf = off */
  float dmult_max;       /* cap on |log2(1 + u_m)|; +inf = off */
  float w_max;           /* final weight clip; +inf = off */
  float wd_add;          /* decoupled additive weight decay lambda; 0 = off */
  int32_t bias_correction; /* 1: Algorithm 1 (u-hat, v-hat); 0: Algorithm 2 */
  int32_t stochastic;    /* 0: round to nearest even, 1: stochastic rounding */
  uint64_t seed;         /* Philox key */
} orc_hparams;

/* Per-step binary32 scalars, each computed in binary64 and rounded once. */
typedef struct {
  float b1, b2;      /* beta1, beta2 */
  float omb1, omb2;  /* 1 - beta1, 1 - beta2 */
  float ka;          /* -eta_a / (1 - beta1^t)   (or -eta_a without bias correction) */
  float c2;          /* 1 / sqrt(1 - beta2^t)    (or 1) */
  float km;          /* -eta_m */
  float ln2;         /* ln 2 */
  float eps, tau;
  float lo, hi;      /* bounds of u_m: rmax and the log2 step cap merged */
  float gmax, wmax, kwd;
  int32_t gmax_on, wmax_on, wd_on;
} orc_scalars;

/* Philox4x32-10 block function (Salmon et al., SC'11). */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);

/* Random bits drawn for global element index i at step t:
 * BF16 storage: 16 bits, E4M3 storage: 32 bits. */
uint32_t orc_rng_lane(uint64_t seed, uint64_t t, uint64_t i, int32_t storage);

uint16_t orc_bf16_rne(float x);
uint16_t orc_bf16_sr(float x, uint32_t r16);
float    orc_bf16_decode(uint16_t h);
uint8_t  orc_e4m3_rne(float x);
uint8_t  orc_e4m3_sr(float x, uint32_t r32);
float    orc_e4m3_decode(uint8_t q);

/* Per-tensor power-of-two scale exponent for the next encode. */
int32_t  orc_fp8_next_exponent(float amax, int32_t e_cur);

/* 0 on success, -1 on invalid hyper-parameters or t < 1. */
int32_t  orc_scalars_for_step(const orc_hparams* hp, int64_t t, orc_scalars* out);

/* The canonical per-element update in binary32. */
void orc_update_element(const orc_scalars* s, float w, float g, float m, float v, float ve,
                        float* wn, float* m1, float* v1, float* ve1);

/* One optimizer step over n elements held in host arrays, updated in place.
 * Element k has global index gidx[k] (or gidx0 + k when gidx is NULL).
 * E4M3 weights decode with 2^e_cur and encode with 2^e_next; *amax is raised
 * to the largest finite |updated weight| seen.  Returns 0 or -1. */
int32_t orc_step_elements(int64_t n, const int64_t* gidx, int64_t gidx0,
                          int32_t wdt, int32_t gdt, int32_t mdt,
                          void* w, const void* g, void* m, void* v, void* ve,
                          const orc_hparams* hp, int64_t t,
                          int32_t e_cur, int32_t e_next, float* amax);

/* Largest finite |decoded E4M3 weight| of a tensor stored with exponent e. */
float orc_e4m3_amax(int64_t n, const uint8_t* q, int32_t e);

/* FP16 bit pattern of 2^k, k in [-24, 15] (exact: subnormal below 2^-14). */
uint16_t orc_fp16_pow2(int32_t k);
/* Value of an FP16 bit pattern (exact). */
float orc_fp16_decode(uint16_t h);
/* Block scale exponent: smallest k with amax <= 448 2^k, clamped to
 * [-24, 15]; k_old when amax is 0. */
int32_t orc_block_exponent(float amax, int32_t k_old);

/* One optimizer step over a whole tensor of E4M3 weights with FP16
 * power-of-two scales per 32-element block (current scaling: each block's
 * new scale comes from the largest finite |updated weight| of that block).
 * q: n codes, bscale: ceil(n/32) FP16 scales (both updated in place);
 * element j has global index gidx0 + j.  Returns 0 or -1. */
int32_t orc_step_block_e4m3(int64_t n, int64_t gidx0, int32_t gdt, int32_t mdt,
                            uint8_t* q, uint16_t* bscale, const void* g, void* m, void* v, void* ve,
                            const orc_hparams* hp, int64_t t);

/* BF16 compute copy of stored E4M3 weights: bf16(decode(q) * scale), exact.
 * Per-tensor scale 2^e (bscale NULL) or per-32-block FP16 scales. */
void orc_dequant_bf16(int64_t n, const uint8_t* q, int32_t e, const uint16_t* bscale, uint16_t* out);

/* E2M1 (OCP FP4: sign, 2 exponent bits with bias 1, 1 mantissa bit; values
 * +-{0, 0.5, 1, 1.5, 2, 3, 4, 6}, no infinity or NaN) codes in the low 4
 * bits.  Nearest-even or stochastic (away from zero iff r32 < floor(fraction
 * * 2^32)); |x| >= 6 and infinities saturate to +-6; NaN gives +0. */
uint8_t orc_e2m1_rne(float x);
uint8_t orc_e2m1_sr(float x, uint32_t r32);
float   orc_e2m1_decode(uint8_t c);

/* NVFP4 block scale: the smallest E4M3 code c in [1, 126] whose block range
 * covers amax, i.e. 6 * (value(c) * G) >= amax with both products rounded to
 * binary32; 126 when none does; c_old when amax is 0. */
int32_t orc_nvfp4_scale_code(float amax, float G, int32_t c_old);

/* One optimizer step over a whole NVFP4 tensor (current block scaling).
 * q: ceil(n/2) bytes of codes, bscale: ceil(n/16) E4M3 scale codes (both
 * updated in place), G the tensor scale (> 0, finite).  Element j decodes as
 * q_j * d_b with d_b = value(bscale[b]) * G (rounded to binary32), and
 * re-encodes x_j = w'_j / d_b' (rounded to binary32) with the block's new
 * scale.  Element j has global index gidx0 + j (32-bit random lanes, as for
 * E4M3).  Returns 0 or -1. */
int32_t orc_step_nvfp4(int64_t n, int64_t gidx0, int32_t gdt, int32_t mdt, uint8_t* q, uint8_t* bscale,
                       float G, const void* g, void* m, void* v, void* ve, const orc_hparams* hp, int64_t t);

/* BF16 compute copy of NVFP4 weights: bf16(q_j * d_b) with d_b as above. */
void orc_dequant_nvfp4_bf16(int64_t n, const uint8_t* q, const uint8_t* bscale, float G, uint16_t* out);

/* BF16-stored matrix-fitting diagnostic (the toy diagnostic of Sec. 5.1 and
 * its appendix).  One step: B entries of W are sampled uniformly with
 * replacement (sample s takes the 32-bit random lane s of step t, as E4M3
 * storage does, masked to the index range); the minibatch loss is
 * c (mean of the sampled squared residuals)^2 -- per half when split (the
 * mixed-scales regime: entries [0, n/2) and [n/2, n) are separate problems
 * with B/2 samples each); the gradient of an entry hit k times is its
 * contribution alpha r added k times, alpha = 4 c M / B_h; the update is
 * the additive, multiplicative or combined step without moments, rounded to
 * BF16 (nearest-even).  Means are perfect binary trees of binary64 sums
 * over adjacent samples. */
typedef struct {
  int32_t mode;      /* 0 additive, 1 multiplicative, 2 combined (eta_a = lr_add, eta_m = lr_mul) */
  int32_t split;     /* 1: the two halves are separate sub-problems */
  int32_t batch;     /* B: a power of two, >= 64 */
  int32_t pad;
  float lr_add, lr_mul;
  float rmax, tau;   /* clip of u_m and floor of rho */
  float c_lo, c_hi;  /* loss constant of the first / second half (c_lo alone when split = 0) */
  uint64_t seed;
} orc_toy_config;

/* Perfect binary tree of binary64 sums over adjacent pairs (n a power of two). */
double orc_tree_sum(int64_t n, const double* x);

/* One step on W (n BF16 entries, n a power of two), updated in place;
 * returns the minibatch loss before the update, or NaN on bad arguments. */
double orc_toy_step(const orc_toy_config* c, int64_t n, uint16_t* w, const float* wstar, int64_t t);

/* Array forms of the scalar functions (plain loops), for the tests. */
void orc_bf16_rne_n(int64_t n, const float* x, uint16_t* out);
void orc_bf16_sr_n(int64_t n, const float* x, const uint32_t* r16, uint16_t* out);
void orc_e4m3_rne_n(int64_t n, const float* x, uint8_t* out);
void orc_e4m3_sr_n(int64_t n, const float* x, const uint32_t* r32, uint8_t* out);
void orc_e4m3_decode_n(int64_t n, const uint8_t* q, float* out);
void orc_rng_lanes_n(uint64_t seed, uint64_t t, int32_t storage, int64_t n,
                     const uint64_t* idx, uint32_t* out);
void orc_philox_n(int64_t n, const uint32_t* ctr, const uint32_t* key, uint32_t* out);
int32_t orc_update_elements_n(const orc_hparams* hp, int64_t t, int64_t n,
                              const float* w, const float* g, const float* m,
                              const float* v, const float* ve,
                              float* wn, float* m1, float* v1, float* ve1);

#ifdef __cplusplus
}
#endif
#endif
