// step_kernel.cuh -- the fused M+Adam step kernel for sm_103a (GB300).
//
// One launch = one pass over every element: each thread takes groups of 8
// consecutive elements, loads w, g, mu, nu, nu_e with one coalesced vector
// load per array (256-bit for binary32 arrays, 128-bit for BF16, 64-bit for
// E4M3 weights), runs the canonical binary32 update (Algorithm 1 with the
// Algorithm 2 options, arxiv 2607.10611), rounds w into its storage format
// (nearest-even or Philox-keyed stochastic rounding) and stores everything
// back with one vector store per array.  The path is HBM-bound streaming:
// no shared-memory staging, no tensor cores (nothing here is a contraction).
//
// Numerics: every floating-point operation is an explicit round-to-nearest
// intrinsic (__fmul_rn, __fadd_rn, __fmaf_rn, __fdiv_rn, __fsqrt_rn), so the
// build flags cannot contract or approximate anything.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "step_args.h"

namespace mpadam {

// ---------------------------------------------------------------------------
// Global memory access: streaming vector loads/stores (no L1 allocation; each
// byte is touched exactly once).  Gradients are read-only for the whole
// launch and use the non-coherent path.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void ld8(const void* p, uint32_t (&r)[8]) {
  asm("ld.global.L1::no_allocate.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7])
      : "l"(p));
}
__device__ __forceinline__ void ld8_ro(const void* p, uint32_t (&r)[8]) {
  asm("ld.global.nc.L1::no_allocate.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7])
      : "l"(p));
}
__device__ __forceinline__ void ld4(const void* p, uint32_t (&r)[4]) {
  asm("ld.global.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
      : "l"(p));
}
__device__ __forceinline__ void ld4_ro(const void* p, uint32_t (&r)[4]) {
  asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
      : "l"(p));
}
__device__ __forceinline__ void ld2(const void* p, uint32_t (&r)[2]) {
  asm("ld.global.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "l"(p));
}
__device__ __forceinline__ void st8(void* p, const uint32_t (&r)[8]) {
  asm volatile("st.global.L1::no_allocate.v8.u32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
               :
               : "l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
                 "r"(r[6]), "r"(r[7])
               : "memory");
}
__device__ __forceinline__ void st4(void* p, const uint32_t (&r)[4]) {
  asm volatile("st.global.L1::no_allocate.v4.u32 [%0], {%1,%2,%3,%4};"
               :
               : "l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3])
               : "memory");
}
__device__ __forceinline__ void st2(void* p, const uint32_t (&r)[2]) {
  asm volatile("st.global.L1::no_allocate.v2.u32 [%0], {%1,%2};"
               :
               : "l"(p), "r"(r[0]), "r"(r[1])
               : "memory");
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds; each round
// takes the 64-bit products of words 0 and 2 with the two multipliers, feeds
// the high halves (xored with words 3 / 1 and the round key) to the other
// lane and the low halves straight through; the key steps by the Weyl pair.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3,
                                               uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t a_lo = 0xD2511F53u * x0;
    const uint32_t a_hi = __umulhi(0xD2511F53u, x0);
    const uint32_t b_lo = 0xCD9E8D57u * x2;
    const uint32_t b_hi = __umulhi(0xCD9E8D57u, x2);
    x0 = b_hi ^ x1 ^ k0;
    x1 = b_lo;
    x2 = a_hi ^ x3 ^ k1;
    x3 = a_lo;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return make_uint4(x0, x1, x2, x3);
}

// ---------------------------------------------------------------------------
// The canonical per-element update.
// ---------------------------------------------------------------------------
struct Upd {
  float wn, m, v, ve;
};

__device__ __forceinline__ Upd madam_update(const StepScalars& s, float w, float g, float m,
                                            float v, float ve) {
  Upd o;
  // additive branch (Adam moments, bias correction folded into ka and c2)
  o.m = __fmaf_rn(s.b1, m, __fmul_rn(s.omb1, g));
  o.v = __fmaf_rn(s.b2, v, __fmul_rn(s.omb2, __fmul_rn(g, g)));
  float ua = __fdiv_rn(__fmul_rn(s.ka, o.m), __fmaf_rn(__fsqrt_rn(o.v), s.c2, s.eps));
  if (s.wd_on) ua = __fsub_rn(ua, __fmul_rn(s.kwd, w));
  // multiplicative branch: exponent gradient, its second moment, proposal
  const float ge = __fmul_rn(__fmul_rn(s.ln2, w), g);
  o.ve = __fmaf_rn(s.b2, ve, __fmul_rn(s.omb2, __fmul_rn(ge, ge)));
  float n = __fdiv_rn(ge, __fmaf_rn(__fsqrt_rn(o.ve), s.c2, s.eps));
  if (s.gmax_on) n = fmaxf(-s.gmax, fminf(n, s.gmax));
  float um = __fdiv_rn(__fmul_rn(s.km, n), fmaxf(fabsf(w), s.tau));
  um = fmaxf(s.lo, fminf(um, s.hi));
  // combine: w + w u_m + u_a
  float wn = __fadd_rn(__fmaf_rn(w, um, w), ua);
  if (s.wmax_on) wn = fmaxf(-s.wmax, fminf(wn, s.wmax));
  o.wn = wn;
  return o;
}

// ---------------------------------------------------------------------------
// Storage formats
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

// Two binary32 -> packed BF16 pair, nearest-even (hardware conversion).
__device__ __forceinline__ uint32_t bf16x2_rn(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// Stochastic BF16 of x given the complement of its 16 random bits in the low
// half of `nr`: adding 0xFFFF - R carries into the kept half exactly when
// R < (low half of x), i.e. with probability (low half) / 2^16.  Returns the
// 32-bit sum whose high half is the result.
__device__ __forceinline__ uint32_t bf16_sr_sum(float x, uint32_t nr16) {
  const uint32_t sum = __float_as_uint(x) + nr16;
  return (x != x) ? 0x7FFF0000u : sum;
}

// E4M3 code -> binary32 (exact).
__device__ __forceinline__ float e4m3_value(uint32_t c) {
  const uint32_t mag = c & 0x7Fu;
  float val;
  if (mag >= 8u) {
    val = __uint_as_float((mag << 20) + (120u << 23));  // exponent field + 120, mantissa
  } else {
    val = __fmul_rn(__uint2float_rn(mag), 0.001953125f);  // mag * 2^-9
  }
  if (mag == 0x7Fu) val = __uint_as_float(0x7FC00000u);
  return (c & 0x80u) ? -val : val;
}

// binary32 (already scaled by 2^-e) -> E4M3 code, saturating at +-448.
template <bool SR>
__device__ __forceinline__ uint32_t e4m3_encode(float x, uint32_t r) {
  const uint32_t b = __float_as_uint(x);
  const uint32_t sign = (b >> 24) & 0x80u;
  const uint32_t a = b & 0x7FFFFFFFu;
  if (a >= 0x43E00000u) return a > 0x7F800000u ? 0x7Fu : (sign | 0x7Eu);  // NaN / >= 448
  uint32_t code;
  if (a >= 0x3C800000u) {  // |x| >= 2^-6: normal E4M3, 20 mantissa bits dropped
    const uint32_t base = (a >> 20) - 960u;
    const uint32_t rem = a & 0xFFFFFu;
    uint32_t up;
    if (SR) up = r < (rem << 12) ? 1u : 0u;
    else up = (rem > 0x80000u || (rem == 0x80000u && (base & 1u))) ? 1u : 0u;
    code = base + up;
  } else {  // subnormal E4M3: count in units of 2^-9 (scaling by 2^9 is exact)
    const float y = __fmul_rn(__uint_as_float(a), 512.0f);
    if (SR) {
      const float fl = truncf(y);
      const float frac = __fsub_rn(y, fl);  // exact
      const uint32_t thr = __float2uint_rz(__fmul_rn(frac, 4294967296.0f));
      code = __float2uint_rz(fl) + (r < thr ? 1u : 0u);
    } else {
      code = __float2uint_rn(y);  // nearest, ties to even
    }
  }
  code = code > 0x7Eu ? 0x7Eu : code;
  return sign | code;
}

// Delayed per-tensor scale: smallest e with A <= 448 * 2^e (A as binary32
// bits, finite and >= 0); keep e_cur when A = 0; clamp to [-100, 100].
__device__ __forceinline__ int32_t fp8_next_exponent(uint32_t a_bits, int32_t e_cur) {
  if (a_bits == 0u) return e_cur;
  const int32_t ef = (int32_t)(a_bits >> 23);
  int32_t k = -100;
  if (ef != 0) k = ef - 127 - 8 + ((a_bits & 0x7FFFFFu) > 0x600000u ? 1 : 0);
  return k < -100 ? -100 : (k > 100 ? 100 : k);
}

__device__ __forceinline__ float pow2f(int32_t e) { return __uint_as_float((uint32_t)(e + 127) << 23); }

// ---------------------------------------------------------------------------
// One group of 8 elements.  FULL: all 8 valid and every pointer aligned for
// vector access; otherwise element-wise loads/stores of the `valid` leading
// elements.
// ---------------------------------------------------------------------------
template <int WD, int GD, int MD, bool SR, bool FULL>
__device__ __forceinline__ void process_group(const StepArgs& a, const TensorDesc& d,
                                              const void* gp, int64_t e0, int valid, int64_t gi,
                                              float dec_scale, float enc_scale,
                                              uint32_t& amax_bits) {
  float w[8], g[8], m[8], v[8], ve[8];
  // ---- loads -------------------------------------------------------------
  if (FULL) {
    if (WD == kBF16) {
      uint32_t r[4];
      ld4(static_cast<const uint16_t*>(d.w) + e0, r);
#pragma unroll
      for (int i = 0; i < 4; ++i) { w[2 * i] = bf16_lo(r[i]); w[2 * i + 1] = bf16_hi(r[i]); }
    } else {
      uint32_t r[2];
      ld2(static_cast<const uint8_t*>(d.w) + e0, r);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        w[j] = __fmul_rn(e4m3_value((r[j >> 2] >> (8 * (j & 3))) & 0xFFu), dec_scale);
    }
    if (GD == kF32) {
      uint32_t r[8];
      ld8_ro(static_cast<const float*>(gp) + e0, r);
#pragma unroll
      for (int j = 0; j < 8; ++j) g[j] = __uint_as_float(r[j]);
    } else {
      uint32_t r[4];
      ld4_ro(static_cast<const uint16_t*>(gp) + e0, r);
#pragma unroll
      for (int i = 0; i < 4; ++i) { g[2 * i] = bf16_lo(r[i]); g[2 * i + 1] = bf16_hi(r[i]); }
    }
    if (MD == kF32) {
      uint32_t rm[8], rv[8], re[8];
      ld8(static_cast<const float*>(d.m) + e0, rm);
      ld8(static_cast<const float*>(d.v) + e0, rv);
      ld8(static_cast<const float*>(d.ve) + e0, re);
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        m[j] = __uint_as_float(rm[j]); v[j] = __uint_as_float(rv[j]); ve[j] = __uint_as_float(re[j]);
      }
    } else {
      uint32_t rm[4], rv[4], re[4];
      ld4(static_cast<const uint16_t*>(d.m) + e0, rm);
      ld4(static_cast<const uint16_t*>(d.v) + e0, rv);
      ld4(static_cast<const uint16_t*>(d.ve) + e0, re);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        m[2 * i] = bf16_lo(rm[i]); m[2 * i + 1] = bf16_hi(rm[i]);
        v[2 * i] = bf16_lo(rv[i]); v[2 * i + 1] = bf16_hi(rv[i]);
        ve[2 * i] = bf16_lo(re[i]); ve[2 * i + 1] = bf16_hi(re[i]);
      }
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      w[j] = g[j] = m[j] = v[j] = ve[j] = 0.0f;
      if (j < valid) {
        const int64_t e = e0 + j;
        if (WD == kBF16) w[j] = __uint_as_float((uint32_t)static_cast<const uint16_t*>(d.w)[e] << 16);
        else w[j] = __fmul_rn(e4m3_value(static_cast<const uint8_t*>(d.w)[e]), dec_scale);
        if (GD == kF32) g[j] = static_cast<const float*>(gp)[e];
        else g[j] = __uint_as_float((uint32_t)static_cast<const uint16_t*>(gp)[e] << 16);
        if (MD == kF32) {
          m[j] = static_cast<const float*>(d.m)[e];
          v[j] = static_cast<const float*>(d.v)[e];
          ve[j] = static_cast<const float*>(d.ve)[e];
        } else {
          m[j] = __uint_as_float((uint32_t)static_cast<const uint16_t*>(d.m)[e] << 16);
          v[j] = __uint_as_float((uint32_t)static_cast<const uint16_t*>(d.v)[e] << 16);
          ve[j] = __uint_as_float((uint32_t)static_cast<const uint16_t*>(d.ve)[e] << 16);
        }
      }
    }
  }

  // ---- random bits (one Philox block per 8 BF16 lanes / 4 E4M3 lanes) ----
  uint32_t rnd[8];
  if (SR) {
    if (WD == kBF16) {
      const uint4 r = philox4x32_10((uint32_t)gi, (uint32_t)((uint64_t)gi >> 32), a.t_lo, a.t_hi,
                                    a.key0, a.key1);
      // complemented 16-bit lanes, ready for the carry trick
      rnd[0] = ~r.x & 0xFFFFu; rnd[1] = ~r.x >> 16;
      rnd[2] = ~r.y & 0xFFFFu; rnd[3] = ~r.y >> 16;
      rnd[4] = ~r.z & 0xFFFFu; rnd[5] = ~r.z >> 16;
      rnd[6] = ~r.w & 0xFFFFu; rnd[7] = ~r.w >> 16;
    } else {
      const uint64_t b0 = 2ull * (uint64_t)gi;
      const uint4 r0 = philox4x32_10((uint32_t)b0, (uint32_t)(b0 >> 32), a.t_lo, a.t_hi, a.key0, a.key1);
      const uint64_t b1 = b0 + 1ull;
      const uint4 r1 = philox4x32_10((uint32_t)b1, (uint32_t)(b1 >> 32), a.t_lo, a.t_hi, a.key0, a.key1);
      rnd[0] = r0.x; rnd[1] = r0.y; rnd[2] = r0.z; rnd[3] = r0.w;
      rnd[4] = r1.x; rnd[5] = r1.y; rnd[6] = r1.z; rnd[7] = r1.w;
    }
  }

  // ---- update ------------------------------------------------------------
  float wn[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const Upd u = madam_update(a.s, w[j], g[j], m[j], v[j], ve[j]);
    wn[j] = u.wn; m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
  }

  // ---- encode + store ------------------------------------------------------
  if (WD == kBF16) {
    uint32_t ow[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (SR) {
        const uint32_t s0 = bf16_sr_sum(wn[2 * i], rnd[2 * i]);
        const uint32_t s1 = bf16_sr_sum(wn[2 * i + 1], rnd[2 * i + 1]);
        ow[i] = __byte_perm(s0, s1, 0x7632);
      } else {
        ow[i] = bf16x2_rn(wn[2 * i], wn[2 * i + 1]);
      }
    }
    if (FULL) {
      st4(static_cast<uint16_t*>(d.w) + e0, ow);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < valid)
          static_cast<uint16_t*>(d.w)[e0 + j] = (uint16_t)((j & 1) ? (ow[j >> 1] >> 16) : (ow[j >> 1] & 0xFFFFu));
    }
  } else {
    uint32_t ow[2] = {0u, 0u};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint32_t wb = __float_as_uint(wn[j]) & 0x7FFFFFFFu;
      if ((FULL || j < valid) && wb < 0x7F800000u) amax_bits = max(amax_bits, wb);
      const uint32_t c = e4m3_encode<SR>(__fmul_rn(wn[j], enc_scale), SR ? rnd[j] : 0u);
      ow[j >> 2] |= c << (8 * (j & 3));
    }
    if (FULL) {
      st2(static_cast<uint8_t*>(d.w) + e0, ow);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < valid) static_cast<uint8_t*>(d.w)[e0 + j] = (uint8_t)(ow[j >> 2] >> (8 * (j & 3)));
    }
  }

  if (MD == kF32) {
    if (FULL) {
      uint32_t om[8], ov[8], oe[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        om[j] = __float_as_uint(m[j]); ov[j] = __float_as_uint(v[j]); oe[j] = __float_as_uint(ve[j]);
      }
      st8(static_cast<float*>(d.m) + e0, om);
      st8(static_cast<float*>(d.v) + e0, ov);
      st8(static_cast<float*>(d.ve) + e0, oe);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < valid) {
          static_cast<float*>(d.m)[e0 + j] = m[j];
          static_cast<float*>(d.v)[e0 + j] = v[j];
          static_cast<float*>(d.ve)[e0 + j] = ve[j];
        }
    }
  } else {
    uint32_t om[4], ov[4], oe[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      om[i] = bf16x2_rn(m[2 * i], m[2 * i + 1]);
      ov[i] = bf16x2_rn(v[2 * i], v[2 * i + 1]);
      oe[i] = bf16x2_rn(ve[2 * i], ve[2 * i + 1]);
    }
    if (FULL) {
      st4(static_cast<uint16_t*>(d.m) + e0, om);
      st4(static_cast<uint16_t*>(d.v) + e0, ov);
      st4(static_cast<uint16_t*>(d.ve) + e0, oe);
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (j < valid) {
          const int sh = (j & 1) ? 16 : 0;
          static_cast<uint16_t*>(d.m)[e0 + j] = (uint16_t)(om[j >> 1] >> sh);
          static_cast<uint16_t*>(d.v)[e0 + j] = (uint16_t)(ov[j >> 1] >> sh);
          static_cast<uint16_t*>(d.ve)[e0 + j] = (uint16_t)(oe[j >> 1] >> sh);
        }
    }
  }
}

__device__ __forceinline__ bool aligned(const void* p, uintptr_t bytes) {
  return (reinterpret_cast<uintptr_t>(p) & (bytes - 1)) == 0;
}

// ---------------------------------------------------------------------------
// The persistent step kernel: one CTA per slice of the global group range.
// ---------------------------------------------------------------------------
template <int WD, int GD, int MD, bool SR>
__global__ void __launch_bounds__(kThreads) step_kernel(const __grid_constant__ StepArgs a) {
  const int64_t G = a.total_groups;
  const int64_t g_begin = (int64_t)blockIdx.x * G / gridDim.x;
  const int64_t g_end = ((int64_t)blockIdx.x + 1) * G / gridDim.x;
  if (g_begin >= g_end) return;
  const int n = a.n_tensors;

  for (int k = a.cta_first[blockIdx.x]; k < n; ++k) {
    const TensorDesc d = a.desc[k];
    const int64_t t0 = d.goff >> 3;
    const int64_t t1 = t0 + ((d.numel + 7) >> 3);
    if (t0 >= g_end) break;
    const int64_t lo = g_begin > t0 ? g_begin : t0;
    const int64_t hi = g_end < t1 ? g_end : t1;
    if (lo >= hi) continue;
    const void* gp = a.grads[k];

    const bool vec = aligned(d.w, WD == kBF16 ? 16 : 8) && aligned(gp, GD == kF32 ? 32 : 16) &&
                     aligned(d.m, MD == kF32 ? 32 : 16) && aligned(d.v, MD == kF32 ? 32 : 16) &&
                     aligned(d.ve, MD == kF32 ? 32 : 16);

    float dec_scale = 1.0f, enc_scale = 1.0f;
    if (WD == kE4M3) {
      const int32_t e_cur = a.fp8_exp[(int64_t)a.e_cur_slot * n + k];
      const uint32_t a_cur = a.fp8_amax[(int64_t)a.a_cur_slot * n + k];
      const int32_t e_next = fp8_next_exponent(a_cur, e_cur);
      dec_scale = pow2f(e_cur);
      enc_scale = pow2f(-e_next);
      if (lo == t0 && threadIdx.x == 0) {  // the CTA holding the tensor's first group
        a.fp8_exp[(int64_t)a.e_next_slot * n + k] = e_next;
        a.fp8_amax[(int64_t)a.a_zero_slot * n + k] = 0u;
      }
    }

    uint32_t amax_bits = 0u;
    for (int64_t gi = lo + threadIdx.x; gi < hi; gi += kThreads) {
      const int64_t e0 = (gi - t0) * kGroup;
      const int64_t left = d.numel - e0;
      const int valid = left < kGroup ? (int)left : kGroup;
      if (vec && valid == kGroup)
        process_group<WD, GD, MD, SR, true>(a, d, gp, e0, valid, gi, dec_scale, enc_scale, amax_bits);
      else
        process_group<WD, GD, MD, SR, false>(a, d, gp, e0, valid, gi, dec_scale, enc_scale, amax_bits);
    }

    if (WD == kE4M3) {
      const uint32_t wmax = __reduce_max_sync(0xFFFFFFFFu, amax_bits);
      if ((threadIdx.x & 31) == 0 && wmax != 0u)
        atomicMax(&a.fp8_amax[(int64_t)a.a_next_slot * n + k], wmax);
    }
  }
}

}  // namespace mpadam
