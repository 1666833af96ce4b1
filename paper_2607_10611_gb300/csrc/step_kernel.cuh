// step_kernel.cuh -- the fused M+Adam step kernel for sm_103a (GB300).
//
// One launch = one pass over every element of the tensor list.  Each CTA
// (one per SM) is a producer/consumer pipeline over its tiles:
//   - one producer warp (one elected lane) picks each tile -- the next of its
//     own range, then chunks claimed from the launch's tail pool -- posts the
//     tile and its tensor beside the stage, and streams the tile's slice of
//     every array (weights w, gradients g and the moments mu, nu, nu_e, each
//     one contiguous run of bytes) into a multi-stage shared-memory ring with
//     1-D TMA bulk copies (cp.async.bulk ... mbarrier::complete_tx), evict-
//     first in L2 since every byte is used once; an end marker in the next
//     stage tells the consumers that the work is done;
//   - fifteen consumer warps wait on the stage's mbarrier, read their 8
//     elements from shared memory, run the canonical binary32 update
//     (Algorithm 1 with the Algorithm 2 options, arxiv 2607.10611), round the
//     weight into its storage format (nearest-even, or stochastic with
//     Philox4x32-10 bits) and store w, mu, nu, nu_e straight back to HBM with
//     vector stores (256-bit for binary32 arrays), then release the stage.
// Memory latency is hidden by the ring, not by occupancy, so the consumers'
// instruction stream is the only other limit.  Tensor tails that are not a
// whole number of 16-byte chunks, and tensors whose pointers are not 16-byte
// aligned, are read by the consumers directly from global memory with the
// same arithmetic.  No tensor cores: nothing here is a contraction.
//
// Numerics: every floating-point operation of the canonical sequence is an
// explicit round-to-nearest intrinsic (__fmul_rn, __fadd_rn, __fmaf_rn,
// __fdiv_rn, __fsqrt_rn), so build flags cannot contract or approximate
// anything.  The certified fast path below uses approximate square roots and
// divisions only where a rounding test proves the stored result equal to the
// canonical one; everything else is recomputed canonically.
//
// Every wait on an mbarrier is bounded; a wait that gives up sets a bit in
// *err, the producer waits (again bounded) for its own copies in flight, and
// the CTA returns.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "step_args.h"

namespace mpadam {

constexpr uint32_t kSpinLimit = 1u << 22;  // mbarrier try_wait attempts before giving up (seconds)

// ---------------------------------------------------------------------------
// Global memory: streaming vector loads/stores (no L1 allocation).
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
// 256-bit stores carry the binary32 moments (nothing else uses them).  HINT
// adds an L2 evict-first policy, chosen per kernel instance as measured (two
// or three alternating runs each): with it the 1.5B list ran 1.4 % faster,
// the ragged list, GPT-2 and the NVFP4 regime with RNE 0.4-0.6 %, the FP8
// regime 0.1 % slower; the NVFP4 regime with SR (issue-bound) 1.2 % slower,
// so its instance stores plain.  The same hint on the 128-bit stores of BF16
// moments slowed the 7B list by 0.2 %, so those stay plain.
template <bool HINT = true>
__device__ __forceinline__ void st8(void* p, const uint32_t (&r)[8]) {
  if constexpr (HINT) {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    asm volatile("st.global.L1::no_allocate.L2::cache_hint.v8.u32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8}, %9;"
                 :
                 : "l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
                   "r"(r[6]), "r"(r[7]), "l"(pol)
                 : "memory");
  } else {
    asm volatile("st.global.L1::no_allocate.v8.u32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
                 :
                 : "l"(p), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
                   "r"(r[6]), "r"(r[7])
                 : "memory");
  }
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
// Shared memory, mbarriers and the TMA bulk copy
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void lds4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void lds2(uint32_t addr, uint32_t (&r)[2]) {
  asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "r"(addr));
}
__device__ __forceinline__ uint32_t lds_u16(uint32_t addr) {
  uint16_t h;
  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(h) : "r"(addr));
  return h;
}
__device__ __forceinline__ uint32_t lds_u8(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait until the phase with the given parity has completed; false after
// kSpinLimit attempts.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (uint32_t i = 0; i < kSpinLimit; ++i)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}
__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
// 1-D bulk copy global -> shared, completing `bytes` of transaction on `bar`.
// Source and destination 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void tma_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                         uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(pol)
      : "memory");
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) with precomputed round
// keys rk[r] = key + r * (Weyl constants): each round takes the 64-bit
// products of words 0 and 2 with the two multipliers, feeds the high halves
// (xored with words 3 / 1 and the round key) across and the low halves
// straight through.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3,
                                               const uint32_t (&rk0)[kPhiloxRounds],
                                               const uint32_t (&rk1)[kPhiloxRounds]) {
#pragma unroll
  for (int r = 0; r < kPhiloxRounds; ++r) {
    const uint64_t pa = static_cast<uint64_t>(x0) * 0xD2511F53u;
    const uint64_t pb = static_cast<uint64_t>(x2) * 0xCD9E8D57u;
    const uint32_t y0 = static_cast<uint32_t>(pb >> 32) ^ x1 ^ rk0[r];
    const uint32_t y2 = static_cast<uint32_t>(pa >> 32) ^ x3 ^ rk1[r];
    x1 = static_cast<uint32_t>(pb);
    x3 = static_cast<uint32_t>(pa);
    x0 = y0;
    x2 = y2;
  }
  return make_uint4(x0, x1, x2, x3);
}

// ---------------------------------------------------------------------------
// The canonical per-element update.
// ---------------------------------------------------------------------------
struct Upd {
  float wn, m, v, ve;
};

template <bool OPT>
__device__ __forceinline__ Upd madam_update(const StepScalars& s, float w, float g, float m, float v,
                                            float ve) {
  Upd o;
  // additive branch (Adam moments, bias correction folded into ka and c2)
  o.m = __fmaf_rn(s.b1, m, __fmul_rn(s.omb1, g));
  o.v = __fmaf_rn(s.b2, v, __fmul_rn(s.omb2, __fmul_rn(g, g)));
  float ua = __fdiv_rn(__fmul_rn(s.ka, o.m), __fmaf_rn(__fsqrt_rn(o.v), s.c2, s.eps));
  if (OPT && s.wd_on) ua = __fsub_rn(ua, __fmul_rn(s.kwd, w));
  // multiplicative branch: exponent gradient, its second moment, proposal
  const float ge = __fmul_rn(__fmul_rn(s.ln2, w), g);
  o.ve = __fmaf_rn(s.b2, ve, __fmul_rn(s.omb2, __fmul_rn(ge, ge)));
  float n = __fdiv_rn(ge, __fmaf_rn(__fsqrt_rn(o.ve), s.c2, s.eps));
  if (OPT && s.gmax_on) n = fmaxf(-s.gmax, fminf(n, s.gmax));
  float um = __fdiv_rn(__fmul_rn(s.km, n), fmaxf(fabsf(w), s.tau));
  um = fmaxf(s.lo, fminf(um, s.hi));
  // combine: w + w u_m + u_a
  float wn = __fadd_rn(__fmaf_rn(w, um, w), ua);
  if (OPT && s.wmax_on) wn = fmaxf(-s.wmax, fminf(wn, s.wmax));
  o.wn = wn;
  return o;
}

// ---------------------------------------------------------------------------
// Certified fast update (Ziv's rounding test: A. Ziv, "Fast evaluation of
// elementary mathematical functions with correctly rounded last bit", ACM
// TOMS 17(3), 1991).  The moments are computed exactly as above; the two
// square roots and three divisions of the weight update use the hardware
// approximations sqrt.approx{.ftz}.f32 and div.approx{.ftz}.f32 (CUDA
// documents at most 2 ulp for approximate division with divisors in
// [2^-126, 2^126]).
// With every approximate result assumed within 2^-19 relative of the
// correctly rounded one -- 8x the documented bound -- plus an absolute 2^-126
// for an operand or result flushed from the subnormal range, the fast weight
// wn' differs from the canonical wn by at most
//     eps = (|w u_m'| + |u_a'|) 2^-17 + (|w + w u_m'| + |wn'|) 2^-22 + 2^-96
// (computed in the looser form (|w u_m'| + |u_a'|)(2^-17 + 2^-20)
// + |w| 2^-21 (1 + 2^-20) + 2^-96, since |t| <= (|w| + |w u_m'|)(1 + 2^-24)
// and |wn'| <= (|t| + |u_a'|)(1 + 2^-24))
// (the relative errors propagate through the divisions, the clamp is
// 1-Lipschitz, each of the two final roundings adds at most one ulp, and the
// constants carry a further factor-of-two margin).  Flushing stays inside
// the 2^-96 term and the relative terms when eps >= 2^-28, c2 <= 2^14 and
// eta_m <= 4: a subnormal numerator of u_a or of n moves them by at most
// 2^-126 / eps <= 2^-98 (and w u_m by at most eta_m 2^-98); a subnormal
// nu or nu_e moves its denominator by at most c2 2^-63 <= 2^-21 eps; a
// flushed u_m moves w u_m by at most |w| 2^-126.  The host enables this path
// only under those conditions (cert_ok); divisors are checked in range here.  The caller stores the
// encoding of wn' only when encoding wn' - eps (rounded down) and wn' + eps
// (rounded up) gives the same code: every encoder here is monotone, so the
// canonical wn, which lies in between, has that code too.  Otherwise the
// element is recomputed with the exact sequence (madam_wn_exact).  Results
// are therefore identical to the canonical sequence bit for bit; the test
// only decides how much work that takes.
// ---------------------------------------------------------------------------
// FTZ selects the flushing forms.  Both forms are covered by the same bound
// (flushing is the larger error); every storage format uses the flushing
// forms, which take fewer instructions (the non-flushing ones also handle
// subnormal operands).
template <bool FTZ>
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  if (FTZ) asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  else asm("sqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
template <bool FTZ>
__device__ __forceinline__ float div_approx(float a, float b) {
  float q;
  if (FTZ) asm("div.approx.ftz.f32 %0, %1, %2;" : "=f"(q) : "f"(a), "f"(b));
  else asm("div.approx.f32 %0, %1, %2;" : "=f"(q) : "f"(a), "f"(b));
  return q;
}

struct CertUpd {
  float wn, lo, hi;  // fast weight and the interval holding the canonical one
  float e;           // the bound: lo = wn - e rounded down, hi = wn + e rounded up
  float m, v, ve;    // exact moments
  bool ok;           // divisors in the documented range and wn' finite
};

template <bool FTZ>
__device__ __forceinline__ CertUpd madam_update_cert(const StepScalars& s, float w, float g, float m, float v,
                                                     float ve) {
  CertUpd o;
  o.m = __fmaf_rn(s.b1, m, __fmul_rn(s.omb1, g));
  o.v = __fmaf_rn(s.b2, v, __fmul_rn(s.omb2, __fmul_rn(g, g)));
  const float ge = __fmul_rn(__fmul_rn(s.ln2, w), g);
  o.ve = __fmaf_rn(s.b2, ve, __fmul_rn(s.omb2, __fmul_rn(ge, ge)));
  const float den_a = __fmaf_rn(sqrt_approx<FTZ>(o.v), s.c2, s.eps);
  const float ua = div_approx<FTZ>(__fmul_rn(s.ka, o.m), den_a);
  const float den_e = __fmaf_rn(sqrt_approx<FTZ>(o.ve), s.c2, s.eps);
  const float n = div_approx<FTZ>(ge, den_e);
  const float rho = fmaxf(fabsf(w), s.tau);
  float um = div_approx<FTZ>(__fmul_rn(s.km, n), rho);
  um = fmaxf(s.lo, fminf(um, s.hi));
  const float t = __fmaf_rn(w, um, w);
  o.wn = __fadd_rn(t, ua);
  // eps with (|t| + |wn'|) 2^-22 <= (2 |w| + 2 |w u_m'| + |u_a'|)(1 + 2^-23) 2^-22
  // folded into the other two terms
  const float e = __fmaf_rn(__fadd_rn(fabsf(__fmul_rn(w, um)), fabsf(ua)), 8.58306884765625e-06f /* 2^-17 + 2^-20 */,
                            __fmaf_rn(fabsf(w), 4.768376129504759e-07f /* 2^-21 (1 + 2^-20) */,
                                      1.2621774483536189e-29f /* 2^-96 */));
  o.e = e;
  o.lo = __fsub_rd(o.wn, e);
  o.hi = __fadd_ru(o.wn, e);
  // The two denominators must stay below 2^125 (their lower bound eps >=
  // 2^-28 is checked on the host), and wn' must be finite.  The third divisor,
  // rho = max(|w|, tau) >= tau >= 2^-125, needs no upper check: when |w| >
  // 2^125 the canonical |w u_m| <= eta_m |n| <= 4 (1 - beta2)^(-1/2) <= 2^14
  // (nu_e' >= (1 - beta2) g_e^2 bounds |n|; eta_m <= 4 on the host) is far
  // below half an ulp of w, so w + w u_m rounds to w, as it does with the
  // approximate quotient (documented within 2 ulp up to 2^126 and 0 above).
  o.ok = fmaxf(den_a, den_e) <= 4.253529586511731e+37f /* 2^125 */ && fabsf(o.wn) < INFINITY;
  return o;
}

// The weight of the canonical sequence from the already updated (exact)
// moments: the exact fallback of the certified path.
static __device__ __noinline__ float madam_wn_exact(const StepScalars& s, float w, float g, float m1, float v1,
                                             float ve1) {
  const float ua = __fdiv_rn(__fmul_rn(s.ka, m1), __fmaf_rn(__fsqrt_rn(v1), s.c2, s.eps));
  const float ge = __fmul_rn(__fmul_rn(s.ln2, w), g);
  const float n = __fdiv_rn(ge, __fmaf_rn(__fsqrt_rn(ve1), s.c2, s.eps));
  float um = __fdiv_rn(__fmul_rn(s.km, n), fmaxf(fabsf(w), s.tau));
  um = fmaxf(s.lo, fminf(um, s.hi));
  return __fadd_rn(__fmaf_rn(w, um, w), ua);
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

// Stochastic BF16 of x given the complement of its 16 random bits (0xFFFF -
// R): the sum carries into the kept half exactly when R < (low half of x),
// i.e. with probability (low half) / 2^16.  The result is the high half.
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

// Eight E4M3 codes (bytes of r[0], r[1], lowest byte first) -> binary32.
// E4M3 -> FP16 -> FP32 are both widening conversions, so this is exact
// (NaN codes give NaN).
__device__ __forceinline__ void e4m3x8_to_f32(const uint32_t (&r)[2], float (&x)[8]) {
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    uint32_t h01, h23;
    asm("{\n .reg .b16 lo, hi;\n mov.b32 {lo, hi}, %2;\n"
        " cvt.rn.f16x2.e4m3x2 %0, lo;\n cvt.rn.f16x2.e4m3x2 %1, hi;\n}"
        : "=r"(h01), "=r"(h23)
        : "r"(r[i]));
    const float2 f01 = __half22float2(*reinterpret_cast<const __half2*>(&h01));
    const float2 f23 = __half22float2(*reinterpret_cast<const __half2*>(&h23));
    x[4 * i + 0] = f01.x;
    x[4 * i + 1] = f01.y;
    x[4 * i + 2] = f23.x;
    x[4 * i + 3] = f23.y;
  }
}

// Both ends of a bound interval (already scaled by 2^-e, outward rounded)
// encoded at once in the E4M3 normal range: code of the lower end, and
// whether the upper end has the same code.  Anything outside [2^-6, 448),
// or a sign change, reports `same` = false (the caller then takes the exact
// path, whose full encoder handles subnormals, saturation and NaN).
template <bool SR>
__device__ __forceinline__ uint32_t e4m3_pair_normal(float xlo, float xhi, uint32_t r, bool& same) {
  const uint32_t blo = __float_as_uint(xlo), bhi = __float_as_uint(xhi);
  const uint32_t alo = blo & 0x7FFFFFFFu, ahi = bhi & 0x7FFFFFFFu;
  uint32_t clo, chi;
  if (SR) {
    clo = (alo >> 20) + (r < (alo << 12) ? 1u : 0u);
    chi = (ahi >> 20) + (r < (ahi << 12) ? 1u : 0u);
  } else {  // nearest, ties to even: carry out of (rem + 0x7FFFF + lsb)
    clo = (alo >> 20) + (((alo & 0xFFFFFu) + 0x7FFFFu + ((alo >> 20) & 1u)) >> 20);
    chi = (ahi >> 20) + (((ahi & 0xFFFFFu) + 0x7FFFFu + ((ahi >> 20) & 1u)) >> 20);
  }
  same = clo == chi && ((blo ^ bhi) >> 31) == 0u && (alo - 0x3C800000u) < (0x43E00000u - 0x3C800000u) &&
         (ahi - 0x3C800000u) < (0x43E00000u - 0x3C800000u);
  return ((blo >> 24) & 0x80u) | (clo - 960u);
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
  const int32_t ef = static_cast<int32_t>(a_bits >> 23);
  int32_t k = -100;
  if (ef != 0) k = ef - 127 - 8 + ((a_bits & 0x7FFFFFu) > 0x600000u ? 1 : 0);
  return k < -100 ? -100 : (k > 100 ? 100 : k);
}

__device__ __forceinline__ float pow2f(int32_t e) {
  return __uint_as_float(static_cast<uint32_t>(e + 127) << 23);
}

// Block scales (FP16 bit patterns).  A scale written by the step is 2^k with
// k in [-24, 15]: every such power is an FP16 number (subnormal below 2^-14).
__device__ __forceinline__ uint32_t fp16_pow2_bits(int32_t k) {
  k = k < -24 ? -24 : (k > 15 ? 15 : k);
  return k >= -14 ? static_cast<uint32_t>(k + 15) << 10 : 1u << (k + 24);
}
// Value of a scale (exact widening conversion).
__device__ __forceinline__ float fp16_value(uint32_t h) {
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h)));
}
// Exponent of a scale: its exponent field minus the bias for normal scales,
// floor(log2) of its subnormal value otherwise (-24 for zero); the sign is
// ignored.  Exact for the powers of two the step writes.
__device__ __forceinline__ int32_t fp16_pow2_exponent(uint32_t h) {
  const int32_t e = static_cast<int32_t>((h >> 10) & 0x1Fu);
  if (e != 0) return e - 15;
  const int32_t k = 7 - __clz(static_cast<int32_t>(h & 0x3FFu));  // floor(log2 f) - 24
  return k < -24 ? -24 : k;
}
// Block scale of the next encode: the smallest k with A <= 448 * 2^k (A as
// binary32 bits, finite and >= 0), clamped to [-24, 15]; k_old when A = 0.
// Non-decreasing in A, which the certified path relies on.
__device__ __forceinline__ int32_t block_exponent(uint32_t a_bits, int32_t k_old) {
  if (a_bits == 0u) return k_old;
  const int32_t ef = static_cast<int32_t>(a_bits >> 23);
  int32_t k = -24;
  if (ef != 0) k = ef - 127 - 8 + ((a_bits & 0x7FFFFFu) > 0x600000u ? 1 : 0);
  return k < -24 ? -24 : (k > 15 ? 15 : k);
}

__device__ __forceinline__ bool aligned(const void* p, uintptr_t bytes) {
  return (reinterpret_cast<uintptr_t>(p) & (bytes - 1)) == 0;
}

// Bytes of a tile's slice of one array that the TMA stages: the largest
// multiple of 16 within the tile, or nothing when the array's base pointer is
// not 16-byte aligned (tile starts are then misaligned too).
__device__ __forceinline__ uint32_t staged_bytes(const void* base, int count, int esize) {
  return aligned(base, 16) ? (static_cast<uint32_t>(count * esize) & ~15u) : 0u;
}

// ---------------------------------------------------------------------------
// Group loads: 8 consecutive elements from shared memory (staged) or global.
// ---------------------------------------------------------------------------
template <bool RO>
__device__ __forceinline__ void get_bf16(float (&x)[8], bool staged, uint32_t saddr, const void* g,
                                         int64_t e0, int valid, bool vec) {
  if (staged || (vec && valid == kGroup)) {
    uint32_t r[4];
    if (staged) lds4(saddr, r);
    else if (RO) ld4_ro(static_cast<const uint16_t*>(g) + e0, r);
    else ld4(static_cast<const uint16_t*>(g) + e0, r);
#pragma unroll
    for (int i = 0; i < 4; ++i) { x[2 * i] = bf16_lo(r[i]); x[2 * i + 1] = bf16_hi(r[i]); }
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      x[j] = j < valid ? __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t*>(g)[e0 + j]) << 16)
                       : 0.0f;
  }
}

template <bool RO>
__device__ __forceinline__ void get_f32(float (&x)[8], bool staged, uint32_t saddr, const void* g,
                                        int64_t e0, int valid, bool vec) {
  if (staged) {
    uint32_t a[4], b[4];
    lds4(saddr, a);
    lds4(saddr + 16, b);
#pragma unroll
    for (int i = 0; i < 4; ++i) { x[i] = __uint_as_float(a[i]); x[4 + i] = __uint_as_float(b[i]); }
  } else if (vec && valid == kGroup) {
    uint32_t r[8];
    if (RO) ld8_ro(static_cast<const float*>(g) + e0, r);
    else ld8(static_cast<const float*>(g) + e0, r);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) x[j] = __uint_as_float(r[j]);
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j) x[j] = j < valid ? static_cast<const float*>(g)[e0 + j] : 0.0f;
  }
}

__device__ __forceinline__ void get_e4m3(float (&x)[8], bool staged, uint32_t saddr, const void* g,
                                         int64_t e0, int valid, bool vec, float scale) {
  if (staged || (vec && valid == kGroup)) {
    uint32_t r[2];
    if (staged) lds2(saddr, r);
    else ld2(static_cast<const uint8_t*>(g) + e0, r);
    e4m3x8_to_f32(r, x);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) x[j] = __fmul_rn(x[j], scale);
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      x[j] = j < valid ? __fmul_rn(e4m3_value(static_cast<const uint8_t*>(g)[e0 + j]), scale) : 0.0f;
  }
}

// Group stores (vector when whole and aligned, else element by element).
__device__ __forceinline__ void put_bf16(const uint32_t (&o)[4], void* g, int64_t e0, int valid, bool vec) {
  if (vec && valid == kGroup) {
    st4(static_cast<uint16_t*>(g) + e0, o);
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      if (j < valid)
        static_cast<uint16_t*>(g)[e0 + j] =
            static_cast<uint16_t>((j & 1) ? (o[j >> 1] >> 16) : (o[j >> 1] & 0xFFFFu));
  }
}
template <bool HINT = true>
__device__ __forceinline__ void put_f32(const float (&x)[8], void* g, int64_t e0, int valid, bool vec) {
  if (vec && valid == kGroup) {
    uint32_t o[8];
#pragma unroll
    for (int j = 0; j < kGroup; ++j) o[j] = __float_as_uint(x[j]);
    st8<HINT>(static_cast<float*>(g) + e0, o);
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      if (j < valid) static_cast<float*>(g)[e0 + j] = x[j];
  }
}
__device__ __forceinline__ void put_e4m3(const uint32_t (&o)[2], void* g, int64_t e0, int valid, bool vec) {
  if (vec && valid == kGroup) {
    st2(static_cast<uint8_t*>(g) + e0, o);
  } else {
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      if (j < valid) static_cast<uint8_t*>(g)[e0 + j] = static_cast<uint8_t>(o[j >> 2] >> (8 * (j & 3)));
  }
}

__host__ __device__ constexpr int esize_of(int dt) { return dt == kF32 ? 4 : (dt == kBF16 ? 2 : 1); }

// A tensor's table entries: from the kernel parameters when the launch
// carries them inline, else from global memory.
__device__ __forceinline__ TensorDesc desc_of(const StepArgs& a, int k) {
  return k < a.n_inline ? a.inl_desc[k] : a.desc[k];
}
__device__ __forceinline__ const void* grad_of(const StepArgs& a, int k) {
  return k < a.n_inline ? a.inl_grads[k] : a.grads[k];
}
__device__ __forceinline__ TensorAux aux_of(const StepArgs& a, int k) {
  return k < a.n_inline ? a.inl_aux[k] : a.aux[k];
}
// The tensor holding this CTA's first tile tb (which exists): scanned from
// the inline descriptors, else the host-computed table.
__device__ __forceinline__ int first_tensor(const StepArgs& a, int64_t tb) {
  if (a.n_inline == 0) return a.cta_first[blockIdx.x];
  int k = 0;
  while (k < a.n_inline - 1 && a.inl_desc[k].tile_off + (a.inl_desc[k].numel + kTile - 1) / kTile <= tb) ++k;
  return k;
}

// Per-tensor values the consumers keep while walking a tensor's tiles.
struct TensorCtx {
  TensorDesc d;
  const void* g;
  int64_t tiles;
  bool vec;            // all pointers aligned for vector access by whole groups
  bool fast;           // every array 16-byte aligned: whole warps of a tile are staged, stored with vector stores
  float dec_scale, enc_scale;
  float cc_scale;      // E4M3 per-tensor: 2^e of the new encode (compute copy)
  void* scale;         // kE4M3B (FP16) / kNVFP4 (E4M3) block scales
  uint16_t* cc;        // BF16 compute copy, or nullptr
  float gscale;        // kNVFP4 tensor scale
  float amax_seed;     // kE4M3: a lower bound of the tensor's largest exact |w'| of this step
};

template <int WD, int GD, int MD>
__device__ __forceinline__ void load_tensor(const StepArgs& a, int k, TensorCtx& c) {
  c.d = desc_of(a, k);
  c.g = grad_of(a, k);
  c.tiles = (c.d.numel + kTile - 1) / kTile;
  c.vec = aligned(c.d.w, WD == kBF16 ? 16 : (WD == kNVFP4 ? 4 : 8)) && aligned(c.g, GD == kF32 ? 32 : 16) &&
          aligned(c.d.m, MD == kF32 ? 32 : 16) && aligned(c.d.v, MD == kF32 ? 32 : 16) &&
          aligned(c.d.ve, MD == kF32 ? 32 : 16);
  c.fast = c.vec && aligned(c.d.w, 16) && aligned(c.g, 16) && aligned(c.d.m, 16) && aligned(c.d.v, 16) &&
           aligned(c.d.ve, 16);
  c.dec_scale = c.enc_scale = c.cc_scale = 1.0f;
  c.scale = nullptr;
  c.cc = nullptr;
  c.gscale = 1.0f;
  c.amax_seed = 0.0f;
  if (WD != kBF16 && a.aux) {  // the launch has aux entries (inline ones too, when it carries its tables)
    const TensorAux x = aux_of(a, k);
    c.scale = x.scale;
    c.cc = x.compute;
    c.gscale = x.gscale;
    // the compute copy joins the vector path only when 16-byte aligned;
    // block scales are staged (whole tiles: 240 bytes) only when 16-byte aligned
    if (c.cc && !aligned(c.cc, 16)) c.vec = c.fast = false;
    if ((WD == kE4M3B || WD == kNVFP4) && !aligned(c.scale, 16)) c.fast = false;
  }
}

// BF16 compute copy of eight stored E4M3 codes: code value x scale (a power
// of two, so exact), rounded to BF16 (exact as well inside BF16's range).
__device__ __forceinline__ void put_compute(const uint32_t (&codes)[2], float scale, void* cc, int64_t e0,
                                            int valid, bool vec) {
  float xd[8];
  e4m3x8_to_f32(codes, xd);
  uint32_t o[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) o[i] = bf16x2_rn(__fmul_rn(xd[2 * i], scale), __fmul_rn(xd[2 * i + 1], scale));
  put_bf16(o, cc, e0, valid, vec);
}

// Store the updated moments (BF16 moments nearest-even).
template <int MD, bool HINT = true>  // HINT: see st8
__device__ __forceinline__ void put_moments(const TensorCtx& x, int64_t e0, int valid, const float (&m)[8],
                                            const float (&v)[8], const float (&ve)[8]) {
  if (MD == kF32) {
    put_f32<HINT>(m, x.d.m, e0, valid, x.vec);
    put_f32<HINT>(v, x.d.v, e0, valid, x.vec);
    put_f32<HINT>(ve, x.d.ve, e0, valid, x.vec);
  } else {
    uint32_t om[4], ov[4], oe[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      om[i] = bf16x2_rn(m[2 * i], m[2 * i + 1]);
      ov[i] = bf16x2_rn(v[2 * i], v[2 * i + 1]);
      oe[i] = bf16x2_rn(ve[2 * i], ve[2 * i + 1]);
    }
    put_bf16(om, x.d.m, e0, valid, x.vec);
    put_bf16(ov, x.d.v, e0, valid, x.vec);
    put_bf16(oe, x.d.ve, e0, valid, x.vec);
  }
}

// Random bits of eight consecutive elements starting at global index gidx (a
// multiple of 8): 16-bit lanes (complemented, see bf16_sr_sum) for BF16
// storage, 32-bit lanes for E4M3 storage.
template <int WD>
__device__ __forceinline__ void group_random_bits(const StepArgs& a, uint64_t gidx, uint32_t (&rnd)[8]) {
  const uint64_t gi = gidx >> 3;  // global group index
  if (WD == kBF16) {
    const uint4 r = philox4x32_10(static_cast<uint32_t>(gi), static_cast<uint32_t>(gi >> 32), a.t_lo, a.t_hi,
                                  a.rk0, a.rk1);
    rnd[0] = ~r.x & 0xFFFFu; rnd[1] = ~r.x >> 16;
    rnd[2] = ~r.y & 0xFFFFu; rnd[3] = ~r.y >> 16;
    rnd[4] = ~r.z & 0xFFFFu; rnd[5] = ~r.z >> 16;
    rnd[6] = ~r.w & 0xFFFFu; rnd[7] = ~r.w >> 16;
  } else {
    const uint64_t b0 = 2ull * gi, b1 = b0 + 1ull;
    const uint4 r0 = philox4x32_10(static_cast<uint32_t>(b0), static_cast<uint32_t>(b0 >> 32), a.t_lo, a.t_hi,
                                   a.rk0, a.rk1);
    const uint4 r1 = philox4x32_10(static_cast<uint32_t>(b1), static_cast<uint32_t>(b1 >> 32), a.t_lo, a.t_hi,
                                   a.rk0, a.rk1);
    rnd[0] = r0.x; rnd[1] = r0.y; rnd[2] = r0.z; rnd[3] = r0.w;
    rnd[4] = r1.x; rnd[5] = r1.y; rnd[6] = r1.z; rnd[7] = r1.w;
  }
}

// The canonical weight of slot j of consumer c (a runtime index), from the
// original inputs in the stage at st (BF16 weights); the stage must still be
// allocated.
template <int GD, int MD>
__device__ __forceinline__ float exact_wn_from_stage(const StepArgs& a, uint32_t st, int c, int j) {
  constexpr int GS = esize_of(GD), MS = esize_of(MD);
  const uint32_t i = static_cast<uint32_t>(kGroup * c + j);
  const float w = __uint_as_float(lds_u16(st + 2u * i) << 16);
  auto ld = [&](uint32_t base, int es) -> float {
    return es == 4 ? __uint_as_float(lds_u32(base + 4u * i)) : __uint_as_float(lds_u16(base + 2u * i) << 16);
  };
  return madam_update<false>(a.s, w, ld(st + a.off_g, GS), ld(st + a.off_m, MS), ld(st + a.off_v, MS),
                             ld(st + a.off_ve, MS)).wn;
}

// The complemented 16-bit random lane of BF16 element j (a runtime index) of
// the group starting at global index gidx, as group_random_bits draws it.
__device__ __forceinline__ uint32_t bf16_element_random_bits(const StepArgs& a, uint64_t gidx, int j) {
  const uint64_t gi = gidx >> 3;
  const uint4 r = philox4x32_10(static_cast<uint32_t>(gi), static_cast<uint32_t>(gi >> 32), a.t_lo, a.t_hi,
                                a.rk0, a.rk1);
  const int q = j >> 1;
  const uint32_t wd = q == 0 ? r.x : (q == 1 ? r.y : (q == 2 ? r.z : r.w));
  return (j & 1) ? (~wd >> 16) : (~wd & 0xFFFFu);
}

// Update 8 loaded elements and store them (vector stores when `vec` and
// whole, else element by element).  STAGED (BF16 weights, whole staged
// tiles): the stage at st stays allocated until this returns, and the
// certified path's rare exact branch takes the undecided elements one at a
// time from there (c: the consumer), in a loop over the set bits.  Otherwise
// that branch uses the inputs held in registers.  (Measured on the 7B list:
// keeping the inputs live through the certified loop for the exact branch,
// 18.64 ms per step; this, 18.27 ms.  Reloading them from global memory was
// slower still, 21.6 ms: about a tenth of the warps' groups take the branch,
// and each reload waits on DRAM while the other warps wait for its stage.)
template <int WD, int GD, int MD, bool SR, bool OPT, bool STAGED>
__device__ __forceinline__ void finish_group(const StepArgs& a, const TensorCtx& x, int64_t e0, int valid,
                                             float (&w)[8], float (&g)[8], float (&m)[8], float (&v)[8],
                                             float (&ve)[8], uint32_t& amax_bits, uint32_t st, int c) {
  // random bits: one Philox block per 8 BF16 lanes, two per 8 E4M3 lanes
  uint32_t rnd[8];
  if (SR) group_random_bits<WD>(a, static_cast<uint64_t>(x.d.goff + e0), rnd);

  if (WD == kBF16 && !OPT && a.s.cert_ok) {  // certified fast path (see madam_update_cert)
    uint32_t ow[4] = {0u, 0u, 0u, 0u};
    uint32_t redo = 0u;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const CertUpd u = madam_update_cert<true>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      bool same;
      uint32_t code;
      if (SR) {
        const uint32_t slo = __float_as_uint(u.lo) + rnd[j], shi = __float_as_uint(u.hi) + rnd[j];
        same = ((slo ^ shi) >> 16) == 0u;
        code = slo >> 16;
      } else {
        const uint32_t pair = bf16x2_rn(u.lo, u.hi);
        same = ((pair ^ (pair >> 16)) & 0xFFFFu) == 0u;
        code = pair & 0xFFFFu;
      }
      ow[j >> 1] |= code << (16 * (j & 1));
      if (!(u.ok && same)) redo |= 1u << j;
      m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
    }
    if (redo) {  // rare: encode the canonical weight of the undecided elements
      if constexpr (STAGED) {
#pragma unroll 1
        for (uint32_t rm = redo; rm != 0u; rm &= rm - 1u) {
          const int j = __ffs(rm) - 1;
          const float xe = exact_wn_from_stage<GD, MD>(a, st, c, j);
          const uint32_t code =
              SR ? (bf16_sr_sum(xe, bf16_element_random_bits(a, static_cast<uint64_t>(x.d.goff + e0), j)) >> 16)
                 : (bf16x2_rn(xe, xe) & 0xFFFFu);
          const int sh = 16 * (j & 1);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            if (i == (j >> 1)) ow[i] = (ow[i] & ~(0xFFFFu << sh)) | (code << sh);
        }
      } else {
#pragma unroll
        for (int j = 0; j < kGroup; ++j) {
          if ((redo >> j) & 1u) {
            const float xe = madam_wn_exact(a.s, w[j], g[j], m[j], v[j], ve[j]);
            const uint32_t code = SR ? (bf16_sr_sum(xe, rnd[j]) >> 16) : (bf16x2_rn(xe, xe) & 0xFFFFu);
            const int sh = 16 * (j & 1);
            ow[j >> 1] = (ow[j >> 1] & ~(0xFFFFu << sh)) | (code << sh);
          }
        }
      }
    }
    put_bf16(ow, x.d.w, e0, valid, x.vec);
  } else if (WD == kE4M3 && !OPT && a.s.cert_ok) {
    // Certified fast path for E4M3: both ends of the bound are scaled by 2^-e
    // with outward rounding and encoded; the largest |w'| must be exact, so an
    // element whose bound reaches the threshold is recomputed as well.  The
    // threshold is the larger of this thread's running maximum and the
    // tensor's maximum flushed so far in this step: both are exact |w'| of
    // elements of this tensor, so no element below them can be the maximum.
    uint32_t ow[2] = {0u, 0u};
    uint32_t redo = 0u;
    const float amax_f = fmaxf(__uint_as_float(amax_bits), x.amax_seed);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const CertUpd u = madam_update_cert<true>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      bool same;
      const uint32_t code = e4m3_pair_normal<SR>(__fmul_rd(u.lo, x.enc_scale), __fmul_ru(u.hi, x.enc_scale),
                                                 SR ? rnd[j] : 0u, same);
      // an undecided element's code may be out of range (it is replaced
      // below): keep it inside its own byte
      ow[j >> 2] |= (code & 0xFFu) << (8 * (j & 3));
      if (!(u.ok && same) || fmaxf(fabsf(u.lo), fabsf(u.hi)) >= amax_f) redo |= 1u << j;
      m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
    }
    if (redo) {  // rare: the canonical weight of undecided elements and maximum candidates
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        if ((redo >> j) & 1u) {
          const float xe = madam_wn_exact(a.s, w[j], g[j], m[j], v[j], ve[j]);
          const uint32_t wb = __float_as_uint(xe) & 0x7FFFFFFFu;
          if (j < valid && wb < 0x7F800000u) amax_bits = max(amax_bits, wb);
          const uint32_t code = e4m3_encode<SR>(__fmul_rn(xe, x.enc_scale), SR ? rnd[j] : 0u);
          const int sh = 8 * (j & 3);
          ow[j >> 2] = (ow[j >> 2] & ~(0xFFu << sh)) | (code << sh);
        }
      }
    }
    put_e4m3(ow, x.d.w, e0, valid, x.vec);
    if (x.cc) put_compute(ow, x.cc_scale, x.cc, e0, valid, x.vec);
  } else {
  float wn[8];
#pragma unroll
  for (int j = 0; j < kGroup; ++j) {
    const Upd u = madam_update<OPT>(a.s, w[j], g[j], m[j], v[j], ve[j]);
    wn[j] = u.wn; m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
  }

  if (WD == kBF16) {
    uint32_t ow[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (SR) ow[i] = __byte_perm(bf16_sr_sum(wn[2 * i], rnd[2 * i]), bf16_sr_sum(wn[2 * i + 1], rnd[2 * i + 1]), 0x7632);
      else ow[i] = bf16x2_rn(wn[2 * i], wn[2 * i + 1]);
    }
    put_bf16(ow, x.d.w, e0, valid, x.vec);
  } else {
    uint32_t ow[2] = {0u, 0u};
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const uint32_t wb = __float_as_uint(wn[j]) & 0x7FFFFFFFu;
      if (j < valid && wb < 0x7F800000u) amax_bits = max(amax_bits, wb);
      ow[j >> 2] |= e4m3_encode<SR>(__fmul_rn(wn[j], x.enc_scale), SR ? rnd[j] : 0u) << (8 * (j & 3));
    }
    put_e4m3(ow, x.d.w, e0, valid, x.vec);
    if (x.cc) put_compute(ow, x.cc_scale, x.cc, e0, valid, x.vec);
  }
  }
  put_moments<MD>(x, e0, valid, m, v, ve);
}

// One group of a partial tile, or of a tensor whose arrays are not all staged
// or aligned: loads each array from the stage when its bytes were staged, else
// from global memory.  The running E4M3 maximum goes in and comes back by
// value: a reference would pin the caller's copy to local memory.
template <int WD, int GD, int MD, bool SR, bool OPT>
__device__ __forceinline__ uint32_t general_group(const StepArgs& a, const TensorCtx& x, int64_t tile_e0,
                                                  int count, int c, uint32_t st, uint32_t amax_bits) {
  constexpr int WS = esize_of(WD), GS = esize_of(GD), MS = esize_of(MD);
  if (kGroup * c >= count) return amax_bits;
  const int valid = count - kGroup * c < kGroup ? count - kGroup * c : kGroup;
  const int64_t e0 = tile_e0 + kGroup * c;
  const uint32_t end = static_cast<uint32_t>(kGroup * (c + 1));  // elements through this group
  float w[8], g[8], m[8], v[8], ve[8];
  if (WD == kBF16)
    get_bf16<false>(w, end * WS <= staged_bytes(x.d.w, count, WS), st + kGroup * WS * c, x.d.w, e0, valid, x.vec);
  else
    get_e4m3(w, end * WS <= staged_bytes(x.d.w, count, WS), st + kGroup * WS * c, x.d.w, e0, valid, x.vec,
             x.dec_scale);
  const bool g_st = end * GS <= staged_bytes(x.g, count, GS);
  if (GD == kF32) get_f32<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  else get_bf16<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  const bool m_st = end * MS <= staged_bytes(x.d.m, count, MS);
  const bool v_st = end * MS <= staged_bytes(x.d.v, count, MS);
  const bool e_st = end * MS <= staged_bytes(x.d.ve, count, MS);
  if (MD == kF32) {
    get_f32<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_f32<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_f32<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  } else {
    get_bf16<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_bf16<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_bf16<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  }
  finish_group<WD, GD, MD, SR, OPT, false>(a, x, e0, valid, w, g, m, v, ve, amax_bits, st, c);
  return amax_bits;
}

// The same, as a call.  Which form a kernel instance uses was measured per
// moment format.  Called, the group costs the caller a stack frame (the live
// state saved around the call), and on a short launch after an L2 flush those
// first local-memory accesses wait on DRAM: a 1 Mi-element list with
// binary32 moments ran 15.9-17.1 us called against 13.0-13.1 us inline, and
// GPT-2, the ragged list and the 1.5B list ran 0.7-1.1 % faster inline.  With
// BF16 moments the inline form slowed the whole-tile loop instead: the 7B list
// took 18.44 ms per step against 18.21 ms called (three runs each).
template <int WD, int GD, int MD, bool SR, bool OPT>
__device__ __noinline__ uint32_t general_group_call(const StepArgs& a, const TensorCtx& x, int64_t tile_e0,
                                                    int count, int c, uint32_t st, uint32_t amax_bits) {
  return general_group<WD, GD, MD, SR, OPT>(a, x, tile_e0, count, c, st, amax_bits);
}

// ---------------------------------------------------------------------------
// Block-scaled E4M3 weights: the four threads of a quad hold one 32-element
// block (8 elements each).  The stored codes decode with the block's old
// scale; the block's new scale 2^k comes from the largest finite |w'| of the
// block (current scaling); the codes re-encode x = w' 2^-k.  Every lane of the
// warp must call this (the block maximum is a quad shuffle); elements j >=
// valid are padding (valid may be 0) and neither count nor get stored.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t quad_max(uint32_t x) {
  x = max(x, __shfl_xor_sync(0xFFFFFFFFu, x, 1));
  return max(x, __shfl_xor_sync(0xFFFFFFFFu, x, 2));
}

template <int GD, int MD, bool SR, bool OPT>
__device__ __forceinline__ void finish_block(const StepArgs& a, const TensorCtx& x, int64_t e0, int valid,
                                             uint32_t h_old, float (&w)[8], float (&g)[8], float (&m)[8],
                                             float (&v)[8], float (&ve)[8]) {
  uint32_t rnd[8];
  if (SR) group_random_bits<kE4M3B>(a, static_cast<uint64_t>(x.d.goff + e0), rnd);
  const int32_t k_old = fp16_pow2_exponent(h_old);
  const uint32_t vmask = valid >= kGroup ? 0xFFu : (valid > 0 ? (1u << valid) - 1u : 0u);
  uint32_t code[8];
  int32_t k_new;
  if (!OPT && a.s.cert_ok) {
    // Certified path (see madam_update_cert).  Keep the fast weights and the
    // thread's largest error bound et; the block maximum then lies in
    // [max |w'| - et, max |w'| + et] (outward rounded).  When both ends give
    // the same exponent (block_exponent is monotone) that is the exact one;
    // otherwise the quad computes its exact maximum.  Each element's code is
    // then taken from its interval [w' - et, w' + et] under the new scale
    // where both ends agree, else from the exact weight.
    float wf[8];
    float et = 0.0f, am = 0.0f;
    uint32_t bad = 0u;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const CertUpd u = madam_update_cert<true>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      wf[j] = u.wn;
      m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
      if (!u.ok) {
        bad |= 1u << j;
      } else {
        et = fmaxf(et, u.e);
        if ((vmask >> j) & 1u) am = fmaxf(am, fabsf(u.wn));
      }
    }
    bad &= vmask;
    const float lo_t = bad ? 0.0f : fmaxf(__fsub_rd(am, et), 0.0f);
    const float hi_t = bad ? INFINITY : __fadd_ru(am, et);
    const uint32_t qlo = quad_max(__float_as_uint(lo_t));  // non-negative floats order as their bits
    const uint32_t qhi = quad_max(__float_as_uint(hi_t));
    const int32_t kl = block_exponent(qlo, k_old);
    const bool certain = qlo != 0u && qhi < 0x7E800000u /* 2^126 */ && kl == block_exponent(qhi, k_old);
    k_new = kl;
    if (__any_sync(0xFFFFFFFFu, !certain)) {  // exact block maximum for the undecided quads
      uint32_t amx = 0u;
      if (!certain) {
#pragma unroll
        for (int j = 0; j < kGroup; ++j) {
          if ((vmask >> j) & 1u) {
            const uint32_t b = __float_as_uint(madam_wn_exact(a.s, w[j], g[j], m[j], v[j], ve[j])) & 0x7FFFFFFFu;
            if (b < 0x7F800000u) amx = max(amx, b);
          }
        }
      }
      amx = quad_max(amx);
      if (!certain) k_new = block_exponent(amx, k_old);
    }
    const float enc = pow2f(-k_new);
    uint32_t redo = bad;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      bool same;
      code[j] = e4m3_pair_normal<SR>(__fmul_rd(__fsub_rd(wf[j], et), enc), __fmul_ru(__fadd_ru(wf[j], et), enc),
                                     SR ? rnd[j] : 0u, same);
      if (!same) redo |= 1u << j;
    }
    redo &= vmask;
    if (redo) {  // rare: the canonical weight of the undecided elements
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        if ((redo >> j) & 1u) {
          const float xe = madam_wn_exact(a.s, w[j], g[j], m[j], v[j], ve[j]);
          code[j] = e4m3_encode<SR>(__fmul_rn(xe, enc), SR ? rnd[j] : 0u);
        }
      }
    }
  } else {
    float wn[8];
    uint32_t amx = 0u;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const Upd u = madam_update<OPT>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      wn[j] = u.wn; m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
      const uint32_t b = __float_as_uint(u.wn) & 0x7FFFFFFFu;
      if (((vmask >> j) & 1u) && b < 0x7F800000u) amx = max(amx, b);
    }
    k_new = block_exponent(quad_max(amx), k_old);
    const float enc = pow2f(-k_new);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) code[j] = e4m3_encode<SR>(__fmul_rn(wn[j], enc), SR ? rnd[j] : 0u);
  }
  uint32_t ow[2];
  ow[0] = code[0] | (code[1] << 8) | (code[2] << 16) | (code[3] << 24);
  ow[1] = code[4] | (code[5] << 8) | (code[6] << 16) | (code[7] << 24);
  put_e4m3(ow, x.d.w, e0, valid, x.vec);
  const uint32_t h_new = fp16_pow2_bits(k_new);
  if ((threadIdx.x & 3) == 0 && valid > 0) static_cast<uint16_t*>(x.scale)[e0 / kBlock] = static_cast<uint16_t>(h_new);
  if (x.cc) put_compute(ow, fp16_value(h_new), x.cc, e0, valid, x.vec);
  put_moments<MD>(x, e0, valid, m, v, ve);
}

// One group of a partial tile, or of a tensor whose arrays are not all
// staged: every consumer lane calls this (lanes past the tile's end with no
// elements), loading each array from the stage when its bytes were staged,
// else from global memory.
template <int GD, int MD, bool SR, bool OPT>
__device__ __forceinline__ void general_block_group(const StepArgs& a, const TensorCtx& x, int64_t tile_e0, int count,
                                                 int c, uint32_t st) {
  constexpr int GS = esize_of(GD), MS = esize_of(MD);
  const int rem = count - kGroup * c;
  const int valid = rem < 0 ? 0 : (rem < kGroup ? rem : kGroup);
  const int64_t e0 = tile_e0 + kGroup * c;
  const uint32_t end = static_cast<uint32_t>(kGroup * (c + 1));  // elements through this group
  // the block's old scale: staged when the tile's scale bytes through this block were
  const int nblk = (count + kBlock - 1) / kBlock, b = c >> 2;
  uint32_t h = 0u;
  const uint16_t* sc = static_cast<const uint16_t*>(x.scale);
  if (static_cast<uint32_t>(2 * (b + 1)) <= staged_bytes(sc + tile_e0 / kBlock, nblk, 2))
    h = lds_u16(st + a.off_s + 2 * b);
  else if (b < nblk)
    h = sc[(tile_e0 / kBlock) + b];
  float w[8], g[8], m[8], v[8], ve[8];
  get_e4m3(w, end <= staged_bytes(x.d.w, count, 1), st + kGroup * c, x.d.w, e0, valid, x.vec, fp16_value(h));
  const bool g_st = end * GS <= staged_bytes(x.g, count, GS);
  if (GD == kF32) get_f32<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  else get_bf16<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  const bool m_st = end * MS <= staged_bytes(x.d.m, count, MS);
  const bool v_st = end * MS <= staged_bytes(x.d.v, count, MS);
  const bool e_st = end * MS <= staged_bytes(x.d.ve, count, MS);
  if (MD == kF32) {
    get_f32<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_f32<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_f32<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  } else {
    get_bf16<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_bf16<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_bf16<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  }
  finish_block<GD, MD, SR, OPT>(a, x, e0, valid, h, w, g, m, v, ve);
}

// The same, as a call: with BF16 moments, as for general_group_call.  Inline,
// the FP8-regime list (block-scaled linears, binary32 moments) ran 6.02 ms per
// step against 6.08 ms called.
template <int GD, int MD, bool SR, bool OPT>
__device__ __noinline__ void general_block_group_call(const StepArgs& a, const TensorCtx& x, int64_t tile_e0, int count,
                                             int c, uint32_t st) {
  general_block_group<GD, MD, SR, OPT>(a, x, tile_e0, count, c, st);
}

// ---------------------------------------------------------------------------
// NVFP4 weights: E2M1 codes (OCP FP4: sign, 2 exponent bits with bias 1, one
// mantissa bit; +-{0, 0.5, 1, 1.5, 2, 3, 4, 6}), an E4M3 scale s per 16
// elements and a binary32 tensor scale G.  A weight decodes as q * d with
// d = s * G (both products rounded to binary32); a step re-encodes
// x = w' / d' (correctly rounded) under the block's new scale.  The two
// threads of a pair (lanes 2p, 2p+1) hold one block.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float e2m1_value(uint32_t c) {
  const uint32_t mag = c & 7u;
  const uint32_t b = mag >= 2u ? ((((mag >> 1) + 126u) << 23) | ((mag & 1u) << 22)) : (mag ? 0x3F000000u : 0u);
  return __uint_as_float(b | ((c & 8u) << 28));
}

// binary32 -> E2M1 code: nearest-even, or stochastic (away from zero iff
// r < floor(fraction * 2^32)); |x| >= 6 and infinities saturate; NaN -> +0.
// Branch-free: with the grid spacing sp = 0.5, 1 or 2 of |x|'s binade
// ([0, 2), [2, 4), [4, 6]), q = |x| / sp (a product with the power of two
// 1 / sp: exact), its integer part k and fraction f give the code
// k + (0, 2 or 4) and the step up.
template <bool SR>
__device__ __forceinline__ uint32_t e2m1_encode(float x, uint32_t r) {
  const float a = fminf(fabsf(x), 6.0f);
  const float rsp = a < 2.0f ? 2.0f : (a < 4.0f ? 1.0f : 0.5f);
  const uint32_t off = a < 2.0f ? 0u : (a < 4.0f ? 2u : 4u);
  const float q = __fmul_rn(a, rsp);
  const float kf = truncf(q);
  const float f = __fsub_rn(q, kf);  // exact
  const uint32_t k = __float2uint_rz(kf);
  uint32_t up;
  if (SR) up = r < __float2uint_rz(__fmul_rn(f, 4294967296.0f)) ? 1u : 0u;
  else up = (f > 0.5f || (f == 0.5f && (k & 1u))) ? 1u : 0u;
  const uint32_t code = ((__float_as_uint(x) >> 28) & 8u) | (k + off + up);
  return x != x ? 0u : code;
}

// Eight packed E2M1 codes (element j in bits [4j, 4j + 4)) -> binary32, with
// the hardware E2M1 -> FP16 conversion (exact) and FP16 -> binary32.
__device__ __forceinline__ void e2m1x8_to_f32(uint32_t packed, float (&x)[8]) {
  uint32_t h[4];
  asm("{\n .reg .b8 b0, b1, b2, b3;\n mov.b32 {b0, b1, b2, b3}, %4;\n"
      " cvt.rn.f16x2.e2m1x2 %0, b0;\n cvt.rn.f16x2.e2m1x2 %1, b1;\n"
      " cvt.rn.f16x2.e2m1x2 %2, b2;\n cvt.rn.f16x2.e2m1x2 %3, b3;\n}"
      : "=r"(h[0]), "=r"(h[1]), "=r"(h[2]), "=r"(h[3])
      : "r"(packed));
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&h[i]));
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}

// Eight binary32 -> packed E2M1 codes, nearest-even with saturation at +-6
// (the hardware conversion; used only on finite values).
// Two binary32 -> two E2M1 codes, nearest-even (hardware conversion; x0 in
// the low nibble).
__device__ __forceinline__ uint32_t e2m1x2_rn(float x0, float x1) {
  uint32_t p;
  asm("{\n .reg .b8 b;\n cvt.rn.satfinite.e2m1x2.f32 b, %2, %1;\n cvt.u32.u8 %0, b;\n}"
      : "=r"(p)
      : "f"(x0), "f"(x1));
  return p;
}

// Stochastic E2M1 code shared by every value of an interval of magnitudes
// [xm, xM] (sign: that of q), decided from its smaller end xm alone, given
// lim = 2^32 - W with W >= 2 (xM - xm) 2^32 + 1.  In xm's binade the grid
// position is Q = |x| rsp (rsp = 2, 1, 1/2 on [0, 2), [2, 4), [4, 6]; 6 and
// above saturate at Q = 3), exact in binary32; with k its integer part and
// F = floor(frac(Q) 2^32), the code is off + k + [r < F].  Every binade edge
// and the saturation point lie at an integer Q of xm's scale, and Q 2^32
// grows by less than W over the interval (slope rsp <= 2); so when F + W and
// ((F + 2^32 - 1 - r) mod 2^32) + W both stay below 2^32, no value of the
// interval crosses a step or changes its rounding decision (same = true).
// xm <= 0 or NaN (an interval reaching zero) reports false.
__device__ __forceinline__ uint32_t e2m1_sr_interval(float xm, float q, uint32_t r, uint32_t lim, bool& same) {
  const float am = fminf(xm, 6.0f);
  const float rsp = am < 2.0f ? 2.0f : (am < 4.0f ? 1.0f : 0.5f);
  const uint32_t off = am < 2.0f ? 0u : (am < 4.0f ? 2u : 4u);
  const float qq = __fmul_rn(am, rsp);  // exact (a power of two)
  const float kf = truncf(qq);
  const uint32_t F = __float2uint_rz(__fmul_rn(__fsub_rn(qq, kf), 4294967296.0f));  // exact
  const uint32_t sl = F + ~r;
  same = xm > 0.0f && max(F, sl) < lim;
  return ((__float_as_uint(q) >> 28) & 8u) | (__float2uint_rz(kf) + off + (r < F ? 1u : 0u));
}

// A block scale code with the two products its covering test and the encode
// use: d = fl(v(c) G) (the block's step) and p = fl(6 d) (the largest
// magnitude the code covers: c covers A iff p >= A).
struct Fp4Code {
  uint32_t c;
  float d, p;
};

// Value of a positive finite E4M3 code (1..126) through the hardware widening
// conversion (exact: every E4M3 value is an FP16 value).
__device__ __forceinline__ float e4m3_value_cvt(uint32_t c) {
  uint32_t h;
  asm("{\n .reg .b16 lo;\n cvt.u16.u32 lo, %1;\n cvt.rn.f16x2.e4m3x2 %0, lo;\n}" : "=r"(h) : "r"(c & 0xFFu));
  return __half2float(__ushort_as_half(static_cast<unsigned short>(h & 0xFFFFu)));
}

// c in [1, 126]
__device__ __forceinline__ Fp4Code fp4_code(uint32_t c, float G) {
  Fp4Code r;
  r.c = c;
  r.d = __fmul_rn(e4m3_value_cvt(c), G);
  r.p = __fmul_rn(6.0f, r.d);
  return r;
}

// Block scale code of the next encode: the smallest code in [1, 126] that
// covers A (finite, >= 0), 126 when none does, c_old when A = 0.  Covering is
// monotone in the code, so c is that code iff c covers A and c - 1 does not
// (or c = 1).  The candidate is A / (6 G) rounded up onto the E4M3 grid;
// both tests run side by side, and only a candidate that fails them (an
// estimate within rounding of a grid point, or a step d out of the normal
// range) walks to the answer one code at a time.
static __device__ __noinline__ Fp4Code nvfp4_scale_code_walk(float A, float G, int32_t c) {
  for (int i = 0; i < 126 && c > 1 && fp4_code(static_cast<uint32_t>(c - 1), G).p >= A; ++i) --c;
  for (int i = 0; i < 126 && c < 126 && !(fp4_code(static_cast<uint32_t>(c), G).p >= A); ++i) ++c;
  return fp4_code(static_cast<uint32_t>(c), G);
}

__device__ __forceinline__ Fp4Code nvfp4_scale_code(float A, float G, uint32_t c_old) {
  if (!(A > 0.0f)) {  // the old code, whatever it holds (zero, NaN, a sign)
    Fp4Code r;
    r.c = c_old;
    r.d = __fmul_rn(e4m3_value(c_old), G);
    r.p = __fmul_rn(6.0f, r.d);
    return r;
  }
  const float est = div_approx<false>(A, __fmul_rn(6.0f, G));
  int32_t c = static_cast<int32_t>(e4m3_encode<true>(est, 0u) & 0x7Fu);  // random bits 0: rounds up
  c = c < 1 ? 1 : (c > 126 ? 126 : c);
  const Fp4Code hi = fp4_code(static_cast<uint32_t>(c), G);
  const float p_lo = c > 1 ? fp4_code(static_cast<uint32_t>(c - 1), G).p : 0.0f;
  if (hi.p >= A && (c == 1 || !(p_lo >= A))) return hi;
  return nvfp4_scale_code_walk(A, G, c);
}

// Eight packed codes (element j in bits [4j, 4j + 4)) -> the group's bytes.
__device__ __forceinline__ void put_fp4(uint32_t packed, void* w, int64_t e0, int valid, bool vec) {
  uint8_t* p = static_cast<uint8_t*>(w) + e0 / 2;
  if (vec && valid == kGroup) {
    asm volatile("st.global.L1::no_allocate.u32 [%0], %1;" ::"l"(p), "r"(packed) : "memory");
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (2 * k < valid) {
        uint32_t byte = (packed >> (8 * k)) & 0xFFu;
        if (2 * k + 1 >= valid) byte &= 0x0Fu;  // past the tensor's end: the spare nibble is 0
        p[k] = static_cast<uint8_t>(byte);
      }
    }
  }
}

__device__ __forceinline__ uint32_t pair_max(uint32_t x) {
  return max(x, __shfl_xor_sync(0xFFFFFFFFu, x, 1));
}

// One element's canonical update recomputed from the stage's original
// inputs (kept until the group is done): the exact weight of the element's
// group slot j.
template <int GD, int MD>
__device__ __forceinline__ float fp4_exact_from_stage(const StepArgs& a, uint32_t st, int c, int j, float d_old) {
  constexpr int GS = esize_of(GD), MS = esize_of(MD);
  const uint32_t word = lds_u32(st + 4 * c);
  float q[8];
  e2m1x8_to_f32(word, q);
  const float w = __fmul_rn(q[j], d_old);
  auto ld = [&](uint32_t base, int es) -> float {
    const uint32_t addr = base + static_cast<uint32_t>(kGroup * es * c + es * j);
    return es == 4 ? __uint_as_float(lds_u32(addr)) : __uint_as_float(lds_u16(addr) << 16);
  };
  const float g = ld(st + a.off_g, GS);
  const float m = ld(st + a.off_m, MS), v = ld(st + a.off_v, MS), ve = ld(st + a.off_ve, MS);
  return madam_update<false>(a.s, w, g, m, v, ve).wn;
}

// One element's canonical weight recomputed from global memory after the
// stage has been released: its code (this thread overwrites it only once the
// group is done), its gradient, and the binary32 moments this thread stored
// right after the update.  Those are the values the canonical sequence feeds
// into the weight update, so this serves binary32 moments only (BF16 moments
// are stored rounded).  L2-only loads: the moments were written by this
// thread.  Out of line: the call is rare and its pointers would otherwise stay
// live through the encode.
template <int GD>
__device__ __noinline__ float fp4_exact_from_global(const StepArgs& a, const TensorCtx& x, int64_t e,
                                                    float d_old) {
  const uint8_t* pw = static_cast<const uint8_t*>(x.d.w) + (e >> 1);
  uint32_t byte, bg, bm, bv, be;
  asm volatile("ld.global.cg.u8 %0, [%1];" : "=r"(byte) : "l"(pw) : "memory");
  const float w = __fmul_rn(e2m1_value((e & 1) ? (byte >> 4) : (byte & 0xFu)), d_old);
  if (GD == kF32) {
    asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(bg) : "l"(static_cast<const float*>(x.g) + e) : "memory");
  } else {
    asm volatile("ld.global.cg.u16 %0, [%1];" : "=r"(bg) : "l"(static_cast<const uint16_t*>(x.g) + e) : "memory");
    bg <<= 16;
  }
  asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(bm) : "l"(static_cast<const float*>(x.d.m) + e) : "memory");
  asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(bv) : "l"(static_cast<const float*>(x.d.v) + e) : "memory");
  asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(be) : "l"(static_cast<const float*>(x.d.ve) + e) : "memory");
  return madam_wn_exact(a.s, w, __uint_as_float(bg), __uint_as_float(bm), __uint_as_float(bv), __uint_as_float(be));
}

// Where the rare exact branch of finish_fp4 finds an element's inputs:
// kExactRegs -- still in registers (the moments are stored at the end);
// kExactStage -- in the stage at `st` (thread c), kept until the group is done;
// kExactGlobal -- in global memory (binary32 moments only; the stage has
// already been released).  The last two store the new moments right after
// the update, so fewer values live in registers through the encode.
constexpr int kExactRegs = 0, kExactStage = 1, kExactGlobal = 2;

template <int GD, int MD, bool SR, bool OPT, int SRC>
__device__ __forceinline__ void finish_fp4(const StepArgs& a, const TensorCtx& x, int64_t e0, int valid,
                                           uint32_t c_old, float (&w)[8], float (&g)[8], float (&m)[8],
                                           float (&v)[8], float (&ve)[8], uint32_t st, int c) {
  const float G = x.gscale;
  const float d_old = __fmul_rn(e4m3_value(c_old), G);
  const uint64_t gi = static_cast<uint64_t>(x.d.goff + e0) >> 3;  // global group index (random lanes)
  const uint32_t vmask = valid >= kGroup ? 0xFFu : (valid > 0 ? (1u << valid) - 1u : 0u);
  uint32_t packed = 0u;  // element j's code in bits [4j, 4j + 4)
  uint32_t c_new;
  float d;
  static_assert(SRC != kExactGlobal || MD == kF32, "exact recompute from global needs binary32 moments");
  auto exact_wn = [&](int j) -> float {
    if constexpr (SRC == kExactStage) return fp4_exact_from_stage<GD, MD>(a, st, c, j, d_old);
    else if constexpr (SRC == kExactGlobal) return fp4_exact_from_global<GD>(a, x, e0 + j, d_old);
    else return madam_wn_exact(a.s, w[j], g[j], m[j], v[j], ve[j]);
  };
  if (!OPT && a.s.cert_ok) {
    // Certified path, as for block-scaled E4M3: fast weights and one error
    // bound et; the pair's maximum bounds decide the scale code (exact
    // maximum where they do not); then each element's interval, divided by
    // d through an approximate reciprocal, is encoded at both ends.
    float wf[8];
    float et = 0.0f, am = 0.0f;
    uint32_t bad = 0u;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const CertUpd u = madam_update_cert<true>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      wf[j] = u.wn;
      m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
      if (!u.ok) {
        bad |= 1u << j;
      } else {
        et = fmaxf(et, u.e);
        if ((vmask >> j) & 1u) am = fmaxf(am, fabsf(u.wn));
      }
    }
    if constexpr (SRC != kExactRegs) put_moments<MD, !SR>(x, e0, valid, m, v, ve);
    bad &= vmask;
    const float lo_t = bad ? 0.0f : fmaxf(__fsub_rd(am, et), 0.0f);
    const float hi_t = bad ? INFINITY : __fadd_ru(am, et);
    const uint32_t plo = pair_max(__float_as_uint(lo_t));
    const uint32_t phi = pair_max(__float_as_uint(hi_t));
    const Fp4Code cl = nvfp4_scale_code(__uint_as_float(plo), G, c_old);
    // the upper bound has the same code iff that code still covers it (or is the top one)
    const bool certain = plo != 0u && phi < 0x7E800000u /* 2^126 */ &&
                         (cl.c == 126u || cl.p >= __uint_as_float(phi));
    Fp4Code cn = cl;
    if (__any_sync(0xFFFFFFFFu, !certain)) {  // exact block maximum for the undecided pairs
      uint32_t amx = 0u;
      if (!certain) {
#pragma unroll
        for (int j = 0; j < kGroup; ++j) {
          if ((vmask >> j) & 1u) {
            const uint32_t bb = __float_as_uint(exact_wn(j)) & 0x7FFFFFFFu;
            if (bb < 0x7F800000u) amx = max(amx, bb);
          }
        }
      }
      amx = pair_max(amx);
      if (!certain) cn = nvfp4_scale_code(__uint_as_float(amx), G, c_old);
    }
    c_new = cn.c;
    d = __fmul_rn(e4m3_value(c_new), G);  // = cn.d, recomputed: fewer values live across the branch
    uint32_t redo = bad;
    if (d >= 1.1754943508222875e-38f /* 2^-126 */ && d <= 8.507059173023462e+37f /* 2^126 */) {
      // w' / d for w' in [wf - et, wf + et]: q = wf * inv (inv = rcp.approx(d),
      // 1 ulp; the product half an ulp) is within 2^-22 |q| of wf / d, and
      // et / d <= et inv (1 + 2^-22); widened to 2^-20 and 2^-126 absolute.
      float inv;
      asm("rcp.approx.f32 %0, %1;" : "=f"(inv) : "f"(d));
      const float ei = __fmaf_ru(et, __fmul_ru(inv, 1.0000009536743164f /* 1 + 2^-20 */), 1.1754943508222875e-38f);
      auto ends = [&](int j, float& xl, float& xh) {
        const float q = __fmul_rn(wf[j], inv);
        const float e2 = __fmaf_ru(fabsf(q), 9.5367431640625e-07f /* 2^-20 */, ei);
        xl = __fsub_rd(q, e2);
        xh = __fadd_ru(q, e2);
      };
      if (SR) {
        uint32_t rnd[8];
        group_random_bits<kNVFP4>(a, gi << 3, rnd);
        // lim = 2^32 - W for the group.  An interval's magnitudes span
        // xM - xm <= 3.5 e2: 2 e2 from ends() (e2 its bound), one directed
        // rounding at each end (each within e2 / 8, since e2 >= |q| 2^-20)
        // and the lower end below taken |q| 2^-20 lower still.  With e2 <=
        // (8 2^-20 + ei)(1 + 2^-23) while |q| <= 8, 2 (xM - xm) 2^32 + 1 <=
        // (2^-17 + ei) 2^35 + 2.  Larger |q| saturates at both ends (or, with
        // ei > 1, leaves lim = 0: nothing is certified).
        const uint32_t lim =
            ei <= 5.9604644775390625e-08f /* 2^-24 */
                ? 4294701056u /* 2^32 - (2^18 + 2^12): W <= 2^18 + 2^11 + 2 when ei <= 2^-24 */
                : __float2uint_rd(__fsub_rd(4294967296.0f,
                                            __fadd_ru(__fmaf_ru(ei, 34359738368.0f /* 2^35 */, 262144.0f /* 2^18 */),
                                                      2.0f)));
        const float inv_lo = __fmul_rd(inv, 0.999998092651367188f /* 1 - 2^-19 */);
#pragma unroll
        for (int j = 0; j < kGroup; ++j) {
          // a lower bound of the smaller magnitude of ends(): |wf| inv (1 - 2^-19)
          // (below |q| (1 - 2^-20), q = wf inv rounded) less ei, rounded down
          const float xm = __fmaf_rd(fabsf(wf[j]), inv_lo, -ei);
          bool same;
          packed |= e2m1_sr_interval(xm, wf[j], rnd[j], lim, same) << (4 * j);
          if (!same) redo |= 1u << j;
        }
      } else {  // two elements at a time, both ends
        uint32_t diff = 0u;
#pragma unroll
        for (int i = 0; i < kGroup / 2; ++i) {
          float l0, h0, l1, h1;
          ends(2 * i, l0, h0);
          ends(2 * i + 1, l1, h1);
          const uint32_t bl = e2m1x2_rn(l0, l1);
          packed |= bl << (8 * i);
          diff |= (bl ^ e2m1x2_rn(h0, h1)) << (8 * i);
        }
#pragma unroll
        for (int j = 0; j < kGroup; ++j)
          if ((diff >> (4 * j)) & 0xFu) redo |= 1u << j;
      }
    } else {
      redo = 0xFFu;
    }
    redo &= vmask;
    if (redo) {  // rare: the canonical weight of the undecided elements
      uint32_t rnd[8];
      if (SR) group_random_bits<kNVFP4>(a, gi << 3, rnd);
#pragma unroll
      for (int j = 0; j < kGroup; ++j) {
        if ((redo >> j) & 1u) {
          const float xe = __fdiv_rn(exact_wn(j), d);
          packed = (packed & ~(0xFu << (4 * j))) | ((e2m1_encode<SR>(xe, SR ? rnd[j] : 0u) & 0xFu) << (4 * j));
        }
      }
    }
    if constexpr (SRC == kExactRegs) put_moments<MD, !SR>(x, e0, valid, m, v, ve);
  } else {
    float wn[8];
    uint32_t amx = 0u;
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const Upd u = madam_update<OPT>(a.s, w[j], g[j], m[j], v[j], ve[j]);
      wn[j] = u.wn; m[j] = u.m; v[j] = u.v; ve[j] = u.ve;
      const uint32_t bb = __float_as_uint(u.wn) & 0x7FFFFFFFu;
      if (((vmask >> j) & 1u) && bb < 0x7F800000u) amx = max(amx, bb);
    }
    const Fp4Code cn = nvfp4_scale_code(__uint_as_float(pair_max(amx)), G, c_old);
    c_new = cn.c;
    d = cn.d;
    uint32_t rnd[8];
    if (SR) group_random_bits<kNVFP4>(a, gi << 3, rnd);
#pragma unroll
    for (int j = 0; j < kGroup; ++j)
      packed |= (e2m1_encode<SR>(__fdiv_rn(wn[j], d), SR ? rnd[j] : 0u) & 0xFu) << (4 * j);
    put_moments<MD, !SR>(x, e0, valid, m, v, ve);
  }
  put_fp4(packed, x.d.w, e0, valid, x.vec);
  if ((threadIdx.x & 1) == 0 && valid > 0) static_cast<uint8_t*>(x.scale)[e0 / kFp4Block] = static_cast<uint8_t>(c_new);
  if (x.cc) {
    float q[8];
    e2m1x8_to_f32(packed, q);
    uint32_t o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = bf16x2_rn(__fmul_rn(q[2 * i], d), __fmul_rn(q[2 * i + 1], d));
    put_bf16(o, x.cc, e0, valid, x.vec);
  }
}

// Eight NVFP4 weights decoded with d: from the stage or global memory as one
// 32-bit word when whole, else nibble by nibble.
__device__ __forceinline__ void get_fp4(float (&w)[8], bool staged, uint32_t saddr, const void* gw, int64_t e0,
                                        int valid, bool vec, float d) {
  if (staged || (vec && valid == kGroup)) {
    uint32_t r;
    if (staged) r = lds_u32(saddr);
    else asm("ld.global.L1::no_allocate.u32 %0, [%1];" : "=r"(r) : "l"(static_cast<const uint8_t*>(gw) + e0 / 2));
    e2m1x8_to_f32(r, w);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) w[j] = __fmul_rn(w[j], d);
  } else {
    const uint8_t* p = static_cast<const uint8_t*>(gw);
#pragma unroll
    for (int j = 0; j < kGroup; ++j) {
      const int64_t k = e0 + j;
      w[j] = j < valid ? __fmul_rn(e2m1_value((k & 1) ? (p[k >> 1] >> 4) : (p[k >> 1] & 0xFu)), d) : 0.0f;
    }
  }
}

// One NVFP4 group of a partial tile or of a tensor whose arrays are not all
// staged; every consumer lane calls this (the block maximum is a pair shuffle).
template <int GD, int MD, bool SR, bool OPT>
__device__ __noinline__ void general_fp4_group(const StepArgs& a, const TensorCtx& x, int64_t tile_e0, int count,
                                               int c, uint32_t st) {
  constexpr int GS = esize_of(GD), MS = esize_of(MD);
  const int rem = count - kGroup * c;
  const int valid = rem < 0 ? 0 : (rem < kGroup ? rem : kGroup);
  const int64_t e0 = tile_e0 + kGroup * c;
  const uint32_t end = static_cast<uint32_t>(kGroup * (c + 1));  // elements through this group
  const int nblk = (count + kFp4Block - 1) / kFp4Block, b = c >> 1;
  const uint8_t* sc = static_cast<const uint8_t*>(x.scale);
  uint32_t s_old = 0u;
  if (static_cast<uint32_t>(b + 1) <= staged_bytes(sc + tile_e0 / kFp4Block, nblk, 1))
    s_old = lds_u8(st + a.off_s + b);
  else if (b < nblk)
    s_old = sc[(tile_e0 / kFp4Block) + b];
  const float d_old = __fmul_rn(e4m3_value(s_old), x.gscale);
  float w[8], g[8], m[8], v[8], ve[8];
  get_fp4(w, end / 2 <= staged_bytes(x.d.w, (count + 1) / 2, 1), st + 4 * c, x.d.w, e0, valid, x.vec, d_old);
  const bool g_st = end * GS <= staged_bytes(x.g, count, GS);
  if (GD == kF32) get_f32<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  else get_bf16<true>(g, g_st, st + a.off_g + kGroup * GS * c, x.g, e0, valid, x.vec);
  const bool m_st = end * MS <= staged_bytes(x.d.m, count, MS);
  const bool v_st = end * MS <= staged_bytes(x.d.v, count, MS);
  const bool e_st = end * MS <= staged_bytes(x.d.ve, count, MS);
  if (MD == kF32) {
    get_f32<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_f32<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_f32<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  } else {
    get_bf16<false>(m, m_st, st + a.off_m + kGroup * MS * c, x.d.m, e0, valid, x.vec);
    get_bf16<false>(v, v_st, st + a.off_v + kGroup * MS * c, x.d.v, e0, valid, x.vec);
    get_bf16<false>(ve, e_st, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, valid, x.vec);
  }
  finish_fp4<GD, MD, SR, OPT, kExactRegs>(a, x, e0, valid, s_old, w, g, m, v, ve, st, c);
}

// ---------------------------------------------------------------------------
// The step kernel.
// ---------------------------------------------------------------------------
template <int WD, int GD, int MD, bool SR, bool OPT>
__global__ void __launch_bounds__(kThreads, 1) step_kernel(const __grid_constant__ StepArgs a) {
  constexpr int WS = esize_of(WD), GS = esize_of(GD), MS = esize_of(MD);
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ int64_t stage_tile[kMaxStages];  // tile the producer put in each stage (-1: no more work)
  __shared__ int32_t stage_k[kMaxStages];     // and its tensor

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int S = a.stages;
  const int64_t T = a.total_tiles;
  const int64_t tb = a.tile_base + static_cast<int64_t>(blockIdx.x) * T / gridDim.x;
  const int64_t te = a.tile_base + (static_cast<int64_t>(blockIdx.x) + 1) * T / gridDim.x;
  if (tb >= te && !a.pool) return;
  // static part of the range; the rest went to the tail pool
  const int64_t ts = a.pool ? tb + (te - tb) * a.static_q / 1024 : te;
  const uint32_t smem0 = smem_addr(smem);

  // ------------------------------------------------------------ producer --
  // One thread (lane 0 of the last warp) fills the ring.  Its state:
  uint64_t pol = 0;  // L2 policy of the bulk copies
  int pk = -1;       // tensor of tile t
  TensorDesc d{};
  const void* gp = nullptr;
  const uint8_t* sp = nullptr;
  int64_t tiles = 0;
  int64_t t = tb, t_end = ts;  // the current run of consecutive tiles
  int ps = 0;                  // next stage to fill, and how many times the ring has wrapped
  uint32_t puse = 0;
  int64_t issued = 0;
  auto load = [&](int kk) {
    pk = kk;
    d = desc_of(a, pk);
    gp = grad_of(a, pk);
    if (WD == kE4M3B || WD == kNVFP4) sp = static_cast<const uint8_t*>(aux_of(a, pk).scale);
    tiles = (d.numel + kTile - 1) / kTile;
  };
  auto issue = [&]() {  // the copies of tile t (of tensor pk) into stage ps, which is free
    const int64_t e0 = (t - d.tile_off) * kTile;
    const int count = static_cast<int>(d.numel - e0 < kTile ? d.numel - e0 : kTile);
    // NVFP4 weights: half a byte per element (tile starts stay 16-byte aligned: 1920 bytes per tile)
    const uint32_t nw = WD == kNVFP4 ? staged_bytes(d.w, (count + 1) / 2, 1) : staged_bytes(d.w, count, WS);
    const uint32_t ng = staged_bytes(gp, count, GS);
    const uint32_t nm = staged_bytes(d.m, count, MS), nv = staged_bytes(d.v, count, MS);
    const uint32_t nve = staged_bytes(d.ve, count, MS);
    const int64_t s0 = WD == kE4M3B ? 2 * (e0 / kBlock) : e0 / kFp4Block;  // the tile's first scale byte
    const uint32_t ns = WD == kE4M3B   ? staged_bytes(sp + s0, 2 * ((count + kBlock - 1) / kBlock), 1)
                        : WD == kNVFP4 ? staged_bytes(sp + s0, (count + kFp4Block - 1) / kFp4Block, 1)
                                       : 0u;
    const uint32_t bar = smem_addr(&full_bar[ps]);
    const uint32_t st = smem0 + static_cast<uint32_t>(ps * a.stage_bytes);
    stage_tile[ps] = t;  // published by the arrive below (release)
    stage_k[ps] = pk;
    mbar_arrive_expect_tx(bar, nw + ng + nm + nv + nve + ns);
    if (nw) tma_load(st, static_cast<const uint8_t*>(d.w) + (WD == kNVFP4 ? e0 / 2 : e0 * WS), nw, bar, pol);
    if (ng) tma_load(st + a.off_g, static_cast<const uint8_t*>(gp) + e0 * GS, ng, bar, pol);
    if (nm) tma_load(st + a.off_m, static_cast<const uint8_t*>(d.m) + e0 * MS, nm, bar, pol);
    if (nv) tma_load(st + a.off_v, static_cast<const uint8_t*>(d.v) + e0 * MS, nv, bar, pol);
    if (nve) tma_load(st + a.off_ve, static_cast<const uint8_t*>(d.ve) + e0 * MS, nve, bar, pol);
    if (ns) tma_load(st + a.off_s, sp + s0, ns, bar, pol);
    ++issued;
    ++t;
    if (++ps == S) { ps = 0; ++puse; }
  };
  if (tid == kConsumers) {
    // The producer sets up the ring and issues the copies of its first tile
    // before the block-wide barrier, in straight-line code next to the
    // kernel's entry: on a launch of a tile or two per CTA these copies are
    // on the critical path (issued 1.3 us after entry, against 2.0 us from
    // the loop below after the barrier).
    for (int i = 0; i < S; ++i) {
      mbar_init(smem_addr(&full_bar[i]), 1);
      mbar_init(smem_addr(&empty_bar[i]), kConsumerWarps);
    }
    mbar_init_fence();
    pol = evict_first_policy();
    if (t < t_end) {
      load(first_tensor(a, tb));
      while (t >= d.tile_off + tiles) load(pk + 1);
      issue();
    }
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    if (lane != 0) return;
    bool failed = false;
    for (;;) {
      if (t >= t_end) {  // static part done: next chunk of the tail pool, if any
        if (!a.pool) break;
        const uint32_t j = atomicAdd(a.pool_next, 1u);
        if (j >= static_cast<uint32_t>(a.pool_chunks)) break;
        const PoolChunk pc = a.pool[j];
        t = pc.start;
        t_end = pc.start + pc.count;
        if (pc.first != pk) load(pc.first);
      }
      while (t >= d.tile_off + tiles) load(pk + 1);
      if (puse > 0 && !mbar_wait(smem_addr(&empty_bar[ps]), (puse - 1) & 1u)) {
        if (a.err) atomicOr(a.err, kErrEmptyWait);
        failed = true;
        break;
      }
      issue();
    }
    if (failed) {  // wait (bounded) for this CTA's copies still in flight, then leave
      const int64_t last = issued < S ? issued : S;
      for (int64_t i = 1; i <= last; ++i) {
        const int64_t it = issued - i;
        if (!mbar_wait(smem_addr(&full_bar[it % S]), static_cast<uint32_t>((it / S) & 1)) && a.err)
          atomicOr(a.err, kErrDrainWait);
      }
      return;
    }
    // no more work: once the next stage is free, post the end marker there
    if (puse > 0 && !mbar_wait(smem_addr(&empty_bar[ps]), (puse - 1) & 1u)) {
      if (a.err) atomicOr(a.err, kErrEmptyWait);
      return;
    }
    stage_tile[ps] = -1;
    mbar_arrive(smem_addr(&full_bar[ps]));
    return;
  }

  // ----------------------------------------------------------- consumers --
  const int c = tid;  // consumer index, owns elements [8c, 8c + 8) of every tile
  const int n = a.n_tensors;
  int k = -1;
  TensorCtx x;
  int32_t e_next = 0;
  auto enter = [&](int kk) {  // take up tensor kk
    k = kk;
    load_tensor<WD, GD, MD>(a, k, x);
    if (WD == kE4M3) {
      const int32_t e_cur = a.fp8_exp[static_cast<int64_t>(a.e_cur_slot) * n + x.d.ring];
      e_next = fp8_next_exponent(a.fp8_amax[static_cast<int64_t>(a.a_cur_slot) * n + x.d.ring], e_cur);
      x.dec_scale = pow2f(e_cur);
      x.enc_scale = pow2f(-e_next);
      x.cc_scale = pow2f(e_next);
      // The tensor's maximum flushed so far in this step, read through L2:
      // the slot was zeroed before this step and is raised only with exact
      // values, so it seeds the recomputation threshold after a tensor change
      // (under the tail pool a CTA changes tensor at almost every chunk).
      uint32_t seed;
      asm volatile("ld.global.cg.u32 %0, [%1];"
                   : "=r"(seed)
                   : "l"(a.fp8_amax + static_cast<int64_t>(a.a_next_slot) * n + x.d.ring)
                   : "memory");
      x.amax_seed = __uint_as_float(seed);
    }
  };
  // The first tile posted is the first of this CTA's own range when it has
  // one: take up its tensor while the copies are in flight.
  if (tb < ts) enter(first_tensor(a, tb));
  uint32_t amax_bits = 0u;
  int s = 0;
  uint32_t use = 0;
  for (;;) {
    if (!__all_sync(0xFFFFFFFFu, mbar_wait(smem_addr(&full_bar[s]), use & 1u))) {  // warp-uniform give-up
      if (a.err && lane == 0) atomicOr(a.err, kErrFullWait);
      return;
    }
    const int64_t t = stage_tile[s];
    if (t < 0) break;  // the producer's end marker
    const int kt = stage_k[s];
    if (kt != k) {  // another tensor: flush this one's E4M3 amax
      if (WD == kE4M3 && k >= 0) {
        const uint32_t wmax = __reduce_max_sync(0xFFFFFFFFu, amax_bits);
        if (lane == 0 && wmax != 0u)
          atomicMax(&a.fp8_amax[static_cast<int64_t>(a.a_next_slot) * n + x.d.ring], wmax);
        amax_bits = 0u;
      }
      enter(kt);
    }
    const int64_t tile_e0 = (t - x.d.tile_off) * kTile;
    if (WD == kE4M3 && tile_e0 == 0 && c == 0) {  // the CTA holding the tensor's first tile
      a.fp8_exp[static_cast<int64_t>(a.e_next_slot) * n + x.d.ring] = e_next;
      a.fp8_amax[static_cast<int64_t>(a.a_zero_slot) * n + x.d.ring] = 0u;
    }
    const int count = static_cast<int>(x.d.numel - tile_e0 < kTile ? x.d.numel - tile_e0 : kTile);
    // Straight-line group: every array aligned, and this warp's 256 elements
    // all inside the tile (every warp of a whole tile; the whole warps of a
    // tensor's last tile, whose bytes the producer staged as well).  A warp
    // that holds the end of a partial tile takes the element-wise path below.
    if (x.fast && kGroup * 32 * (warp + 1) <= count) {
      const uint32_t st = smem0 + static_cast<uint32_t>(s * a.stage_bytes);
      const int64_t e0 = tile_e0 + kGroup * c;
      float w[8], g[8], m[8], v[8], ve[8];
      uint32_t h_old = 0u;
      if (WD == kBF16) {
        get_bf16<false>(w, true, st + kGroup * WS * c, x.d.w, e0, kGroup, true);
      } else if (WD == kE4M3) {
        get_e4m3(w, true, st + kGroup * WS * c, x.d.w, e0, kGroup, true, x.dec_scale);
      } else if (WD == kE4M3B) {
        h_old = lds_u16(st + a.off_s + 2 * (c >> 2));
        get_e4m3(w, true, st + kGroup * WS * c, x.d.w, e0, kGroup, true, fp16_value(h_old));
      } else {
        h_old = lds_u8(st + a.off_s + (c >> 1));
        get_fp4(w, true, st + 4 * c, x.d.w, e0, kGroup, true, __fmul_rn(e4m3_value(h_old), x.gscale));
      }
      if (GD == kF32) get_f32<true>(g, true, st + a.off_g + kGroup * GS * c, x.g, e0, kGroup, true);
      else get_bf16<true>(g, true, st + a.off_g + kGroup * GS * c, x.g, e0, kGroup, true);
      if (MD == kF32) {
        get_f32<false>(m, true, st + a.off_m + kGroup * MS * c, x.d.m, e0, kGroup, true);
        get_f32<false>(v, true, st + a.off_v + kGroup * MS * c, x.d.v, e0, kGroup, true);
        get_f32<false>(ve, true, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, kGroup, true);
      } else {
        get_bf16<false>(m, true, st + a.off_m + kGroup * MS * c, x.d.m, e0, kGroup, true);
        get_bf16<false>(v, true, st + a.off_v + kGroup * MS * c, x.d.v, e0, kGroup, true);
        get_bf16<false>(ve, true, st + a.off_ve + kGroup * MS * c, x.d.ve, e0, kGroup, true);
      }
      if constexpr (WD == kNVFP4 && MD == kF32) {
        // released at once: the rare exact branch re-reads global memory
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&empty_bar[s]));
        finish_fp4<GD, MD, SR, OPT, kExactGlobal>(a, x, e0, kGroup, h_old, w, g, m, v, ve, st, c);
      } else if constexpr (WD == kNVFP4) {
        // BF16 moments: the stage stays until the group is done (its exact
        // branch re-reads the binary32 originals there)
        finish_fp4<GD, MD, SR, OPT, kExactStage>(a, x, e0, kGroup, h_old, w, g, m, v, ve, st, c);
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&empty_bar[s]));
      } else if constexpr (WD == kBF16) {
        // the stage stays until the group is done: the rare exact branch reads
        // its inputs there
        finish_group<WD, GD, MD, SR, OPT, true>(a, x, e0, kGroup, w, g, m, v, ve, amax_bits, st, c);
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&empty_bar[s]));
      } else {
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_addr(&empty_bar[s]));
        if constexpr (WD == kE4M3B) finish_block<GD, MD, SR, OPT>(a, x, e0, kGroup, h_old, w, g, m, v, ve);
        else finish_group<WD, GD, MD, SR, OPT, false>(a, x, e0, kGroup, w, g, m, v, ve, amax_bits, st, c);
      }
      if (++s == S) { s = 0; ++use; }
      continue;
    }
    // partial tile or unstaged arrays: element-wise fallback (inline or a
    // call, by moment format; the NVFP4 one is always a call: inline it slowed
    // the stochastic-rounding loop by 5 %)
    if constexpr (WD == kE4M3B) {
      if constexpr (MD == kF32)
        general_block_group<GD, MD, SR, OPT>(a, x, tile_e0, count, c, smem0 + static_cast<uint32_t>(s * a.stage_bytes));
      else
        general_block_group_call<GD, MD, SR, OPT>(a, x, tile_e0, count, c,
                                                  smem0 + static_cast<uint32_t>(s * a.stage_bytes));
    } else if constexpr (WD == kNVFP4)
      general_fp4_group<GD, MD, SR, OPT>(a, x, tile_e0, count, c, smem0 + static_cast<uint32_t>(s * a.stage_bytes));
    else
      amax_bits = MD == kF32 ? general_group<WD, GD, MD, SR, OPT>(a, x, tile_e0, count, c,
                                                                   smem0 + static_cast<uint32_t>(s * a.stage_bytes),
                                                                   amax_bits)
                             : general_group_call<WD, GD, MD, SR, OPT>(
                                   a, x, tile_e0, count, c, smem0 + static_cast<uint32_t>(s * a.stage_bytes), amax_bits);
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&empty_bar[s]));
    if (++s == S) { s = 0; ++use; }
  }
  if (WD == kE4M3 && k >= 0) {
    const uint32_t wmax = __reduce_max_sync(0xFFFFFFFFu, amax_bits);
    if (lane == 0 && wmax != 0u) atomicMax(&a.fp8_amax[static_cast<int64_t>(a.a_next_slot) * n + x.d.ring], wmax);
  }
}

}  // namespace mpadam
