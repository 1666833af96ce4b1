// toy.cu -- the BF16-stored matrix-fitting diagnostic (the toy diagnostic of
// Sec. 5.1 and its appendix) on the GPU: one step samples B entries of W
// with replacement, forms the minibatch loss c (mean squared residual)^2
// (per half when the halves are separate problems), and applies the
// additive, multiplicative or combined step (no moments) to every sampled
// entry, rounding it to BF16.  Two launches per step:
//   1. one CTA per aligned chunk of 256 samples draws them (Philox lanes;
//      residuals, hit counts and each entry's first sample, with atomics on
//      two n-entry scratch arrays that are zero between steps) and sums
//      their squared residuals as a subtree of the perfect binary tree of
//      binary64 sums over adjacent samples: each thread draws the adjacent
//      pair that is the tree's first level;
//   2. every CTA completes the tree from the partials (at most 32 per
//      problem), forms M, the loss and alpha = 4 c M / B_h; the first sample
//      of each entry applies the entry's update (its contribution alpha r
//      added once per hit) and clears the scratch.
// Every result is deterministic and equals the oracle's bit for bit.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "step_kernel.cuh"
#include "toy.h"

namespace mpadam {
namespace {

// This step's number: from the device counter in run mode, else the argument.
__device__ __forceinline__ void toy_step_number(const ToyArgs& a, uint32_t& lo, uint32_t& hi) {
  if (a.t_dev) {
    const uint64_t t = static_cast<uint64_t>(*a.t_dev);
    lo = static_cast<uint32_t>(t);
    hi = static_cast<uint32_t>(t >> 32);
  } else {
    lo = a.t_lo;
    hi = a.t_hi;
  }
}

__global__ void toy_set_step_kernel(int64_t* t_dev, int64_t first) {
  t_dev[0] = first;
  t_dev[1] = first;
}

// Sample s drawn with 32-bit lane `lane` of this step: its entry, residual,
// hit count and first-sample mark.  Returns r^2, exact in binary64.
__device__ __forceinline__ double toy_draw(const ToyArgs& a, int64_t s, uint32_t lane) {
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int64_t range = a.n / (a.split ? 2 : 1);
  const int64_t h = a.split ? s / Bh : 0;
  const int64_t idx = h * range + static_cast<int64_t>(static_cast<uint64_t>(lane) & static_cast<uint64_t>(range - 1));
  const float wv = __uint_as_float(static_cast<uint32_t>(a.w[idx]) << 16);
  const float r = __fsub_rn(wv, a.wstar[idx]);
  a.idx[s] = static_cast<int32_t>(idx);
  a.res[s] = r;
  atomicAdd(&a.cnt[idx], 1);
  atomicMax(&a.first[idx], INT_MAX - static_cast<int32_t>(s));  // the smallest sample wins
  return static_cast<double>(r) * static_cast<double>(r);
}

// Stage 1: CTA b of a problem draws the aligned chunk of C = min(256, B_h)
// samples [bC, bC + C) and sums their squared residuals as a perfect binary
// tree (adjacent pairs per thread, then adjacent lanes, then adjacent warps)
// into partial[problem][b].  Small chunks spread the random gathers over many
// SMs: at 65,536 samples per step, 2048-sample chunks (32 CTAs) took 14.8 us
// per step, 512 took 12.7 and 256 (256 CTAs) 12.6.
constexpr int kToyChunk = 256;
constexpr int kToyMaxPartials = 32 * 2048 / kToyChunk;  // per problem, at 65,536 samples

__global__ void __launch_bounds__(kToyChunk / 2) toy_sample_partial_kernel(const __grid_constant__ ToyArgs a) {
  __shared__ double warp_sum[32];
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int64_t C = Bh < kToyChunk ? Bh : kToyChunk;
  const int64_t per = Bh / C;  // chunks per problem
  const int h = static_cast<int>(blockIdx.x / per), b = static_cast<int>(blockIdx.x % per);
  const int pairs = static_cast<int>(C / 2);
  const int t = threadIdx.x;
  double x = 0.0;
  if (t < pairs) {
    uint32_t t_lo, t_hi;
    toy_step_number(a, t_lo, t_hi);
    // samples s and s + 1 (s even): lanes s mod 4 and s mod 4 + 1 of Philox block s / 4
    const int64_t s = h * Bh + b * C + 2 * t;
    const uint64_t blk = static_cast<uint64_t>(s) >> 2;
    const uint4 r4 = philox4x32_10(static_cast<uint32_t>(blk), static_cast<uint32_t>(blk >> 32), t_lo, t_hi, a.rk0,
                                   a.rk1);
    const bool upper = (s & 2) != 0;
    x = toy_draw(a, s, upper ? r4.z : r4.x) + toy_draw(a, s + 1, upper ? r4.w : r4.y);
  }
  const int span = pairs < 32 ? pairs : 32;  // lanes holding pair sums
  for (int off = 1; off < span; off <<= 1) {
    const double y = __shfl_xor_sync(0xFFFFFFFFu, x, off);
    x = (t & off) ? y + x : x + y;
  }
  const int nw = (pairs + 31) / 32;
  if ((t & 31) == 0 && t < pairs) warp_sum[t >> 5] = x;
  __syncthreads();
  if (t < 32) {
    double w = t < nw ? warp_sum[t] : 0.0;
    for (int off = 1; off < nw; off <<= 1) {
      const double y = __shfl_xor_sync(0xFFFFFFFFu, w, off);
      w = (t & off) ? y + w : w + y;
    }
    if (t == 0) a.partial[h * per + b] = w;
  }
}

// Stage 2 (every update CTA): the problem's partial sums, a perfect tree
// over at most 256 adjacent chunks (each lane first sums up to 8 adjacent
// ones), then M, the loss and alpha.
__device__ __forceinline__ void toy_finish_mean(const ToyArgs& a, int h, double& loss_h, float& alpha_h) {
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int64_t C = Bh < kToyChunk ? Bh : kToyChunk;
  const int per = static_cast<int>(Bh / C);
  const int lane = threadIdx.x & 31;
  const int q = per > 32 ? per / 32 : 1;        // adjacent partials per lane (a power of two)
  const int lanes = per > 32 ? 32 : per;        // lanes holding them
  double v[kToyMaxPartials / 32];
#pragma unroll
  for (int j = 0; j < kToyMaxPartials / 32; ++j) v[j] = j < q && lane < lanes ? a.partial[h * per + lane * q + j] : 0.0;
#pragma unroll
  for (int step = 1; step < kToyMaxPartials / 32; step <<= 1)
#pragma unroll
    for (int j = 0; j + step < kToyMaxPartials / 32; j += 2 * step)
      if (step < q) v[j] = v[j] + v[j + step];
  double w = v[0];
  for (int off = 1; off < lanes; off <<= 1) {
    const double y = __shfl_xor_sync(0xFFFFFFFFu, w, off);
    w = (lane & off) ? y + w : w + y;
  }
  const double M = w / static_cast<double>(Bh);
  const double ch = static_cast<double>(h == 0 ? a.c_lo : a.c_hi);
  loss_h = ch * M * M;
  alpha_h = static_cast<float>(((4.0 * ch) * M) / static_cast<double>(Bh));
}

__global__ void toy_update_kernel(const __grid_constant__ ToyArgs a) {
  __shared__ double s_loss[2];
  __shared__ float s_alpha[2];
  const int64_t s = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  // This sample's inputs, loaded while warps 0 and 1 form the mean: the
  // entry's first-sample mark, hit count and weight are independent reads
  // (a sample that is not its entry's first uses none of them; only the first
  // writes the entry, after reading it).
  int32_t idx = 0, first = 0, k = 0;
  uint16_t wbits = 0;
  float r = 0.0f;
  if (s < a.batch) {
    idx = a.idx[s];
    first = a.first[idx];
    k = a.cnt[idx];
    wbits = a.w[idx];
    r = a.res[s];
  }
  if (threadIdx.x < 64) {  // warp 0: the first problem, warp 1: the second
    const int h = threadIdx.x >> 5;
    if (h < (a.split ? 2 : 1)) {
      double l;
      float al;
      toy_finish_mean(a, h, l, al);
      if ((threadIdx.x & 31) == 0) { s_loss[h] = l; s_alpha[h] = al; }
    }
  }
  __syncthreads();
  if (s == 0) {
    const double loss = a.split ? (0.0 + s_loss[0]) + s_loss[1] : 0.0 + s_loss[0];
    if (a.t_dev) {  // run mode: record the loss by step, then advance the step counter
      const int64_t t = *a.t_dev;
      if (a.loss_base) a.loss_base[t - a.t_dev[1]] = loss;
      *a.t_dev = t + 1;  // read again only by the next step's kernels
    } else if (a.loss_out) {
      *a.loss_out = loss;
    }
  }
  if (s >= a.batch) return;
  if (first != INT_MAX - static_cast<int32_t>(s)) return;  // the entry's first sample applies its update
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int h = a.split ? static_cast<int>(s / Bh) : 0;
  const float x = __fmul_rn(s_alpha[h], r);
  float g = x;
  for (int32_t i = 1; i < k; ++i) g = __fadd_rn(g, x);
  const float wf = __uint_as_float(static_cast<uint32_t>(wbits) << 16);
  const float ln2 = 0.693147180559945309417232121458f;
  const float ua = __fmul_rn(-a.lr_add, g);
  const float ge = __fmul_rn(__fmul_rn(ln2, wf), g);
  const float ut = __fmul_rn(-a.lr_mul, ge);
  const float rho = fabsf(wf) > a.tau ? fabsf(wf) : a.tau;
  float um = __fdiv_rn(ut, rho);
  um = um > a.rmax ? a.rmax : um;
  um = um < -a.rmax ? -a.rmax : um;
  float wn;
  if (a.mode == 0) wn = __fadd_rn(wf, ua);
  else if (a.mode == 1) wn = __fmaf_rn(wf, um, wf);
  else wn = __fadd_rn(__fmaf_rn(wf, um, wf), ua);
  a.w[idx] = static_cast<uint16_t>(bf16x2_rn(wn, wn) & 0xFFFFu);
  a.cnt[idx] = 0;
  a.first[idx] = 0;
}

}  // namespace

cudaError_t launch_toy_step(const ToyArgs& a, cudaStream_t stream) {
  const int halves = a.split ? 2 : 1;
  const int64_t Bh = a.batch / halves;
  const int64_t C = Bh < kToyChunk ? Bh : kToyChunk;
  toy_sample_partial_kernel<<<static_cast<unsigned>(halves * (Bh / C)), kToyChunk / 2, 0, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const unsigned blocks = static_cast<unsigned>((a.batch + 255) / 256);
  toy_update_kernel<<<blocks, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_toy_set_step(int64_t* t_dev, int64_t first, cudaStream_t stream) {
  toy_set_step_kernel<<<1, 1, 0, stream>>>(t_dev, first);
  return cudaGetLastError();
}

}  // namespace mpadam
