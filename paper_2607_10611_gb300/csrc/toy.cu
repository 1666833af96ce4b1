// toy.cu -- the BF16-stored matrix-fitting diagnostic (the toy diagnostic of
// Sec. 5.1 and its appendix) on the GPU: one step samples B entries of W
// with replacement, forms the minibatch loss c (mean squared residual)^2
// (per half when the halves are separate problems), and applies the
// additive, multiplicative or combined step (no moments) to every sampled
// entry, rounding it to BF16.  Three launches per step:
//   1. sample (Philox lanes), residuals, hit counts and each entry's first
//      sample (atomics on two n-entry scratch arrays, zero between steps);
//   2. one CTA per half: the mean of the squared residuals as a perfect
//      binary tree of binary64 sums over adjacent samples, the gradient
//      scale alpha = 4 c M / B_h and the loss;
//   3. the first sample of each entry applies the entry's update (its
//      contribution alpha r added once per hit) and clears the scratch.
// Every result is deterministic and equals the oracle's bit for bit.
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "step_kernel.cuh"
#include "toy.h"

namespace mpadam {
namespace {

__global__ void toy_sample_kernel(const __grid_constant__ ToyArgs a) {
  const int64_t s = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (s >= a.batch) return;
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int64_t range = a.n / (a.split ? 2 : 1);
  const int64_t h = a.split ? s / Bh : 0;
  // 32-bit random lane s of step t: word s mod 4 of Philox block s / 4
  const uint64_t blk = static_cast<uint64_t>(s) >> 2;
  const uint4 r4 = philox4x32_10(static_cast<uint32_t>(blk), static_cast<uint32_t>(blk >> 32), a.t_lo, a.t_hi, a.rk0,
                                 a.rk1);
  const uint32_t lanes[4] = {r4.x, r4.y, r4.z, r4.w};
  const uint32_t lane = lanes[s & 3];
  const int64_t idx = h * range + static_cast<int64_t>(static_cast<uint64_t>(lane) & static_cast<uint64_t>(range - 1));
  const float wv = __uint_as_float(static_cast<uint32_t>(a.w[idx]) << 16);
  const float r = __fsub_rn(wv, a.wstar[idx]);
  a.idx[s] = static_cast<int32_t>(idx);
  a.res[s] = r;
  a.sq[s] = static_cast<double>(r) * static_cast<double>(r);  // exact
  atomicAdd(&a.cnt[idx], 1);
  atomicMax(&a.first[idx], INT_MAX - static_cast<int32_t>(s));  // the smallest sample wins
}

// Tree sum of one half's squared residuals: thread t takes the contiguous
// chunk of L = B_h / T samples (a binary-counter stack keeps the pairing of
// a perfect tree), then adjacent lanes, then adjacent warps.
__global__ void __launch_bounds__(1024) toy_reduce_kernel(const __grid_constant__ ToyArgs a) {
  __shared__ double warp_sum[32];
  const int h = blockIdx.x;
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int T = blockDim.x;
  const int64_t L = Bh / T;
  const double* v = a.sq + h * Bh + threadIdx.x * L;
  double stk[40];
  int top = 0;
  for (int64_t i = 0; i < L; ++i) {
    double x = v[i];
    int lvl = 0;
    for (uint64_t j = static_cast<uint64_t>(i); j & 1u; j >>= 1) x = stk[lvl++] + x;
    stk[lvl] = x;
    top = lvl;
  }
  double x = stk[top];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const double y = __shfl_xor_sync(0xFFFFFFFFu, x, off);
    x = (threadIdx.x & off) ? y + x : x + y;
  }
  if ((threadIdx.x & 31) == 0) warp_sum[threadIdx.x >> 5] = x;
  __syncthreads();
  if (threadIdx.x < 32) {
    const int nw = T >> 5;
    double w = threadIdx.x < nw ? warp_sum[threadIdx.x] : 0.0;
    for (int off = 1; off < nw; off <<= 1) {
      const double y = __shfl_xor_sync(0xFFFFFFFFu, w, off);
      w = (threadIdx.x & off) ? y + w : w + y;
    }
    if (threadIdx.x == 0) {
      const double M = w / static_cast<double>(Bh);
      const double ch = static_cast<double>(h == 0 ? a.c_lo : a.c_hi);
      a.loss_h[h] = ch * M * M;
      a.alpha[h] = static_cast<float>(((4.0 * ch) * M) / static_cast<double>(Bh));
    }
  }
}

__global__ void toy_update_kernel(const __grid_constant__ ToyArgs a) {
  const int64_t s = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (s == 0 && a.loss_out) *a.loss_out = a.split ? (0.0 + a.loss_h[0]) + a.loss_h[1] : 0.0 + a.loss_h[0];
  if (s >= a.batch) return;
  const int32_t idx = a.idx[s];
  if (a.first[idx] != INT_MAX - static_cast<int32_t>(s)) return;  // the entry's first sample applies its update
  const int64_t Bh = a.batch / (a.split ? 2 : 1);
  const int h = a.split ? static_cast<int>(s / Bh) : 0;
  const int32_t k = a.cnt[idx];
  const float x = __fmul_rn(a.alpha[h], a.res[s]);
  float g = x;
  for (int32_t i = 1; i < k; ++i) g = __fadd_rn(g, x);
  const float wf = __uint_as_float(static_cast<uint32_t>(a.w[idx]) << 16);
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
  const unsigned blocks = static_cast<unsigned>((a.batch + 255) / 256);
  toy_sample_kernel<<<blocks, 256, 0, stream>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  toy_reduce_kernel<<<halves, static_cast<unsigned>(Bh < 1024 ? Bh : 1024), 0, stream>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  toy_update_kernel<<<blocks, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace mpadam
