// step_args.h -- host/device shared layout of the fused M+Adam step launch.
//
// Internal to the CUDA library (not part of the C ABI).  The work of one step
// is the padded global element index space [0, 8 * total_groups), split into
// groups of 8 consecutive indices (a group never straddles two tensors,
// because every tensor starts at a multiple of 8).  CTA b of a grid of B
// owns groups [b * G / B, (b + 1) * G / B): equal work per CTA, contiguous
// in memory, walked tensor by tensor starting at cta_first[b].
#pragma once

#include <cstdint>

namespace mpadam {

constexpr int kThreads = 256;  // threads per CTA of the step kernel
constexpr int kGroup = 8;      // elements per thread per iteration

enum Dtype : int { kF32 = 0, kBF16 = 1, kE4M3 = 2 };

// One tensor of the list: caller-owned device buffers and its place in the
// global element index space.  64 bytes, loaded once per tensor per CTA.
struct TensorDesc {
  void* w;
  void* m;
  void* v;
  void* ve;
  int64_t numel;
  int64_t goff;  // global index of element 0 (multiple of 8)
  int64_t pad0;
  int64_t pad1;
};
static_assert(sizeof(TensorDesc) == 64, "TensorDesc must stay 64 bytes");

// Per-step binary32 scalars of the canonical update (computed on the host in
// binary64 and rounded once).
struct StepScalars {
  float b1, b2;      // beta1, beta2
  float omb1, omb2;  // 1 - beta1, 1 - beta2
  float ka;          // -eta_a / (1 - beta1^t)
  float c2;          // 1 / sqrt(1 - beta2^t)
  float km;          // -eta_m
  float ln2;         // ln 2
  float eps, tau;
  float lo, hi;      // bounds of u_m
  float gmax, wmax;  // active when gmax_on / wmax_on
  float kwd;         // eta_a * lambda, active when wd_on
  int32_t gmax_on, wmax_on, wd_on;
  int32_t pad;
};

struct StepArgs {
  const TensorDesc* desc;    // [n_tensors]
  const void* const* grads;  // [n_tensors] device pointers
  const int32_t* cta_first;  // [gridDim.x] first tensor of each CTA's range
  int64_t total_groups;
  int32_t n_tensors;
  int32_t pad;
  StepScalars s;
  uint32_t key0, key1;       // Philox key = seed
  uint32_t t_lo, t_hi;       // step number (Philox counter words 2, 3)
  // E4M3 delayed-scaling rings (caller-owned); unused for BF16 weights
  int32_t* fp8_exp;          // [2][n_tensors]
  uint32_t* fp8_amax;        // [3][n_tensors] binary32 bits
  int32_t e_cur_slot, e_next_slot;
  int32_t a_cur_slot, a_next_slot, a_zero_slot;
  int32_t pad2;
};

// Kernel entry for the given formats (grad f32/bf16, moments f32/bf16,
// rounding nearest/stochastic); defined in step_bf16.cu / step_e4m3.cu.
const void* step_kernel_bf16(int grad_dtype, int moment_dtype, int stochastic);
const void* step_kernel_e4m3(int grad_dtype, int moment_dtype, int stochastic);

}  // namespace mpadam
