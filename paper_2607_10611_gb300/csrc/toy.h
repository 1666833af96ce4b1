// toy.h -- launch arguments of the matrix-fitting diagnostic (internal to
// the CUDA library; the C ABI is mpadam_toy_* in include/mpadam.h).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "step_args.h"

namespace mpadam {

struct ToyArgs {
  uint16_t* w;          // [n] BF16 bits, updated in place
  const float* wstar;   // [n]
  int32_t* cnt;         // [n] hit counts (0 between steps)
  int32_t* first;       // [n] INT_MAX - (first sample of each entry); 0 between steps
  int32_t* idx;         // [batch]
  float* res;           // [batch]
  double* sq;           // [batch]
  float* alpha;         // [2]
  double* loss_h;       // [2]
  double* loss_out;     // caller's device double, or nullptr
  int64_t n, batch;     // powers of two; batch / halves >= 32, <= 2^16 * 1024
  int32_t mode, split;
  float lr_add, lr_mul, rmax, tau, c_lo, c_hi;
  uint32_t rk0[kPhiloxRounds], rk1[kPhiloxRounds];
  uint32_t t_lo, t_hi;
};

cudaError_t launch_toy_step(const ToyArgs& a, cudaStream_t stream);

}  // namespace mpadam
