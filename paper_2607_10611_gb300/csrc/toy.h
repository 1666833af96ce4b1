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
  double* partial;      // [batch / 256 + 2] chunk sums of the squared residuals
  double* loss_out;     // caller's device double, or nullptr (step-by-step mode)
  int64_t* t_dev;       // run mode: [0] = this step's t (advanced by the update kernel), [1] = the run's first t;
                        // nullptr in step-by-step mode (t from t_lo / t_hi)
  double* loss_base;    // run mode: the loss of step t goes to loss_base[t - t_dev[1]] (or nowhere if nullptr)
  int64_t n, batch;     // powers of two; 32 <= batch / halves <= 32 * 2048
  int32_t mode, split;
  float lr_add, lr_mul, rmax, tau, c_lo, c_hi;
  uint32_t rk0[kPhiloxRounds], rk1[kPhiloxRounds];
  uint32_t t_lo, t_hi;
};

cudaError_t launch_toy_step(const ToyArgs& a, cudaStream_t stream);
// Run mode: sets t_dev = {first, first} on `stream` (before the steps).
cudaError_t launch_toy_set_step(int64_t* t_dev, int64_t first, cudaStream_t stream);

}  // namespace mpadam
