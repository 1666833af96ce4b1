// step_args.h -- host/device shared layout of the fused M+Adam step launch.
//
// Internal to the CUDA library (not part of the C ABI).
//
// Work decomposition.  Every tensor is cut into tiles of kTile consecutive
// elements (the last tile of a tensor may be short); tile j of tensor k starts
// at local element j * kTile, which keeps every tile's start 16-byte aligned in
// each array whenever the tensor's base pointers are.  Tiles are numbered
// tensor by tensor (tensor k owns tiles [tile_off[k], tile_off[k] + tiles_k)),
// and CTA b of a grid of B owns tiles [b * T / B, (b + 1) * T / B), walked in
// order starting at tensor cta_first[b].  Inside a tile, consumer thread c
// owns the 8 elements [8c, 8c + 8).
//
// Element indices for stochastic rounding are independent of this
// decomposition: element j of tensor k has global index goff[k] + j, where
// goff[0] = 0 and goff[k+1] = goff[k] + numel[k] rounded up to a multiple of 8.
#pragma once

#include <cstdint>

namespace mpadam {

constexpr int kGroup = 8;                           // elements per consumer thread per tile
constexpr int kConsumerWarps = 15;                  // 16 warps per CTA: 4 per scheduler, <= 128 registers
constexpr int kConsumers = 32 * kConsumerWarps;     // 480 consumer threads
constexpr int kThreads = kConsumers + 32;           // + 1 producer warp
constexpr int kTile = kConsumers * kGroup;          // 3840 elements per tile (16-byte multiple in every format)
constexpr int kMaxStages = 8;
constexpr int kPhiloxRounds = 10;

enum Dtype : int { kF32 = 0, kBF16 = 1, kE4M3 = 2 };

// Error bits a step kernel may set in *err (bounded waits that gave up).
enum DeviceError : int32_t { kErrFullWait = 1, kErrEmptyWait = 2, kErrDrainWait = 4 };

// One tensor of the list: caller-owned device buffers and its place in the
// global element index space and in the tile numbering.  64 bytes.
struct TensorDesc {
  void* w;
  void* m;
  void* v;
  void* ve;
  int64_t numel;
  int64_t goff;      // global index of element 0 (multiple of 8)
  int64_t tile_off;  // index of the tensor's first tile
  int64_t pad;
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
  int32_t cert_ok;   // eps >= 2^-28, tau >= 2^-125, c2 <= 2^14, eta_m <= 4: certified fast path allowed
};

struct StepArgs {
  const TensorDesc* desc;    // [n_tensors]
  const void* const* grads;  // [n_tensors] device pointers
  const int32_t* cta_first;  // [gridDim.x] tensor holding each CTA's first tile
  int64_t tile_base;         // this launch covers tiles [tile_base, tile_base + total_tiles)
  int64_t total_tiles;
  int32_t n_tensors;
  int32_t stages;            // shared-memory pipeline depth (2..kMaxStages)
  int32_t stage_bytes;       // bytes of one stage: w | g | m | v | ve regions
  int32_t off_g, off_m, off_v, off_ve;  // region offsets inside a stage (w at 0)
  int32_t pad0;
  StepScalars s;
  uint32_t rk0[kPhiloxRounds], rk1[kPhiloxRounds];  // Philox round keys: seed + r * Weyl
  uint32_t t_lo, t_hi;       // step number (Philox counter words 2, 3)
  // E4M3 delayed-scaling rings (caller-owned); unused for BF16 weights
  int32_t* fp8_exp;          // [2][n_tensors]
  uint32_t* fp8_amax;        // [3][n_tensors] binary32 bits
  int32_t e_cur_slot, e_next_slot;
  int32_t a_cur_slot, a_next_slot, a_zero_slot;
  int32_t pad1;
  int32_t* err;              // DeviceError bits, or nullptr
};

// Kernel entry for the given formats (grad f32/bf16, moments f32/bf16,
// rounding nearest/stochastic, optional clips/decay present); defined in
// step_bf16.cu / step_e4m3.cu.
const void* step_kernel_bf16(int grad_dtype, int moment_dtype, int stochastic, int options);
const void* step_kernel_e4m3(int grad_dtype, int moment_dtype, int stochastic, int options);

}  // namespace mpadam
