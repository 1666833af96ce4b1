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
// Tail pool.  A launch may keep only a prefix of each CTA's range static:
// CTA b then walks [tb, tb + (te - tb) * static_q / 1024) and the rest of
// every range is cut into PoolChunks, handed out in order by an atomic
// counter to whichever CTA runs out of work first.  SMs do not all stream
// at the same rate, so a fixed split leaves the kernel waiting on the
// slowest; the pool evens out the end.  The producer warp decides each
// tile and posts its index and tensor beside the stage.
//
// Element indices for stochastic rounding are independent of this
// decomposition: element j of tensor k has global index goff[k] + j, where
// goff[0] = 0 and goff[k+1] = goff[k] + numel[k] rounded up to a multiple of 8.
//
// A list that mixes weight formats is stepped by one launch per format; each
// launch sees only its own tensors (its own descriptor, gradient and CTA
// tables), while global indices and the E4M3 scale rings stay those of the
// whole list.  Block-scaled E4M3 weights carry one FP16 power-of-two scale
// per kBlock consecutive elements; a tile holds kTileBlocks whole blocks, and
// the four consumer threads of a quad (lanes 4q .. 4q+3) own one block.
#pragma once

#include <cstdint>

namespace mpadam {

constexpr int kGroup = 8;                           // elements per consumer thread per tile
constexpr int kConsumerWarps = 15;                  // 16 warps per CTA: 4 per scheduler, <= 128 registers
constexpr int kConsumers = 32 * kConsumerWarps;     // 480 consumer threads
constexpr int kThreads = kConsumers + 32;           // + 1 producer warp
constexpr int kTile = kConsumers * kGroup;          // 3840 elements per tile (16-byte multiple in every format)
constexpr int kMaxStages = 8;
constexpr int kInlineTensors = 4;                   // launches of at most this many tensors carry their tables inline
constexpr int kPhiloxRounds = 10;
constexpr int kBlock = 32;                          // elements per block scale (block-scaled E4M3)
constexpr int kTileBlocks = kTile / kBlock;         // 120 block scales per tile (240 bytes)
static_assert(kTile % kBlock == 0 && kBlock == 4 * kGroup, "a block is one quad of consumer threads");
constexpr int kFp4Block = 16;                       // elements per NVFP4 block scale
constexpr int kTileFp4Blocks = kTile / kFp4Block;   // 240 E4M3 block scales per tile (240 bytes)
static_assert(kTile % kFp4Block == 0 && kFp4Block == 2 * kGroup, "an NVFP4 block is a pair of consumer threads");

// kE4M3B: E4M3 codes with FP16 block scales (one per kBlock elements).
// kNVFP4: E2M1 codes, two per byte (even element in the low nibble), with an
// E4M3 scale per kFp4Block elements and a binary32 scale per tensor.
enum Dtype : int { kF32 = 0, kBF16 = 1, kE4M3 = 2, kE4M3B = 3, kNVFP4 = 4 };

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
  int64_t tile_off;  // index of the tensor's first tile (in this launch's numbering)
  int32_t ring;      // the tensor's position in the whole list (its E4M3 scale-ring entries)
  int32_t pad;
};
static_assert(sizeof(TensorDesc) == 64, "TensorDesc must stay 64 bytes");

// Per-tensor extras of the E4M3 formats; one entry per descriptor, or no
// table at all when no tensor of the launch has any.
struct TensorAux {
  void* scale;        // kE4M3B: ceil(numel / kBlock) FP16 block scales; kNVFP4: ceil(numel / kFp4Block)
                      // E4M3 block scales; updated in place
  uint16_t* compute;  // BF16 copy of the updated stored weights (dequantised), or nullptr
  float gscale;       // kNVFP4: the tensor's binary32 scale
  int32_t pad;
};

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

// A run of consecutive tiles of the tail pool.
struct PoolChunk {
  int64_t start;  // first tile (this launch's numbering)
  int32_t count;  // tiles
  int32_t first;  // tensor holding tile `start`
};
static_assert(sizeof(PoolChunk) == 16, "PoolChunk must stay 16 bytes");

struct StepArgs {
  const TensorDesc* desc;    // [n_tensors]
  const void* const* grads;  // [n_tensors] device pointers
  const int32_t* cta_first;  // [gridDim.x] tensor holding each CTA's first tile
  const TensorAux* aux;      // [descriptors] or nullptr
  int64_t tile_base;         // this launch covers tiles [tile_base, tile_base + total_tiles)
  int64_t total_tiles;
  int32_t n_tensors;         // length of the whole list (stride of the scale rings)
  int32_t stages;            // shared-memory pipeline depth (2..kMaxStages)
  int32_t stage_bytes;       // bytes of one stage: w | g | m | v | ve | block-scale regions
  int32_t off_g, off_m, off_v, off_ve;  // region offsets inside a stage (w at 0)
  int32_t off_s;             // block scales (kE4M3B, kNVFP4)
  StepScalars s;
  uint32_t rk0[kPhiloxRounds], rk1[kPhiloxRounds];  // Philox round keys: seed + r * Weyl
  uint32_t t_lo, t_hi;       // step number (Philox counter words 2, 3)
  // E4M3 delayed-scaling rings (caller-owned); unused for BF16 weights
  int32_t* fp8_exp;          // [2][n_tensors]
  uint32_t* fp8_amax;        // [3][n_tensors] binary32 bits
  int32_t e_cur_slot, e_next_slot;
  int32_t a_cur_slot, a_next_slot, a_zero_slot;
  int32_t static_q;          // static prefix of each CTA's range, in 1/1024 (1024 when pool is nullptr)
  int32_t* err;              // DeviceError bits, or nullptr
  const PoolChunk* pool;     // [pool_chunks] tail pool, or nullptr (static ranges only)
  uint32_t* pool_next;       // next unclaimed pool chunk; zero when the launch starts
  int32_t pool_chunks;
  // Launches of at most kInlineTensors tensors (a flat parameter buffer, a
  // short list) carry their descriptors, aux entries and gradient pointers
  // here as well, so that a CTA finds its first tensor and issues its first
  // copies without dependent loads from global memory.  0: use the tables.
  int32_t n_inline;
  TensorDesc inl_desc[kInlineTensors];
  TensorAux inl_aux[kInlineTensors];
  const void* inl_grads[kInlineTensors];
};

// Kernel entry for the given formats (grad f32/bf16, moments f32/bf16,
// rounding nearest/stochastic, optional clips/decay present); defined in
// step_bf16.cu / step_e4m3.cu.
const void* step_kernel_bf16(int grad_dtype, int moment_dtype, int stochastic, int options);
const void* step_kernel_e4m3(int grad_dtype, int moment_dtype, int stochastic, int options);
const void* step_kernel_e4m3b(int grad_dtype, int moment_dtype, int stochastic, int options);
const void* step_kernel_nvfp4(int grad_dtype, int moment_dtype, int stochastic, int options);

}  // namespace mpadam
