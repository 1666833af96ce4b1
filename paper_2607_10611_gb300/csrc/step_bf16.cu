// step_bf16.cu -- instantiations of the fused step kernel for BF16 weights.
#include "step_kernel.cuh"

namespace mpadam {

template <int GD, int MD, bool SR>
static const void* pick_bf16(int options) {
  return options ? reinterpret_cast<const void*>(&step_kernel<kBF16, GD, MD, SR, true>)
                 : reinterpret_cast<const void*>(&step_kernel<kBF16, GD, MD, SR, false>);
}

template <int GD, int MD>
static const void* pick_bf16(int sr, int options) {
  return sr ? pick_bf16<GD, MD, true>(options) : pick_bf16<GD, MD, false>(options);
}

const void* step_kernel_bf16(int gd, int md, int sr, int options) {
  if (gd == kF32 && md == kF32) return pick_bf16<kF32, kF32>(sr, options);
  if (gd == kF32 && md == kBF16) return pick_bf16<kF32, kBF16>(sr, options);
  if (gd == kBF16 && md == kF32) return pick_bf16<kBF16, kF32>(sr, options);
  if (gd == kBF16 && md == kBF16) return pick_bf16<kBF16, kBF16>(sr, options);
  return nullptr;
}

}  // namespace mpadam
