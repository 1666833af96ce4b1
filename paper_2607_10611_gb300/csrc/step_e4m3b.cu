// step_e4m3b.cu -- instantiations of the fused step kernel for E4M3 weights
// with FP16 block scales (one per 32 elements).
#include "step_kernel.cuh"

namespace mpadam {

template <int GD, int MD, bool SR>
static const void* pick_e4m3b(int options) {
  return options ? reinterpret_cast<const void*>(&step_kernel<kE4M3B, GD, MD, SR, true>)
                 : reinterpret_cast<const void*>(&step_kernel<kE4M3B, GD, MD, SR, false>);
}

template <int GD, int MD>
static const void* pick_e4m3b(int sr, int options) {
  return sr ? pick_e4m3b<GD, MD, true>(options) : pick_e4m3b<GD, MD, false>(options);
}

const void* step_kernel_e4m3b(int gd, int md, int sr, int options) {
  if (gd == kF32 && md == kF32) return pick_e4m3b<kF32, kF32>(sr, options);
  if (gd == kF32 && md == kBF16) return pick_e4m3b<kF32, kBF16>(sr, options);
  if (gd == kBF16 && md == kF32) return pick_e4m3b<kBF16, kF32>(sr, options);
  if (gd == kBF16 && md == kBF16) return pick_e4m3b<kBF16, kBF16>(sr, options);
  return nullptr;
}

}  // namespace mpadam
