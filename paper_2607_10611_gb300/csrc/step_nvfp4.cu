// step_nvfp4.cu -- instantiations of the fused step kernel for NVFP4 weights
// (E2M1 codes, an E4M3 scale per 16 elements, a binary32 tensor scale).
#include "step_kernel.cuh"

namespace mpadam {

template <int GD, int MD, bool SR>
static const void* pick_nvfp4(int options) {
  return options ? reinterpret_cast<const void*>(&step_kernel<kNVFP4, GD, MD, SR, true>)
                 : reinterpret_cast<const void*>(&step_kernel<kNVFP4, GD, MD, SR, false>);
}

template <int GD, int MD>
static const void* pick_nvfp4(int sr, int options) {
  return sr ? pick_nvfp4<GD, MD, true>(options) : pick_nvfp4<GD, MD, false>(options);
}

const void* step_kernel_nvfp4(int gd, int md, int sr, int options) {
  if (gd == kF32 && md == kF32) return pick_nvfp4<kF32, kF32>(sr, options);
  if (gd == kF32 && md == kBF16) return pick_nvfp4<kF32, kBF16>(sr, options);
  if (gd == kBF16 && md == kF32) return pick_nvfp4<kBF16, kF32>(sr, options);
  if (gd == kBF16 && md == kBF16) return pick_nvfp4<kBF16, kBF16>(sr, options);
  return nullptr;
}

}  // namespace mpadam
