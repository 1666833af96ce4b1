// step_e4m3.cu -- instantiations of the fused step kernel for E4M3 weights.
#include "step_kernel.cuh"

namespace mpadam {

template <int GD, int MD>
static const void* pick_e4m3(int sr) {
  return sr ? reinterpret_cast<const void*>(&step_kernel<kE4M3, GD, MD, true>)
            : reinterpret_cast<const void*>(&step_kernel<kE4M3, GD, MD, false>);
}

const void* step_kernel_e4m3(int gd, int md, int sr) {
  if (gd == kF32 && md == kF32) return pick_e4m3<kF32, kF32>(sr);
  if (gd == kF32 && md == kBF16) return pick_e4m3<kF32, kBF16>(sr);
  if (gd == kBF16 && md == kF32) return pick_e4m3<kBF16, kF32>(sr);
  if (gd == kBF16 && md == kBF16) return pick_e4m3<kBF16, kBF16>(sr);
  return nullptr;
}

}  // namespace mpadam
