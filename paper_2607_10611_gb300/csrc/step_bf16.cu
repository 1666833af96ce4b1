// step_bf16.cu -- instantiations of the fused step kernel for BF16 weights.
#include "step_kernel.cuh"

namespace mpadam {

template <int GD, int MD>
static const void* pick_bf16(int sr) {
  return sr ? reinterpret_cast<const void*>(&step_kernel<kBF16, GD, MD, true>)
            : reinterpret_cast<const void*>(&step_kernel<kBF16, GD, MD, false>);
}

const void* step_kernel_bf16(int gd, int md, int sr) {
  if (gd == kF32 && md == kF32) return pick_bf16<kF32, kF32>(sr);
  if (gd == kF32 && md == kBF16) return pick_bf16<kF32, kBF16>(sr);
  if (gd == kBF16 && md == kF32) return pick_bf16<kBF16, kF32>(sr);
  if (gd == kBF16 && md == kBF16) return pick_bf16<kBF16, kBF16>(sr);
  return nullptr;
}

}  // namespace mpadam
