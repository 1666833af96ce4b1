// Test-only probe: the largest relative error of the hardware approximations
// the step kernel's certified fast path relies on (sqrt.approx.f32 and
// div.approx.f32, flushing and not) against the correctly rounded
// operations, over caller-supplied normal operands with normal results.  The
// certificate assumes 2^-19.
#include <cstdint>
#include <cuda_runtime.h>

__global__ void probe(const float* a, const float* b, int64_t n, float* out_rel) {
  float worst_sqrt = 0.0f, worst_div = 0.0f;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const float x = fabsf(a[i]);
    float sa, sb;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(sa) : "f"(x));
    asm("sqrt.approx.f32 %0, %1;" : "=f"(sb) : "f"(x));
    const float se = __fsqrt_rn(x);
    if (se > 0.0f) worst_sqrt = fmaxf(worst_sqrt, fmaxf(fabsf(sa - se), fabsf(sb - se)) / se);
    float da, db;
    asm("div.approx.ftz.f32 %0, %1, %2;" : "=f"(da) : "f"(a[i]), "f"(b[i]));
    asm("div.approx.f32 %0, %1, %2;" : "=f"(db) : "f"(a[i]), "f"(b[i]));
    const float de = __fdiv_rn(a[i], b[i]);
    if (de != 0.0f && fabsf(de) >= 1.17549435e-38f)
      worst_div = fmaxf(worst_div, fmaxf(fabsf(da - de), fabsf(db - de)) / fabsf(de));
  }
  atomicMax(reinterpret_cast<int*>(&out_rel[0]), __float_as_int(worst_sqrt));
  atomicMax(reinterpret_cast<int*>(&out_rel[1]), __float_as_int(worst_div));
}

extern "C" int approx_probe(const float* a, const float* b, int64_t n, float* out_rel) {
  probe<<<1024, 256>>>(a, b, n, out_rel);
  return (int)cudaDeviceSynchronize();
}
