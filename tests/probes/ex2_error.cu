// Largest relative error of the hardware ex2.approx.ftz.f32 over every float t in [-126, 0],
// against exp2 in double precision.  The acceptance kernels' certified error bound assumes an
// upper bound on it (kEx2RelErr in csrc/common.cuh); tests/test_ex2_bound_gpu.py runs this probe.
#include <cstdint>
#include <cstring>
#include <cuda_runtime.h>

__global__ void ex2_err_kernel(uint32_t first, uint32_t count, unsigned int *max_bits) {
  float worst = 0.0f;
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < count; i += gridDim.x * blockDim.x) {
    const float t = __uint_as_float(first + i);  // negative floats: bit patterns grow with |t|
    float e;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(t));
    const double ref = exp2((double)t);
    const float rel = (float)(fabs((double)e - ref) / ref);
    worst = fmaxf(worst, rel);
  }
  atomicMax(max_bits, __float_as_uint(worst));  // non-negative floats order like their bits
}

extern "C" int ex2_max_rel_error(float *out) {
  unsigned int *d = nullptr;
  if (cudaMalloc(&d, sizeof(unsigned int)) != cudaSuccess) return 1;
  cudaMemset(d, 0, sizeof(unsigned int));
  const uint32_t first = 0x80000000u;                  // -0.0
  const uint32_t last = 0xC2FC0000u;                   // -126.0
  ex2_err_kernel<<<152 * 8, 256>>>(first, last - first + 1, d);
  unsigned int h = 0;
  const cudaError_t e = cudaMemcpy(&h, d, sizeof h, cudaMemcpyDeviceToHost);
  cudaFree(d);
  if (e != cudaSuccess) return 2;
  float f;
  memcpy(&f, &h, sizeof f);
  *out = f;
  return 0;
}
