// Seeded synthetic input generation on the device (not part of the method).
// Element i of stream `key`: SplitMix64 draws 2i and 2i+1 (Steele, Lea &
// Flood 2014; Vigna's constants), the sum s of their eight 16-bit fields,
// value = float32(2s - 8*65535) * scale as one IEEE fp32 multiply, then bf16
// round-to-nearest-even for bf16 tensors.  Integer work and single IEEE
// roundings only, so the values are bit-identical to the host generator.
#include "common.cuh"

namespace dck {
namespace {

__device__ __forceinline__ uint64_t splitmix_draw(uint64_t key, uint64_t i) {
  uint64_t z = key + (i + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ int field_sum(uint64_t z) {
  return (int)(z & 0xFFFF) + (int)((z >> 16) & 0xFFFF) + (int)((z >> 32) & 0xFFFF) + (int)(z >> 48);
}

__device__ __forceinline__ uint16_t bf16_rne_bits(float f) {
  const uint32_t u = __float_as_uint(f);
  return (uint16_t)((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

__global__ void synth_gaussian_kernel(void* dst, int64_t n, uint64_t key, int64_t start, float scale, int dtype) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t e = (uint64_t)(start + i);
    const int s = field_sum(splitmix_draw(key, 2 * e)) + field_sum(splitmix_draw(key, 2 * e + 1));
    const float v = __fmul_rn((float)(2 * s - 8 * 65535), scale);
    if (dtype == DCK_F32) static_cast<float*>(dst)[i] = v;
    else static_cast<uint16_t*>(dst)[i] = bf16_rne_bits(v);
  }
}

}  // namespace

cudaError_t launch_synth_gaussian(void* dst, int64_t n, uint64_t key, int64_t start, float scale, int dtype,
                                  cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (n + 255) / 256;
  const int blocks = (int)(want < (int64_t)sms * 16 ? want : (int64_t)sms * 16);
  synth_gaussian_kernel<<<blocks, 256, 0, s>>>(dst, n, key, start, scale, dtype);
  return cudaGetLastError();
}

}  // namespace dck
