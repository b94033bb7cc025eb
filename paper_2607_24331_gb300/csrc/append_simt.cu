// CUDA-core latent append: key and value latents of new tokens,
//   kcache[rows[i]] = x_i A_k,  vcache[rows[i]] = x_i A_v     (Sec. III-A z = x L)
// with fp32 accumulation; a plain 64x64-tiled GEMM.  Used for fp32 layers and
// as the general kernel; bf16 layers take the tensor-core kernel.
#include "common.cuh"

namespace dck {
namespace {

constexpr int kBM = 64, kBN = 64, kBK = 16;

template <typename T>
__global__ void __launch_bounds__(256) append_simt_kernel(const T* __restrict__ x, int n_tok, int D,
                                                          const T* __restrict__ Ak, const T* __restrict__ Av,
                                                          int Rk, int rv, const int64_t* __restrict__ rows,
                                                          T* kc, T* vc, int64_t n_rows, int* err) {
  __shared__ float sx[kBK][kBM + 1];
  __shared__ float sa[kBK][kBN];
  const int n0 = blockIdx.x * kBN;  // column over [0, Rk + rv)
  const int m0 = blockIdx.y * kBM;
  const int N = Rk + rv;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < D; k0 += kBK) {
    for (int i = threadIdx.x; i < kBK * kBM; i += 256) {
      const int mm = i / kBK, kk = i % kBK;
      const int m = m0 + mm, k = k0 + kk;
      sx[kk][mm] = (m < n_tok && k < D) ? to_f32(x[(int64_t)m * D + k]) : 0.f;
    }
    for (int i = threadIdx.x; i < kBK * kBN; i += 256) {
      const int kk = i / kBN, nn = i % kBN;
      const int n = n0 + nn, k = k0 + kk;
      float v = 0.f;
      if (k < D && n < N) v = n < Rk ? to_f32(Ak[(int64_t)k * Rk + n]) : to_f32(Av[(int64_t)k * rv + (n - Rk)]);
      sa[kk][nn] = v;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kBK; ++kk) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(sx[kk][ty * 4 + i], sa[kk][tx * 4 + j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= n_tok) continue;
    const int64_t row = rows[m];
    if (row < 0 || row >= n_rows) {
      atomicOr(err, kErrBadRow);
      continue;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n < Rk) kc[row * Rk + n] = from_f32<T>(acc[i][j]);
      else if (n < N) vc[row * rv + (n - Rk)] = from_f32<T>(acc[i][j]);
    }
  }
}

}  // namespace

cudaError_t launch_append_simt(const void* x, int n_tok, int D, const void* A_k, const void* A_v, int Rk, int rv,
                               const int64_t* rows, void* kc, void* vc, int64_t n_rows, int dtype, int* err,
                               cudaStream_t s) {
  dim3 grid((Rk + rv + kBN - 1) / kBN, (n_tok + kBM - 1) / kBM);
  if (dtype == DCK_F32)
    append_simt_kernel<float><<<grid, 256, 0, s>>>((const float*)x, n_tok, D, (const float*)A_k, (const float*)A_v,
                                                   Rk, rv, rows, (float*)kc, (float*)vc, n_rows, err);
  else
    append_simt_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(
        (const __nv_bfloat16*)x, n_tok, D, (const __nv_bfloat16*)A_k, (const __nv_bfloat16*)A_v, Rk, rv, rows,
        (__nv_bfloat16*)kc, (__nv_bfloat16*)vc, n_rows, err);
  return cudaGetLastError();
}

}  // namespace dck
