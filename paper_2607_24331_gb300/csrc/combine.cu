// Split merge and value up-projection of decode attention.
//
// Every work item wrote, for each sequence b it touched and each query head j,
// the un-normalised latent accumulator u = sum_t 2^(s_t - m) v_t, its reference
// max m (log2 units) and l = sum_t 2^(s_t - m).  For sequence b this kernel
// takes the items covering b's tiles, merges them with
//   M = max m_c,  u = sum_c 2^(m_c - M) u_c,  l = sum_c 2^(m_c - M) l_c
// and applies the value up-factor once per head (Sec. III-D, x W^(v) ~ z_v R_v):
//   o_j = (u / l) B_v[:, h d : (h+1) d],  h = KV head of j.
// Block (chunk of sequences, KV head h): each B_v column block is read once for
// up to 8 (sequence, query head) rows at a time.
#include <algorithm>

#include "common.cuh"

namespace dck {
namespace {

constexpr int kThreads = 128;
constexpr int kSmemU = 48 * 1024;
constexpr int kAcc = 8;

template <typename T>
__global__ void __launch_bounds__(kThreads) combine_kernel(const LayerTable lt, const DecodeArgs a, int bchunk) {
  extern __shared__ float smem[];
  const int B = a.B;
  const int qpg = lt.qpg, rv = lt.rv, Hq = lt.Hq, d = lt.d;
  const int nrow_pad = (bchunk * qpg + kAcc - 1) / kAcc * kAcc;
  int* prefix = reinterpret_cast<int*>(smem);             // [B+1]
  int* scan = prefix + (B + 1);                            // [kThreads]
  float* su = reinterpret_cast<float*>(scan + kThreads);  // [nrow_pad][rv]
  float* sinv = su + (size_t)nrow_pad * rv;                // [nrow_pad]
  float* red = sinv + nrow_pad;                            // [kThreads][kAcc]

  const int NT = build_tile_prefix(a.seq_len, a.seq_start, B, a.n_rows, prefix, scan, a.err, false);
  const int h = blockIdx.y;
  const int b0 = blockIdx.x * bchunk;
  const int nb = min(bchunk, B - b0);
  const int nrow = nb * qpg;

  for (int i = nrow; i < nrow_pad; ++i) {
    for (int rr = threadIdx.x; rr < rv; rr += kThreads) su[(size_t)i * rv + rr] = 0.f;
    if (threadIdx.x == 0) sinv[i] = 0.f;
  }
  for (int bi = 0; bi < nb; ++bi) {
    const int b = b0 + bi;
    const int ntile = prefix[b + 1] - prefix[b];
    for (int jj = 0; jj < qpg; ++jj) {
      const int j = h * qpg + jj;
      float* u = su + ((size_t)bi * qpg + jj) * rv;
      for (int rr = threadIdx.x; rr < rv; rr += kThreads) u[rr] = 0.f;
      if (ntile == 0) {
        if (threadIdx.x == 0) sinv[bi * qpg + jj] = 0.f;
        continue;
      }
      const int c0 = item_of_tile(prefix[b], NT, a.n_items);
      const int c1 = item_of_tile(prefix[b + 1] - 1, NT, a.n_items);
      float M = -INFINITY;
      for (int cc = c0; cc <= c1; ++cc) {
        if (item_begin(cc, NT, a.n_items) == item_begin(cc + 1, NT, a.n_items)) continue;
        M = fmaxf(M, a.part_ml[(((int64_t)cc + b) * Hq + j) * 2]);
      }
      float l = 0.f;
      for (int cc = c0; cc <= c1; ++cc) {
        if (item_begin(cc, NT, a.n_items) == item_begin(cc + 1, NT, a.n_items)) continue;
        const int64_t sl = ((int64_t)cc + b) * Hq + j;
        const float w = exp2f(a.part_ml[sl * 2] - M);
        l += w * a.part_ml[sl * 2 + 1];
        const float* pu = a.part_u + sl * rv;
        for (int rr = threadIdx.x; rr < rv; rr += kThreads) u[rr] = fmaf(w, pu[rr], u[rr]);
      }
      if (threadIdx.x == 0) sinv[bi * qpg + jj] = l > 0.f ? 1.f / l : 0.f;
    }
  }
  __syncthreads();
  // o[row, e] = sum_r u[row, r] B_v[r, h d + e] / l, threads over (e, r-split)
  const T* __restrict__ Bv = static_cast<const T*>(a.Bv) + (int64_t)h * d;
  const int64_t ldv = (int64_t)lt.Hkv * d;
  T* out = static_cast<T*>(a.out);
  const int nsplit = kThreads / d;  // 1 (d = 128) or 2 (d = 64)
  const int e = threadIdx.x % d;
  const int part = threadIdx.x / d;
  for (int i0 = 0; i0 < nrow; i0 += kAcc) {
    float acc[kAcc];
#pragma unroll
    for (int k = 0; k < kAcc; ++k) acc[k] = 0.f;
    const float* ub = su + (size_t)i0 * rv;
    for (int rr = part; rr < rv; rr += nsplit) {
      const float bv = to_f32(Bv[(int64_t)rr * ldv + e]);
#pragma unroll
      for (int k = 0; k < kAcc; ++k) acc[k] = fmaf(ub[(size_t)k * rv + rr], bv, acc[k]);
    }
    if (nsplit > 1) {
      __syncthreads();
#pragma unroll
      for (int k = 0; k < kAcc; ++k) red[threadIdx.x * kAcc + k] = acc[k];
      __syncthreads();
      if (part == 0)
        for (int p = 1; p < nsplit; ++p)
#pragma unroll
          for (int k = 0; k < kAcc; ++k) acc[k] += red[(p * d + e) * kAcc + k];
    }
    if (part == 0) {
#pragma unroll
      for (int k = 0; k < kAcc; ++k) {
        const int i = i0 + k;
        if (i < nrow) {
          const int bi = i / qpg, jj = i % qpg;
          out[((int64_t)(b0 + bi) * Hq + h * qpg + jj) * d + e] = from_f32<T>(acc[k] * sinv[i]);
        }
      }
    }
  }
}

template <typename T>
cudaError_t launch_t(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  int bchunk = kSmemU / (int)(sizeof(float) * lt.qpg * lt.rv);
  bchunk = std::max(1, std::min(bchunk, std::min(a.B, 16)));
  const int nrow_pad = (bchunk * lt.qpg + kAcc - 1) / kAcc * kAcc;
  const size_t smem = sizeof(int) * (a.B + 1 + kThreads) +
                      sizeof(float) * ((size_t)nrow_pad * lt.rv + nrow_pad + kThreads * kAcc);
  auto k = combine_kernel<T>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.B + bchunk - 1) / bchunk, lt.Hkv);
  k<<<grid, kThreads, smem, s>>>(lt, a, bchunk);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_combine(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s) {
  return dtype == DCK_F32 ? launch_t<float>(lt, a, s) : launch_t<__nv_bfloat16>(lt, a, s);
}

}  // namespace dck
