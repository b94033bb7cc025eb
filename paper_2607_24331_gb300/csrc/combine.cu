// Split merge and value up-projection of decode attention.
//
// Every work item wrote, for each sequence b it touched and each query head j,
// the un-normalised latent accumulator u = sum_t 2^(s_t - m) v_t, its reference
// max m (log2 units) and l = sum_t 2^(s_t - m).  For sequence b this kernel
// takes the items covering b's tiles, merges them with
//   M = max m_c,  u = sum_c 2^(m_c - M) u_c,  l = sum_c 2^(m_c - M) l_c
// and applies the value up-factor once per head (Sec. III-D, x W^(v) ~ z_v R_v):
//   o_j = (u / l) B_v[:, h d : (h+1) d],  h = KV head of j.
//
// Block (KV head h, chunk of sequences): rows are the chunk's (sequence,
// query head) pairs (at most 8).  The merge reads every partial with
// independent float4 loads; B_v's column block streams through shared memory
// in 32-row chunks with double-buffered cp.async, so each B_v element is read
// once per block.
#include <algorithm>

#include "common.cuh"

namespace dck {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxRows = 8;
constexpr int kChunkRows = 32;

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) combine_kernel(const LayerTable lt, const DecodeArgs a, int bchunk) {
  extern __shared__ __align__(16) uint8_t smem_c[];
  const int B = a.B;
  const int qpg = lt.qpg, rv = lt.rv, Hq = lt.Hq;
  const int h = blockIdx.x;
  const int b0 = blockIdx.y * bchunk;
  const int nb = min(bchunk, B - b0);
  const int nrow = nb * qpg;
  constexpr int kRowBytes = D * (int)sizeof(T);
  constexpr int kChunkBytes = kChunkRows * kRowBytes;

  // shared layout: B_v chunks (2 buffers) | u rows | reductions | prefix
  uint8_t* bvbuf = smem_c;                                                   // [2][32][D] T
  float* su = reinterpret_cast<float*>(smem_c + 2 * kChunkBytes);           // [nrow][rv]
  float* sM = su + (size_t)kMaxRows * rv;                                    // [kMaxRows]
  float* sinv = sM + kMaxRows;                                               // [kMaxRows]
  float* red = sinv + kMaxRows;                                              // [4][kMaxRows][D]
  int* scan = reinterpret_cast<int*>(red + 4 * kMaxRows * D);               // [kThreads]
  int* prefix = scan + kThreads;                                             // [B+1]

  // start streaming the first B_v chunk while the partials are merged
  const T* __restrict__ Bv = static_cast<const T*>(a.Bv) + (int64_t)h * D;
  const int64_t ldv = (int64_t)lt.Hkv * D;
  const int nchunks = (rv + kChunkRows - 1) / kChunkRows;
  constexpr int kSeg = kChunkBytes / 16;  // 16-byte segments per chunk
  auto issue_chunk = [&](int ch, int buf) {
    for (int i = threadIdx.x; i < kSeg; i += kThreads) {
      const int r = ch * kChunkRows + i / (kRowBytes / 16);
      const int cseg = i % (kRowBytes / 16);
      uint8_t* dst = bvbuf + buf * kChunkBytes + i * 16;
      if (r < rv) cp_async16(dst, reinterpret_cast<const uint8_t*>(Bv + r * ldv) + cseg * 16);
      else *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
    cp_async_commit();
  };
  issue_chunk(0, 0);

  const int NT = build_tile_prefix(a.seq_len, a.seq_start, B, a.n_rows, prefix, scan, a.err, false);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // per row: reference max over the items and 1 / l
  for (int i = warp; i < nrow; i += kThreads / 32) {
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    const int nt = prefix[b + 1] - prefix[b];
    float M = -INFINITY, l = 0.f;
    if (nt > 0) {
      const int c0 = item_of_tile(prefix[b], NT, a.n_items);
      const int c1 = item_of_tile(prefix[b + 1] - 1, NT, a.n_items);
      for (int cc = c0 + lane; cc <= c1; cc += 32)
        if (item_begin(cc, NT, a.n_items) != item_begin(cc + 1, NT, a.n_items))
          M = fmaxf(M, a.part_ml[(((int64_t)cc + b) * Hq + j) * 2]);
#pragma unroll
      for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      for (int cc = c0 + lane; cc <= c1; cc += 32)
        if (item_begin(cc, NT, a.n_items) != item_begin(cc + 1, NT, a.n_items)) {
          const int64_t sl = ((int64_t)cc + b) * Hq + j;
          l += exp2f(a.part_ml[sl * 2] - M) * a.part_ml[sl * 2 + 1];
        }
#pragma unroll
      for (int o = 16; o; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    }
    if (lane == 0) {
      sM[i] = M;
      sinv[i] = l > 0.f ? 1.f / l : 0.f;
    }
  }
  __syncthreads();
  // u rows: sum of the items' partials weighted by 2^(m_c - M)
  const int rv4 = rv / 4;
  for (int idx = threadIdx.x; idx < nrow * rv4; idx += kThreads) {
    const int i = idx / rv4, r4 = idx % rv4;
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (prefix[b + 1] > prefix[b]) {
      const int c0 = item_of_tile(prefix[b], NT, a.n_items);
      const int c1 = item_of_tile(prefix[b + 1] - 1, NT, a.n_items);
      for (int cc = c0; cc <= c1; ++cc) {
        if (item_begin(cc, NT, a.n_items) == item_begin(cc + 1, NT, a.n_items)) continue;
        const int64_t sl = ((int64_t)cc + b) * Hq + j;
        const float w = exp2f(a.part_ml[sl * 2] - sM[i]);
        const float4 v = reinterpret_cast<const float4*>(a.part_u + sl * rv)[r4];
        acc.x = fmaf(w, v.x, acc.x);
        acc.y = fmaf(w, v.y, acc.y);
        acc.z = fmaf(w, v.z, acc.z);
        acc.w = fmaf(w, v.w, acc.w);
      }
    }
    reinterpret_cast<float4*>(su + (size_t)i * rv)[r4] = acc;
  }
  // projection: thread = (column pair, row phase); rows of each B_v chunk are split 4 ways
  constexpr int kPairs = D / 2;
  constexpr int kPhases = kThreads / kPairs;  // 4 (D = 128) or 8 (D = 64)
  const int cp = threadIdx.x % kPairs, ph = threadIdx.x / kPairs;
  float acc[kMaxRows][2];
#pragma unroll
  for (int i = 0; i < kMaxRows; ++i) acc[i][0] = acc[i][1] = 0.f;
  for (int ch = 0; ch < nchunks; ++ch) {
    if (ch + 1 < nchunks) {
      issue_chunk(ch + 1, (ch + 1) & 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const T* bc = reinterpret_cast<const T*>(bvbuf + (ch & 1) * kChunkBytes);
    for (int rr = ph; rr < kChunkRows; rr += kPhases) {
      const int r = ch * kChunkRows + rr;
      if (r >= rv) break;
      const float x0 = to_f32(bc[rr * D + 2 * cp]), x1 = to_f32(bc[rr * D + 2 * cp + 1]);
#pragma unroll
      for (int i = 0; i < kMaxRows; ++i) {
        if (i < nrow) {
          const float uv = su[(size_t)i * rv + r];
          acc[i][0] = fmaf(uv, x0, acc[i][0]);
          acc[i][1] = fmaf(uv, x1, acc[i][1]);
        }
      }
    }
    __syncthreads();
  }
  if (ph < 4) {
#pragma unroll
    for (int i = 0; i < kMaxRows; ++i)
      if (i < nrow) {
        red[(ph * kMaxRows + i) * D + 2 * cp] = acc[i][0];
        red[(ph * kMaxRows + i) * D + 2 * cp + 1] = acc[i][1];
      }
  }
  __syncthreads();
  if (ph >= 4) {  // D = 64: phases 4..7 add into phases 0..3
#pragma unroll
    for (int i = 0; i < kMaxRows; ++i)
      if (i < nrow) {
        atomicAdd(&red[((ph - 4) * kMaxRows + i) * D + 2 * cp], acc[i][0]);
        atomicAdd(&red[((ph - 4) * kMaxRows + i) * D + 2 * cp + 1], acc[i][1]);
      }
  }
  __syncthreads();
  T* out = static_cast<T*>(a.out);
  for (int idx = threadIdx.x; idx < nrow * D; idx += kThreads) {
    const int i = idx / D, e = idx % D;
    const float v = red[(0 * kMaxRows + i) * D + e] + red[(1 * kMaxRows + i) * D + e] +
                    red[(2 * kMaxRows + i) * D + e] + red[(3 * kMaxRows + i) * D + e];
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    out[((int64_t)b * Hq + j) * D + e] = from_f32<T>(v * sinv[i]);
  }
}

template <typename T, int D>
cudaError_t launch_t(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int maxb = std::max(1, kMaxRows / lt.qpg);
  int bchunk = (a.B * lt.Hkv + sms - 1) / std::max(1, sms);
  bchunk = std::max(1, std::min(bchunk, maxb));
  const size_t smem = 2 * kChunkRows * D * sizeof(T) + sizeof(float) * ((size_t)kMaxRows * lt.rv + 2 * kMaxRows +
                                                                         4 * kMaxRows * D) +
                      sizeof(int) * (kThreads + a.B + 1);
  auto k = combine_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(lt.Hkv, (a.B + bchunk - 1) / bchunk);
  k<<<grid, kThreads, smem, s>>>(lt, a, bchunk);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_combine(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s) {
  if (dtype == DCK_F32) return lt.d == 64 ? launch_t<float, 64>(lt, a, s) : launch_t<float, 128>(lt, a, s);
  return lt.d == 64 ? launch_t<__nv_bfloat16, 64>(lt, a, s) : launch_t<__nv_bfloat16, 128>(lt, a, s);
}

}  // namespace dck
