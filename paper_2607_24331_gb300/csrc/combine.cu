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
// Grid: (KV head h, chunk of sequences) x cluster of `split` CTAs along r_v
// (8 where r_v allows, else 4); a chunk holds as many (sequence, query head)
// rows as fit kMaxRows, so each head's B_v block is staged about once.
// CTA `rank` of a cluster owns rows [rank*rv/split, (rank+1)*rv/split) of u
// and of B_v's column block: it merges those rows of every (sequence, query
// head) row of its chunk (eight items' loads in flight at a time), stages its
// B_v rows in shared memory with cp.async (all issued up front), and forms the
// partial product over its rows.  The cluster adds the partial outputs through
// distributed shared memory and rank 0 writes o.
#include <algorithm>

#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace dck {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxSplit = 8;    // CTAs per cluster (r_v split), portable cluster size
constexpr int kMaxRows = 16;    // (sequence, query head) rows per cluster
constexpr int kItemBatch = 8;   // partial items whose loads are in flight together

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) combine_kernel(const LayerTable lt, const DecodeArgs a, int bchunk,
                                                          int split) {
  extern __shared__ __align__(16) uint8_t smem_c[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int B = a.B;
  const int qpg = lt.qpg, rv = lt.rv, Hq = lt.Hq;
  const int h = blockIdx.x / split;
  const int b0 = blockIdx.y * bchunk;
  const int nb = min(bchunk, B - b0);
  const int nrow = nb * qpg;
  const int rr = rv / split;            // rows of u / B_v owned by this CTA (a multiple of 4)
  const int r0 = rank * rr;

  // shared layout: B_v rows [rr][D] T | u rows [kMaxRows][rr] | partial o [kMaxRows][D] | m, 1/l | scan | prefix
  T* sbv = reinterpret_cast<T*>(smem_c);
  float* su = reinterpret_cast<float*>(smem_c + (size_t)rr * D * sizeof(T));
  float* so = su + (size_t)kMaxRows * rr;
  float* sM = so + kMaxRows * D;
  float* sinv = sM + kMaxRows;
  int* scan = reinterpret_cast<int*>(sinv + kMaxRows);
  int* prefix = scan + kThreads;

  // stage this CTA's B_v rows (all copies in flight at once)
  {
    const T* Bv = static_cast<const T*>(a.Bv) + (int64_t)h * D;
    const int64_t ldv = (int64_t)lt.Hkv * D;
    constexpr int kSegRow = D * (int)sizeof(T) / 16;
    for (int i = threadIdx.x; i < rr * kSegRow; i += kThreads) {
      const int r = i / kSegRow, c = i % kSegRow;
      cp_async16(reinterpret_cast<uint8_t*>(sbv + (size_t)r * D) + c * 16,
                 reinterpret_cast<const uint8_t*>(Bv + (int64_t)(r0 + r) * ldv) + c * 16);
    }
    cp_async_commit();
  }

  const int NT = build_tile_prefix(a.seq_len, a.seq_start, B, a.n_rows, prefix, scan, a.err, false);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // per row: reference max over the items and 1 / l (every CTA of the cluster does this)
  for (int i = warp; i < nrow; i += kThreads / 32) {
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    float M = -INFINITY, l = 0.f;
    if (prefix[b + 1] > prefix[b]) {
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
  // u rows restricted to [r0, r0 + rr): items summed with independent float4 loads
  const int rr4 = rr / 4;
  for (int idx = threadIdx.x; idx < nrow * rr4; idx += kThreads) {
    const int i = idx / rr4, r4 = idx % rr4;
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (prefix[b + 1] > prefix[b]) {
      const int c0 = item_of_tile(prefix[b], NT, a.n_items);
      const int c1 = item_of_tile(prefix[b + 1] - 1, NT, a.n_items);
      const float Mi = sM[i];
      for (int cc = c0; cc <= c1; cc += kItemBatch) {
        float w[kItemBatch];
        float4 v[kItemBatch];
#pragma unroll
        for (int u = 0; u < kItemBatch; ++u) {
          const int c = cc + u;
          const bool live = c <= c1 && item_begin(c, NT, a.n_items) != item_begin(c + 1, NT, a.n_items);
          const int64_t sl = ((int64_t)(live ? c : c0) + b) * Hq + j;
          w[u] = live ? exp2f(a.part_ml[sl * 2] - Mi) : 0.f;
          v[u] = reinterpret_cast<const float4*>(a.part_u + sl * rv + r0)[r4];
        }
#pragma unroll
        for (int u = 0; u < kItemBatch; ++u) {
          acc.x = fmaf(w[u], v[u].x, acc.x);
          acc.y = fmaf(w[u], v[u].y, acc.y);
          acc.z = fmaf(w[u], v[u].z, acc.z);
          acc.w = fmaf(w[u], v[u].w, acc.w);
        }
      }
    }
    reinterpret_cast<float4*>(su + (size_t)i * rr)[r4] = acc;
  }
  cp_async_wait_all();
  __syncthreads();
  // partial o over this CTA's rows: thread = (column pair, row phase)
  constexpr int kPairs = D / 2;
  constexpr int kPhases = kThreads / kPairs;  // 4 (D = 128) or 8 (D = 64)
  const int cp = threadIdx.x % kPairs, ph = threadIdx.x / kPairs;
  float acc[kMaxRows][2];
#pragma unroll
  for (int i = 0; i < kMaxRows; ++i) acc[i][0] = acc[i][1] = 0.f;
  for (int r = ph; r < rr; r += kPhases) {
    const float x0 = to_f32(sbv[(size_t)r * D + 2 * cp]), x1 = to_f32(sbv[(size_t)r * D + 2 * cp + 1]);
#pragma unroll
    for (int i = 0; i < kMaxRows; ++i) {
      if (i < nrow) {
        const float uv = su[(size_t)i * rr + r];
        acc[i][0] = fmaf(uv, x0, acc[i][0]);
        acc[i][1] = fmaf(uv, x1, acc[i][1]);
      }
    }
  }
  for (int i = threadIdx.x; i < kMaxRows * D; i += kThreads) so[i] = 0.f;
  __syncthreads();
#pragma unroll
  for (int i = 0; i < kMaxRows; ++i)
    if (i < nrow) {
      atomicAdd(&so[i * D + 2 * cp], acc[i][0]);
      atomicAdd(&so[i * D + 2 * cp + 1], acc[i][1]);
    }
  // cluster-wide sum of the partial outputs; rank 0 writes
  cluster.sync();
  if (rank == 0) {
    T* out = static_cast<T*>(a.out);
    for (int idx = threadIdx.x; idx < nrow * D; idx += kThreads) {
      float v = 0.f;
      for (int q = 0; q < split; ++q) v += cluster.map_shared_rank(so, q)[idx];
      const int i = idx / D, e = idx % D;
      const int b = b0 + i / qpg, j = h * qpg + i % qpg;
      out[((int64_t)b * Hq + j) * D + e] = from_f32<T>(v * sinv[i]);
    }
  }
  cluster.sync();  // keep every CTA's shared memory alive until rank 0 has read it
}

template <typename T, int D>
cudaError_t launch_t(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int split = lt.rv % (4 * kMaxSplit) == 0 ? kMaxSplit : kMaxSplit / 2;
  // as many sequences per cluster as its rows allow: each head's B_v block is staged once per chunk
  const int bchunk = std::max(1, std::min(a.B, kMaxRows / lt.qpg));
  const int rr = lt.rv / split;
  const size_t smem = (size_t)rr * D * sizeof(T) +
                      sizeof(float) * ((size_t)kMaxRows * rr + kMaxRows * D + 2 * kMaxRows) +
                      sizeof(int) * (kThreads + a.B + 1);
  auto k = combine_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(lt.Hkv * split, (a.B + bchunk - 1) / bchunk);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = split;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k, lt, a, bchunk, split);
}

}  // namespace

// r_v must split into at least four parts of whole float4 and 16-byte rows.
bool combine_supports(const LayerTable& lt) { return lt.rv % (4 * kMaxSplit / 2) == 0 && lt.rv <= kMaxRankV; }

cudaError_t launch_combine(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s) {
  if (dtype == DCK_F32) return lt.d == 64 ? launch_t<float, 64>(lt, a, s) : launch_t<float, 128>(lt, a, s);
  return lt.d == 64 ? launch_t<__nv_bfloat16, 64>(lt, a, s) : launch_t<__nv_bfloat16, 128>(lt, a, s);
}

}  // namespace dck
