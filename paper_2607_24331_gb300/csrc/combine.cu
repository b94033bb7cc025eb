// Split merge and value up-projection of decode attention.
//
// Every work item wrote, for each sequence b it touched and each query head j,
// the un-normalised latent accumulator u = sum_t 2^(s_t - m) v_t, its reference
// max m (log2 units) and l = sum_t 2^(s_t - m).  CUDA-core path: item c covers
// a contiguous range of 128-token tiles and writes slot c + b.  Tensor-core
// path (the pair-tile plan of tc_common.cuh): each half of CTA pair p writes
// slot 2 (p + b) + half, and each half of an extra pair tile e its own slot;
// a slot whose half holds no token of b is not read.  For sequence b this
// kernel takes the partials covering b's tiles, merges them with
//   M = max m_c,  u = sum_c 2^(m_c - M) u_c,  l = sum_c 2^(m_c - M) l_c
// and applies the value up-factor once per head (Sec. III-D, x W^(v) ~ z_v R_v):
//   o_j = (u / l) B_v[:, h d : (h+1) d],  h = KV head of j.
//
// Grid: (KV head h, chunk of sequences) x cluster of `split` CTAs along r_v
// (8 where r_v allows, else 4); a chunk holds as many (sequence, query head)
// rows as fit kMaxRows, so each head's B_v block is staged about once.
// CTA `rank` of a cluster owns rows [rank*rv/split, (rank+1)*rv/split) of u
// and of B_v's column block.  It stages its B_v rows in shared memory with
// cp.async (all issued up front), lists each (sequence, query head) row's live
// partial slots with their maxima and sums in shared memory, forms every row's
// merged maximum M, weights 2^(m_c - M) and 1/l, then sums its rows of u with
// those weights (the loads of a row are independent, so they are all in
// flight together), and forms the partial product over its rows of B_v, each
// output owned by one thread.  The cluster adds the partial outputs through
// distributed shared memory, every rank reducing and writing a share of o.
#include <algorithm>
#include <type_traits>

#include <cooperative_groups.h>

#include "common.cuh"
#include "tc_common.cuh"

namespace cg = cooperative_groups;

#ifndef DCK_CB_TRACE
#define DCK_CB_TRACE(code) ((void)0)
#endif

namespace dck {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxSplit = 8;    // CTAs per cluster (r_v split), portable cluster size
constexpr int kMaxRows = 16;    // (sequence, query head) rows per cluster
constexpr int kMergeBatch = 16; // partial loads of a row in flight together

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ uint32_t f32_to_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}
// d += a b for one 16 x 8 x 8 tile, tf32 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Row stride (elements) of the staged B_v rows: padded by 16 bytes on the
// tensor-core path, whose fragments read four rows at one column.
template <typename T, int D>
__host__ __device__ constexpr int ldb() {
  return D + (std::is_same<T, __nv_bfloat16>::value && D == 128 ? 8 : 0);
}

// Two adjacent elements (16-byte aligned row, even column) as floats.
__device__ __forceinline__ float2 pair_f32(const float* p) { return *reinterpret_cast<const float2*>(p); }
__device__ __forceinline__ float2 pair_f32(const __nv_bfloat16* p) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 2) combine_kernel(const LayerTable lt, const DecodeArgs a, int bchunk,
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
  DCK_CB_TRACE(99);

  // shared layout: B_v rows [rr][ldb] T | u rows [kMaxRows][rr + 4] | received partial o [split][kMaxRows * D / split]
  // | 1/l | per row: partial weights [kMaxRows][cap] f32, sums [kMaxRows][cap] f32, slots [kMaxRows][cap] i32,
  // partial counts [kMaxRows] | row slot ranges [kMaxRows][4] | row 128-token tiles [kMaxRows] | prefix [B + 1]
  // | item starts [n_items + 1]
  const int cap = 2 * a.n_items;  // partials a row can have, on either work plan
  T* sbv = reinterpret_cast<T*>(smem_c);
  float* su = reinterpret_cast<float*>(smem_c + (size_t)rr * ldb<T, D>() * sizeof(T));
  const int ldu = rr + 4;  // padded u rows: the tensor-core fragments read 8 rows at one column
  float* so = su + (size_t)kMaxRows * ldu;
  float* sinv = so + kMaxRows * D;
  float* pw = sinv + kMaxRows;
  float* pl = pw + (size_t)kMaxRows * cap;
  int* ps = reinterpret_cast<int*>(pl + (size_t)kMaxRows * cap);
  int* pn = ps + (size_t)kMaxRows * cap;
  int* rc = pn + kMaxRows;
  int* rn128 = rc + 4 * kMaxRows;
  int* prefix = rn128 + kMaxRows;
  int* ibeg = prefix + B + 1;

  // stage this CTA's B_v rows (all copies in flight at once)
  {
    const T* Bv = static_cast<const T*>(a.Bv) + (int64_t)h * D;
    const int64_t ldv = (int64_t)lt.Hkv * D;
    constexpr int kSegRow = D * (int)sizeof(T) / 16;
    for (int i = threadIdx.x; i < rr * kSegRow; i += kThreads) {
      const int r = i / kSegRow, c = i % kSegRow;
      cp_async16(reinterpret_cast<uint8_t*>(sbv + (size_t)r * ldb<T, D>()) + c * 16,
                 reinterpret_cast<const uint8_t*>(Bv + (int64_t)(r0 + r) * ldv) + c * 16);
    }
    cp_async_commit();
  }

  // tiles: pair tiles (tensor-core path) or 128-token tiles; items: CTA pairs or CTAs
  const bool pairs = a.split_extra != 0;
  const int n_it = pairs ? a.n_items / 2 : a.n_items;
  // tiles per sequence (every thread a share), then an exclusive prefix by warp 0
  const int tile = pairs ? 2 * kTile : kTile;
  for (int b = threadIdx.x; b < B; b += kThreads)
    prefix[b + 1] = (valid_len(a.seq_len, a.seq_start, b, a.n_rows) + tile - 1) / tile;
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int run = 0;
    for (int b0s = 0; b0s < B; b0s += 32) {
      int v = b0s + lane < B ? prefix[b0s + lane + 1] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
      }
      if (b0s + lane < B) prefix[b0s + lane + 1] = run + v;
      run += __shfl_sync(0xffffffffu, v, 31);
    }
    if (lane == 0) prefix[0] = 0;
  }
  __syncthreads();
  const int NT = prefix[B];
  // Partials of sequence b: the items whose main tiles (the first NTm, split
  // evenly in whole tiles) cover b's; on the tensor-core path also the extra
  // pair tiles of b (x >= NTm), two slots (halves) per item and per extra tile.
  const int NTm = main_tiles(NT, n_it, pairs);
  for (int c = threadIdx.x; c <= n_it; c += kThreads) ibeg[c] = item_begin(c, NTm, n_it);
  if (threadIdx.x < nrow) {
    const int b = b0 + threadIdx.x / qpg;
    const int me = min(prefix[b + 1], NTm);  // end of b's main tiles
    const bool any = me > prefix[b];
    int* r = rc + 4 * threadIdx.x;
    rn128[threadIdx.x] = (valid_len(a.seq_len, a.seq_start, b, a.n_rows) + kTile - 1) / kTile;
    r[0] = any ? item_of_tile(prefix[b], NTm, n_it) : 0;           // first main item
    r[1] = any ? item_of_tile(me - 1, NTm, n_it) - r[0] + 1 : 0;  // main items
    r[2] = max(prefix[b], NTm) - NTm;                              // first extra tile
    r[3] = max(prefix[b + 1] - NTm, r[2]) - r[2];                  // extra tiles
  }
  __syncthreads();

  DCK_CB_TRACE(1);
  // Launched under programmatic dependent launch: everything above reads only the
  // call's inputs; the partials come from the kernels before, complete once the
  // preceding grid is.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  DCK_CB_TRACE(2);

  // (1) one warp per row: each live partial's slot, reference max m (log2
  // units) and sum l, their loads all in flight together (a lane per
  // partial); then M = max m, the weights 2^(m - M) and 1/l; (2) this CTA's
  // rows of u as the weighted sum, all of a row's loads independent.
  {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nps = pairs ? 2 : 1;  // slots per item or extra tile
    for (int i = warp; i < nrow; i += kThreads / 32) {
      const int b = b0 + i / qpg, j = h * qpg + i % qpg;
      const int c0 = rc[4 * i], nm = rc[4 * i + 1], e0 = rc[4 * i + 2];
      const int ns = nps * (nm + rc[4 * i + 3]);
      const int n128 = rn128[i];
      float M = -INFINITY;
      for (int q = lane; q < ns; q += 32) {
        const int k = q / nps, hh = q % nps;
        bool live;
        int64_t slot;
        if (k < nm) {  // item c0 + k
          const int c = c0 + k;
          live = ibeg[c] != ibeg[c + 1];
          if (pairs) {
            const int i0 = max(ibeg[c], prefix[b]) - prefix[b];  // b's first pair tile in the item
            live = live && 2 * i0 + hh < n128;
            slot = tc::pair_slot(c, b, hh);
          } else {
            slot = (int64_t)c + b;
          }
        } else {  // extra pair tile e (tensor-core path only)
          const int e = e0 + k - nm;
          live = 2 * (NTm + e - prefix[b]) + hh < n128;
          slot = tc::pair_xslot(n_it, B, e, hh);
        }
        float m = -INFINITY, l = 0.f;
        if (live) {
          const float2 ml = reinterpret_cast<const float2*>(a.part_ml)[slot * Hq + j];
          m = ml.x;
          l = ml.y;
        }
        pw[(size_t)i * cap + q] = m;
        pl[(size_t)i * cap + q] = l;
        ps[(size_t)i * cap + q] = live ? (int)slot : -1;
        M = fmaxf(M, m);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
      float l = 0.f;
      for (int q = lane; q < ns; q += 32) {  // entries this lane wrote itself
        const float wq = M == -INFINITY ? 0.f : exp2f(pw[(size_t)i * cap + q] - M);  // 0 for slots not live
        pw[(size_t)i * cap + q] = wq;
        l = fmaf(wq, pl[(size_t)i * cap + q], l);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
      if (lane == 0) {
        sinv[i] = l > 0.f ? 1.f / l : 0.f;
        pn[i] = ns;
      }
    }
  }
  __syncthreads();
  DCK_CB_TRACE(3);
  const int rr4 = rr / 4;
  for (int idx = threadIdx.x; idx < nrow * rr4; idx += kThreads) {
    const int i = idx / rr4, r4 = idx % rr4;
    const int j = h * qpg + i % qpg;
    const int n = pn[i];
    const float* wrow = pw + (size_t)i * cap;
    const int* srow = ps + (size_t)i * cap;
    float4 acc0 = make_float4(0.f, 0.f, 0.f, 0.f), acc1 = acc0;
    // batches of kMergeBatch partials, every load of a batch in flight before
    // the first is used (a row has up to a few tens of partials: one or two
    // L2 round trips per row instead of one per partial)
    for (int q0 = 0; q0 < n; q0 += kMergeBatch) {
      float4 v[kMergeBatch];
#pragma unroll
      for (int u = 0; u < kMergeBatch; ++u) {
        const int sl = q0 + u < n ? srow[q0 + u] : -1;
        v[u] = sl >= 0 ? __ldcg(reinterpret_cast<const float4*>(a.part_u + ((int64_t)sl * Hq + j) * rv + r0) + r4)
                       : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < kMergeBatch; ++u) {
        float4& ac = (u & 1) ? acc1 : acc0;
        const float wq = q0 + u < n ? wrow[q0 + u] : 0.f;
        ac.x = fmaf(wq, v[u].x, ac.x);
        ac.y = fmaf(wq, v[u].y, ac.y);
        ac.z = fmaf(wq, v[u].z, ac.z);
        ac.w = fmaf(wq, v[u].w, ac.w);
      }
    }
    reinterpret_cast<float4*>(su + (size_t)i * ldu)[r4] =
        make_float4(acc0.x + acc1.x, acc0.y + acc1.y, acc0.z + acc1.z, acc0.w + acc1.w);
  }
  DCK_CB_TRACE(4);
  cp_async_wait_all();
  __syncthreads();
  DCK_CB_TRACE(5);
  const int share = kMaxRows * D / split;
  if constexpr (std::is_same<T, __nv_bfloat16>::value && D == 128) {
    // partial o over this CTA's rows of B_v on the tensor cores: o[16 x 128] =
    // u[16 x rr] B_v[rr x 128], mma m16n8k8 tf32 (B_v's bf16 converts exactly;
    // u rounds to tf32, a relative 2^-11); warp w owns columns [16 w, 16 w + 16)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int gid = lane >> 2, tig = lane & 3;
    float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll 4
    for (int k0 = 0; k0 < rr; k0 += 8) {
      uint32_t af[4];
      af[0] = f32_to_tf32(su[(size_t)gid * ldu + k0 + tig]);
      af[1] = f32_to_tf32(su[(size_t)(gid + 8) * ldu + k0 + tig]);
      af[2] = f32_to_tf32(su[(size_t)gid * ldu + k0 + tig + 4]);
      af[3] = f32_to_tf32(su[(size_t)(gid + 8) * ldu + k0 + tig + 4]);
#pragma unroll
      for (int nt = 0; nt < 2; ++nt) {
        const int col = 16 * warp + 8 * nt + gid;
        const uint32_t b0 = (uint32_t)__bfloat16_as_ushort(sbv[(size_t)(k0 + tig) * ldb<T, D>() + col]) << 16;
        const uint32_t b1 = (uint32_t)__bfloat16_as_ushort(sbv[(size_t)(k0 + tig + 4) * ldb<T, D>() + col]) << 16;
        mma_tf32(acc[nt], af, b0, b1);
      }
    }
    // outputs (row, col): this thread has rows gid, gid + 8 and columns 2 tig, 2 tig + 1 of each n-tile
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int i = gid + 8 * (q >> 1), col = 16 * warp + 8 * nt + 2 * tig + (q & 1);
        if (i < nrow) {
          const int e = i * D + col;
          cluster.map_shared_rank(so, e % split)[rank * share + e / split] = acc[nt][q];
        }
      }
  } else {
  // partial o over this CTA's rows of B_v: thread = (column pair, every
  // kGroups-th row of the chunk), so each output has one owner
  constexpr int kPairs = D / 2;
  constexpr int kGroups = kThreads / kPairs;        // 4 (D = 128) or 8 (D = 64)
  constexpr int kRowsPer = kMaxRows / kGroups;      // 4 or 2
  const int cp = threadIdx.x % kPairs, ig = threadIdx.x / kPairs;
  float acc[kRowsPer][2];
#pragma unroll
  for (int q = 0; q < kRowsPer; ++q) acc[q][0] = acc[q][1] = 0.f;
  for (int r = 0; r < rr; r += 4) {
    float x0[4], x1[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const float2 xv = pair_f32(sbv + (size_t)(r + t) * ldb<T, D>() + 2 * cp);
      x0[t] = xv.x;
      x1[t] = xv.y;
    }
#pragma unroll
    for (int q = 0; q < kRowsPer; ++q) {
      const int i = ig + kGroups * q;
      if (i < nrow) {
        const float4 uv = *reinterpret_cast<const float4*>(&su[(size_t)i * ldu + r]);
        acc[q][0] = fmaf(uv.x, x0[0], fmaf(uv.y, x0[1], fmaf(uv.z, x0[2], fmaf(uv.w, x0[3], acc[q][0]))));
        acc[q][1] = fmaf(uv.x, x1[0], fmaf(uv.y, x1[1], fmaf(uv.z, x1[2], fmaf(uv.w, x1[3], acc[q][1]))));
      }
    }
  }
  // cluster-wide sum: output e = i * D + col belongs to rank e % split, which
  // receives every rank's partial in its slot [rank][e / split] (remote stores,
  // made visible by the cluster barrier), then reduces and writes its outputs
#pragma unroll
  for (int q = 0; q < kRowsPer; ++q) {
    const int i = ig + kGroups * q;
    if (i < nrow)
#pragma unroll
      for (int t = 0; t < 2; ++t) {
        const int e = i * D + 2 * cp + t;
        cluster.map_shared_rank(so, e % split)[rank * share + e / split] = acc[q][t];
      }
  }
  }
  DCK_CB_TRACE(6);
  cluster.sync();
  DCK_CB_TRACE(7);
  T* out = static_cast<T*>(a.out);
  for (int pos = threadIdx.x; pos * split < nrow * D; pos += kThreads) {
    const int e = pos * split + rank;
    if (e >= nrow * D) break;
    float v = 0.f;
    for (int q = 0; q < split; ++q) v += so[q * share + pos];
    const int i = e / D, col = e % D;
    const int b = b0 + i / qpg, j = h * qpg + i % qpg;
    out[((int64_t)b * Hq + j) * D + col] = from_f32<T>(v * sinv[i]);
  }
}

// Dynamic shared memory of one CTA for an r_v split.
template <typename T, int D>
size_t combine_smem(const LayerTable& lt, const DecodeArgs& a, int split) {
  const int rr = lt.rv / split;
  const int cap = 2 * a.n_items;
  return (size_t)rr * ldb<T, D>() * sizeof(T) +
         sizeof(float) * ((size_t)kMaxRows * (rr + 4) + kMaxRows * D + kMaxRows + 2 * (size_t)kMaxRows * cap) +
         sizeof(int) * ((size_t)kMaxRows * cap + kMaxRows + 4 * kMaxRows + kMaxRows + a.B + 1 + a.n_items + 1);
}

template <typename T, int D>
cudaLaunchConfig_t combine_config(const LayerTable& lt, const DecodeArgs& a, int split, int bchunk, size_t smem,
                                  cudaStream_t s, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(lt.Hkv * split, (a.B + bchunk - 1) / bchunk);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = split;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // may start while the previous kernel finishes (B_v staging and tables overlap it)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cfg;
}

template <typename T, int D>
cudaError_t launch_t(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  // as many sequences per cluster as its rows allow: each head's B_v block is staged once per chunk
  const int bchunk = std::max(1, std::min(a.B, kMaxRows / lt.qpg));
  const int n_clusters = lt.Hkv * ((a.B + bchunk - 1) / bchunk);
  // r_v split over a cluster of 8 CTAs where r_v allows.  Clusters of 8 CTAs
  // that need two CTAs per SM were not all placed at once (7B MHA layer, B16:
  // 30 of 32 clusters ran, the other two as a second wave that cost as much
  // as the first), so where clusters of 4 fit one CTA per SM, 4 it is.
  // (The wider r_v slice of a CTA of 4 must still fit its shared memory.)
  int split = lt.rv % (4 * kMaxSplit) == 0 ? kMaxSplit : kMaxSplit / 2;
  int dev = 0, sms = 0, smem_optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (split == kMaxSplit && n_clusters * kMaxSplit > sms && n_clusters * (kMaxSplit / 2) <= sms &&
      combine_smem<T, D>(lt, a, kMaxSplit / 2) <= (size_t)smem_optin)
    split = kMaxSplit / 2;
  auto k = combine_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)combine_smem<T, D>(lt, a, split));
  if (e != cudaSuccess) return e;
  const size_t smem = combine_smem<T, D>(lt, a, split);
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = combine_config<T, D>(lt, a, split, bchunk, smem, s, attr);
  e = cudaLaunchKernelEx(&cfg, k, lt, a, bchunk, split);
  return e != cudaSuccess ? e : hook_launched(a.hook, s);
}

}  // namespace

// r_v must split into at least four parts of whole float4 and 16-byte rows.
bool combine_supports(const LayerTable& lt) { return lt.rv % (4 * kMaxSplit / 2) == 0 && lt.rv <= kMaxRankV; }

cudaError_t launch_combine(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s) {
  if (dtype == DCK_F32) return lt.d == 64 ? launch_t<float, 64>(lt, a, s) : launch_t<float, 128>(lt, a, s);
  return lt.d == 64 ? launch_t<__nv_bfloat16, 64>(lt, a, s) : launch_t<__nv_bfloat16, 128>(lt, a, s);
}

}  // namespace dck
