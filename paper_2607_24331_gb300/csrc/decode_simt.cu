// CUDA-core decode attention over the DynaCalKV latent caches.
//
// The general kernel: any head_dim in {64, 128}, fp32 or bf16 storage, fp32
// arithmetic with fp64 RoPE angles.  It is the kernel for fp32 layers (whose
// 1e-5 tolerance tensor-core bf16/tf32 products cannot meet) and for shapes the
// tensor-core kernel does not take.
//
// Block (item c, KV head h): for every sequence segment in item c's tile
// range, 32-token chunks are processed as
//   k_t = c_t^g B_g[:, slot(h)]        (Sec. III-A/III-C reconstruction)
//   RoPE(k_t, t); scores against RoPE(q_j, L-1) / sqrt(d) for the query heads
//   of h; online softmax in log2 units;
//   u_j += p_t v_t                      (value latent, Sec. III-D; B_v is
//                                        applied once after the split merge)
// and the segment's (u_j, m_j, l_j) is written to partial slot c + b.
#include "common.cuh"

namespace dck {
namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 32;
constexpr int kMaxRankK = 256;  // per-group rank handled by this kernel
constexpr float kLog2e = 1.4426950408889634f;

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) decode_simt_kernel(const LayerTable lt, const DecodeArgs a) {
  extern __shared__ float smem[];
  const int c = blockIdx.x;
  const int h = blockIdx.y;
  const int tid = threadIdx.x;
  const int B = a.B;

  int* prefix = reinterpret_cast<int*>(smem);           // [B+1]
  int* scan = prefix + (B + 1);                          // [kThreads]
  float* fbase = reinterpret_cast<float*>(scan + kThreads);
  float* sq = fbase;                                     // [qpg][D] rotated, scaled queries
  float* sC = sq + kMaxQPerKv * D;                       // [kChunk][r]
  float* sK = sC + kChunk * kMaxRankK;                   // [kChunk][D]
  float* sP = sK + kChunk * D;                           // [qpg][kChunk]
  float* sAlpha = sP + kMaxQPerKv * kChunk;              // [qpg]

  const int NT = build_tile_prefix(a.seq_len, a.seq_start, B, a.n_rows, prefix, scan, a.err,
                                   c == 0 && h == 0);
  const int x0 = item_begin(c, NT, a.n_items);
  const int x1 = item_begin(c + 1, NT, a.n_items);
  if (x0 >= x1) return;

  const int g = lt.head_group[h];
  const int slot = lt.head_slot[h];
  const int r = lt.grp_rank[g];
  const int roff = lt.grp_roff[g];
  const int ng = lt.grp_nh[g];
  const int qpg = lt.qpg;
  const int rv = lt.rv;
  const int Rk = lt.Rk;
  const T* __restrict__ kc = static_cast<const T*>(a.kc);
  const T* __restrict__ vc = static_cast<const T*>(a.vc);
  const T* __restrict__ Bg = static_cast<const T*>(a.Bk) + lt.grp_boff[g] + (int64_t)slot * D;
  const int64_t bg_ld = (int64_t)ng * D;
  const double log2_theta = log2((double)a.theta);

  constexpr int TG = kThreads / D;          // token groups in the reconstruction
  constexpr int TPT = kChunk / TG;          // tokens per thread
  const int e = tid % D;
  const int tg = tid / D;
  const int warp = tid >> 5, lane = tid & 31;
  constexpr int kRvPerThread = kMaxRankV / kThreads;

  for (int x = x0; x < x1;) {
    const int b = seq_of_tile(prefix, B, x);
    const int seg_end_tile = min(x1, prefix[b + 1]);
    const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
    const int64_t row0 = a.seq_start[b];
    const int t_begin = (x - prefix[b]) * kTile;
    const int t_end = min(L, (seg_end_tile - prefix[b]) * kTile);
    x = seg_end_tile;

    // rotated, scaled query heads of this KV head (position L-1)
    const int P = L - 1;
    const float qscale = rsqrtf((float)D) * kLog2e;
    for (int i = tid; i < qpg * (D / 2); i += kThreads) {
      const int jj = i / (D / 2), p = i % (D / 2);
      const int j = h * qpg + jj;
      const T* qp = static_cast<const T*>(a.q) + ((int64_t)b * lt.Hq + j) * D;
      const double ang = (double)P * exp2(-2.0 * p / D * log2_theta);
      double sn, cs;
      sincos(ang, &sn, &cs);
      const float x1v = to_f32(qp[p]), x2v = to_f32(qp[p + D / 2]);
      sq[jj * D + p] = (float)(x1v * cs - x2v * sn) * qscale;
      sq[jj * D + p + D / 2] = (float)(x1v * sn + x2v * cs) * qscale;
    }
    float acc[kMaxQPerKv][kRvPerThread];
#pragma unroll
    for (int jj = 0; jj < kMaxQPerKv; ++jj)
#pragma unroll
      for (int k = 0; k < kRvPerThread; ++k) acc[jj][k] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;  // meaningful in warp jj (lane 0) for jj < qpg
    __syncthreads();

    for (int t0 = t_begin; t0 < t_end; t0 += kChunk) {
      const int nt = min(kChunk, t_end - t0);
      // latent chunk of group g
      for (int i = tid; i < kChunk * r; i += kThreads) {
        const int t = i / r, k = i % r;
        sC[t * r + k] = t < nt ? to_f32(kc[(row0 + t0 + t) * Rk + roff + k]) : 0.f;
      }
      __syncthreads();
      // reconstruction k_t[e] = sum_k c_t[k] B_g[k][slot*D + e]
      float kacc[TPT];
#pragma unroll
      for (int u = 0; u < TPT; ++u) kacc[u] = 0.f;
      for (int k = 0; k < r; ++k) {
        const float bv = to_f32(Bg[(int64_t)k * bg_ld + e]);
#pragma unroll
        for (int u = 0; u < TPT; ++u) kacc[u] = fmaf(sC[(tg + u * TG) * r + k], bv, kacc[u]);
      }
#pragma unroll
      for (int u = 0; u < TPT; ++u) sK[(tg + u * TG) * D + e] = kacc[u];
      __syncthreads();
      // RoPE on the chunk's keys, pair (p, p + D/2), angle t * omega_p in fp64
      for (int i = tid; i < kChunk * (D / 2); i += kThreads) {
        const int t = i / (D / 2), p = i % (D / 2);
        const double ang = (double)(t0 + t) * exp2(-2.0 * p / D * log2_theta);
        double sn, cs;
        sincos(ang, &sn, &cs);
        const float k1 = sK[t * D + p], k2 = sK[t * D + p + D / 2];
        sK[t * D + p] = (float)(k1 * cs - k2 * sn);
        sK[t * D + p + D / 2] = (float)(k1 * sn + k2 * cs);
      }
      __syncthreads();
      // scores (log2 units), one warp per (query head, token) pair
      for (int pr = warp; pr < qpg * kChunk; pr += kThreads / 32) {
        const int jj = pr / kChunk, t = pr % kChunk;
        float s = 0.f;
        for (int i = lane; i < D; i += 32) s = fmaf(sq[jj * D + i], sK[t * D + i], s);
#pragma unroll
        for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) sP[jj * kChunk + t] = t < nt ? s : -INFINITY;
      }
      __syncthreads();
      // online softmax: warp jj owns query head jj
      if (warp < qpg) {
        const float s = sP[warp * kChunk + lane];
        float mx = s;
#pragma unroll
        for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        const float m_new = fmaxf(m_run, mx);
        const float alpha = exp2f(m_run - m_new);  // 0 on the first chunk
        const float p = exp2f(s - m_new);
        float ps = p;
#pragma unroll
        for (int o = 16; o; o >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, o);
        l_run = l_run * alpha + ps;
        m_run = m_new;
        sP[warp * kChunk + lane] = p;
        if (lane == 0) sAlpha[warp] = alpha;
      }
      __syncthreads();
      // u_j = alpha u_j + sum_t p_t v_t
#pragma unroll
      for (int k = 0; k < kRvPerThread; ++k) {
        const int rr = tid + k * kThreads;
        if (rr < rv) {
          float vs[kChunk];
#pragma unroll 8
          for (int t = 0; t < kChunk; ++t) vs[t] = t < nt ? to_f32(vc[(row0 + t0 + t) * rv + rr]) : 0.f;
#pragma unroll
          for (int jj = 0; jj < kMaxQPerKv; ++jj) {
            if (jj < qpg) {
              float s = acc[jj][k] * sAlpha[jj];
#pragma unroll 8
              for (int t = 0; t < kChunk; ++t) s = fmaf(sP[jj * kChunk + t], vs[t], s);
              acc[jj][k] = s;
            }
          }
        }
      }
      __syncthreads();
    }
    // partial of (item c, sequence b) -> slot c + b
    const int64_t slot_id = (int64_t)c + b;
#pragma unroll
    for (int jj = 0; jj < kMaxQPerKv; ++jj) {
      if (jj < qpg) {
        const int j = h * qpg + jj;
        float* pu = a.part_u + (slot_id * lt.Hq + j) * (int64_t)rv;
#pragma unroll
        for (int k = 0; k < kRvPerThread; ++k) {
          const int rr = tid + k * kThreads;
          if (rr < rv) pu[rr] = acc[jj][k];
        }
      }
    }
    if (warp < qpg && lane == 0) {
      const int j = h * qpg + warp;
      float* pm = a.part_ml + (slot_id * lt.Hq + j) * 2;
      pm[0] = t_end > t_begin ? m_run : -INFINITY;
      pm[1] = l_run;
    }
    __syncthreads();
  }
}

template <typename T, int D>
cudaError_t launch_t(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(int) * (a.B + 1 + kThreads) +
                      sizeof(float) * (kMaxQPerKv * D + kChunk * kMaxRankK + kChunk * D +
                                       kMaxQPerKv * kChunk + kMaxQPerKv);
  auto k = decode_simt_kernel<T, D>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.n_items, lt.Hkv);
  if ((e = hook_begin(a.hook, s)) != cudaSuccess) return e;
  k<<<grid, kThreads, smem, s>>>(lt, a);
  return hook_launched(a.hook, s);
}

}  // namespace

bool simt_supports(const LayerTable& lt) {
  if (lt.d != 64 && lt.d != 128) return false;
  if (lt.qpg > kMaxQPerKv || lt.rv > kMaxRankV) return false;
  for (int g = 0; g < lt.G; ++g)
    if (lt.grp_rank[g] > kMaxRankK) return false;
  return true;
}

cudaError_t launch_decode_simt(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s) {
  if (dtype == DCK_F32) return lt.d == 64 ? launch_t<float, 64>(lt, a, s) : launch_t<float, 128>(lt, a, s);
  return lt.d == 64 ? launch_t<__nv_bfloat16, 64>(lt, a, s) : launch_t<__nv_bfloat16, 128>(lt, a, s);
}

}  // namespace dck
