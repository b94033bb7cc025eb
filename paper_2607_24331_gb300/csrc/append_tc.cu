// Tensor-core latent append (Sec. III-A z = x L, with the key factors of all
// Sec. III-C groups side by side and the Sec. III-D value factor):
//   kcache[rows[i]] = x_i A_k,   vcache[rows[i]] = x_i A_v
// as a tcgen05 GEMM, bf16 in, fp32 accumulate in TMEM, bf16 out.
//
// CTA tile 128 tokens x N_t (<= 256) columns of one of the two outputs; K in
// 64-wide stages staged by TMA (x: K-major, 128B swizzle; A: MN-major, 128B
// swizzle) through a 4-deep mbarrier ring.  Warp 0 issues TMA, warp 1 owns
// TMEM and issues tcgen05.mma, warps 2-5 drain the accumulator (one TMEM lane
// quadrant each).  Small batches (<= 256 tokens, the decode-step append) split
// K over CTAs, each storing its fp32 partial in its own slice of the caller's
// workspace; a second kernel sums the slices, rounds and scatters.  The ring
// has only as many stages as a CTA has K blocks, so split CTAs of two K blocks
// fit two to an SM and the whole split runs in one wave.
#include <algorithm>

#include "common.cuh"
#include "sm100.cuh"
#include "tmap.h"

namespace dck {
namespace {

using namespace sm100;

constexpr int kBM = 128, kBK = 64, kMaxBN = 256, kStages = 4;
constexpr int kABytes = kBM * kBK * 2;          // 16 KB
constexpr int kBBytes = kBK * kMaxBN * 2;       // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kThreads = 192;
constexpr int kSplitMaxTok = 256;
constexpr int kMaxSplit = 32;  // K splits of a small batch

struct AppendParams {
  int n_tok, D, Rk, rv;
  int nt_k;      // N tiles over the key output
  int kblocks;   // ceil(D / 64)
  int ksplit;
  int stages;    // ring depth: min(kStages, K blocks of one CTA)
  const int64_t* rows;
  __nv_bfloat16* kc;
  __nv_bfloat16* vc;
  int64_t n_rows;
  float* ws;     // split-K partials [ksplit][n_tok][Rk + rv] (ksplit > 1)
  int* err;
};

__device__ __forceinline__ void tile_of(const AppendParams& p, int t, bool& is_k, int& n0, int& nt) {
  is_k = t < p.nt_k;
  const int N = is_k ? p.Rk : p.rv;
  n0 = (is_k ? t : t - p.nt_k) * kMaxBN;
  nt = min(kMaxBN, N - n0);
}

__global__ void __launch_bounds__(kThreads, 1)
    append_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_ak,
                     const __grid_constant__ CUtensorMap tm_av, const AppendParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nst = p.stages;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + nst * kStageBytes);
  uint64_t* empty = full + kStages;
  uint64_t* acc_bar = empty + kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_bar + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  bool is_k;
  int n0, nt;
  tile_of(p, blockIdx.x, is_k, n0, nt);
  const int m0 = blockIdx.y * kBM;
  const int kb0 = (int)((int64_t)blockIdx.z * p.kblocks / p.ksplit);
  const int kb1 = (int)((int64_t)(blockIdx.z + 1) * p.kblocks / p.ksplit);
  const int nboxes = (nt + 63) / 64;

  if (threadIdx.x == 0) {
    for (int s = 0; s < nst; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_bar, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // programmatic dependent launch: the set-up above overlaps the previous
  // kernel's tail; every global access comes after that kernel is complete
  pdl_wait();
  pdl_launch_dependents();
  const uint32_t tmem = *tmem_slot;
  const CUtensorMap* tmb = is_k ? &tm_ak : &tm_av;

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_x);
    tma_prefetch_desc(tmb);
    for (int kb = kb0; kb < kb1; ++kb) {
      const int i = kb - kb0, s = i % nst;
      if (i >= nst && !mbar_wait(&empty[s], ((i / nst) - 1) & 1, abort_flag)) break;
      uint8_t* a = smem + s * kStageBytes;
      uint8_t* b = a + kABytes;
      mbar_expect_tx(&full[s], kABytes + nboxes * (kBK * 64 * 2));
      tma_load_2d(a, &tm_x, &full[s], kb * kBK, m0);
      for (int j = 0; j < nboxes; ++j) tma_load_2d(b + j * (kBK * 64 * 2), tmb, &full[s], n0 + 64 * j, kb * kBK);
    }
  } else if (warp == 1 && lane == 0) {
    const uint32_t idesc = idesc_bf16(kBM, nt, false, true);
    for (int kb = kb0; kb < kb1; ++kb) {
      const int i = kb - kb0, s = i % nst;
      if (!mbar_wait(&full[s], (i / nst) & 1, abort_flag)) break;
      tc_fence_after();
      const uint32_t a = smem_u32(smem + s * kStageBytes);
      const uint32_t b = a + kABytes;
#pragma unroll
      for (int k = 0; k < kBK / 16; ++k) {
        const uint64_t ad = sdesc(a + k * 32, 16, 1024, kSw128);
        const uint64_t bd = sdesc(b + k * 2048, kBK * 64 * 2, 1024, kSw128);
        umma_f16(tmem, ad, bd, idesc, (i > 0 || k > 0) ? 1u : 0u);
      }
      umma_commit(&empty[s]);
    }
    umma_commit(acc_bar);
  } else if (warp >= 2) {
    const int quad = warp & 3;
    const int m = m0 + quad * 32 + lane;
    const bool ok = mbar_wait(acc_bar, 0, abort_flag);
    tc_fence_after();
    int64_t row = -1;
    if (ok && m < p.n_tok && p.ksplit == 1) {
      row = p.rows[m];
      if (row < 0 || row >= p.n_rows) {
        atomicOr(p.err, kErrBadRow);
        row = -1;
      }
    }
    const int N = is_k ? p.Rk : p.rv;
    __nv_bfloat16* dst = is_k ? p.kc : p.vc;
    for (int c = 0; c < nt && ok; c += 16) {
      float v[16];
      tmem_ld16(tmem_addr(tmem, quad * 32, c), v);
      tmem_wait_ld();
      if (m >= p.n_tok) continue;
      if (p.ksplit == 1) {
        if (row >= 0) {
          uint4 pk[2];
          __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(pk);
#pragma unroll
          for (int i = 0; i < 8; ++i) h2[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
          uint4* o = reinterpret_cast<uint4*>(dst + row * N + n0 + c);
          o[0] = pk[0];
          o[1] = pk[1];
        }
      } else {
        float4* w = reinterpret_cast<float4*>(p.ws + ((int64_t)blockIdx.z * p.n_tok + m) * (p.Rk + p.rv) +
                                              (is_k ? 0 : p.Rk) + n0 + c);
#pragma unroll
        for (int i = 0; i < 4; ++i) w[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.err, kErrTimeout);
}

__global__ void append_finalize_kernel(const float* __restrict__ ws, int n_tok, int Rk, int rv, int ksplit,
                                       const int64_t* __restrict__ rows, __nv_bfloat16* kc, __nv_bfloat16* vc,
                                       int64_t n_rows, int* err) {
  pdl_wait();  // the split partials come from the kernel before
  pdl_launch_dependents();
  const int N = Rk + rv;
  const int m = blockIdx.y;
  const int64_t row = rows[m];
  if (row < 0 || row >= n_rows) {
    if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(err, kErrBadRow);
    return;
  }
  const int64_t zs = (int64_t)n_tok * N;  // stride between the splits' slices
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < N; c += gridDim.x * blockDim.x) {
    const float* w = ws + (int64_t)m * N + c;
    float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f;  // four loads in flight, summed in split order per chain
    int z = 0;
    for (; z + 4 <= ksplit; z += 4) {
      const float a0 = w[z * zs], a1 = w[(z + 1) * zs], a2 = w[(z + 2) * zs], a3 = w[(z + 3) * zs];
      v0 += a0;
      v1 += a1;
      v2 += a2;
      v3 += a3;
    }
    for (; z < ksplit; ++z) v0 += w[z * zs];
    const float v = (v0 + v1) + (v2 + v3);
    if (c < Rk) kc[row * Rk + c] = __float2bfloat16_rn(v);
    else vc[row * rv + (c - Rk)] = __float2bfloat16_rn(v);
  }
}

int plan_ksplit(int n_tok, int D, int Rk, int rv, int sms) {
  if (n_tok > kSplitMaxTok) return 1;
  const int mt = (n_tok + kBM - 1) / kBM;
  const int ntiles = (Rk + kMaxBN - 1) / kMaxBN + (rv + kMaxBN - 1) / kMaxBN;
  const int kblocks = (D + kBK - 1) / kBK;
  // up to two CTAs per SM (split CTAs of at most two K blocks take 96 KB of shared memory)
  int ks = 2 * sms / max(1, mt * ntiles);
  ks = max(1, min(ks, min(kMaxSplit, kblocks)));
  return ks;
}

}  // namespace

bool tc_append_supports(int D, int Rk, int rv, int dtype) {
  return dtype == DCK_BF16 && D % 8 == 0 && Rk % 16 == 0 && rv % 16 == 0;
}

size_t tc_append_workspace(int n_tok, int Rk, int rv) {
  return n_tok <= kSplitMaxTok ? align_up((size_t)kMaxSplit * n_tok * (Rk + rv) * sizeof(float), 256) : 0;
}

cudaError_t launch_append_tc(const void* x, int n_tok, int D, const void* A_k, const void* A_v, int Rk, int rv,
                             const int64_t* rows, void* kc, void* vc, int64_t n_rows, void* ws, size_t ws_bytes,
                             int* err, cudaStream_t s, int* n_launches) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  AppendParams p;
  p.n_tok = n_tok;
  p.D = D;
  p.Rk = Rk;
  p.rv = rv;
  p.nt_k = (Rk + kMaxBN - 1) / kMaxBN;
  p.kblocks = (D + kBK - 1) / kBK;
  p.ksplit = plan_ksplit(n_tok, D, Rk, rv, sms);
  p.stages = std::min(kStages, (p.kblocks + p.ksplit - 1) / p.ksplit);
  p.rows = rows;
  p.kc = static_cast<__nv_bfloat16*>(kc);
  p.vc = static_cast<__nv_bfloat16*>(vc);
  p.n_rows = n_rows;
  p.ws = static_cast<float*>(ws);
  p.err = err;
  if (n_tok <= kSplitMaxTok && (!ws || ws_bytes < tc_append_workspace(n_tok, Rk, rv))) return cudaErrorInvalidValue;
  CUtensorMap tx, tk, tv;
  if (!make_tmap_2d_bf16(&tx, x, D, n_tok, (uint64_t)D * 2, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_2d_bf16(&tk, A_k, Rk, D, (uint64_t)Rk * 2, 64, kBK, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_2d_bf16(&tv, A_v, rv, D, (uint64_t)rv * 2, 64, kBK, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  const int ntiles = p.nt_k + (rv + kMaxBN - 1) / kMaxBN;
  const size_t smem = (size_t)p.stages * kStageBytes + 1024 + 256;
  // the attribute is an upper bound for every launch (prefill uses all kStages stages)
  cudaError_t e = cudaFuncSetAttribute(append_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(kStages * kStageBytes + 1024 + 256));
  if (e != cudaSuccess) return e;
  dim3 grid(ntiles, (n_tok + kBM - 1) / kBM, p.ksplit);
  *n_launches = p.ksplit > 1 ? 2 : 1;
  e = launch_pdl(append_tc_kernel, grid, dim3(kThreads), smem, s, tx, tk, tv, p);
  if (e != cudaSuccess || p.ksplit == 1) return e;
  dim3 g2((Rk + rv + 255) / 256, n_tok);
  return launch_pdl(append_finalize_kernel, g2, dim3(256), 0, s, (const float*)p.ws, n_tok, Rk, rv, p.ksplit, rows,
                    p.kc, p.vc, n_rows, err);
}

}  // namespace dck
