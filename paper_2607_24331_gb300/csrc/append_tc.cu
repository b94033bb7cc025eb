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
// fit two to an SM and the whole split runs in one wave.  Longer appends (a
// prefill) with R_k and r_v multiples of 64 run on persistent CTA pairs
// (append_pair_kernel below).
#include <algorithm>
#include <cstring>

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
  const int64_t* rows;  // cache row of each token (pair kernel: null writes token m to row m)
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

// ---------------------------------------------------------------------------
// Long appends (prefill): persistent CTA pairs.
//
// A pair tile covers 256 tokens (128 per CTA, its rows of the UMMA operand A:
// x) and w = 128 or 256 output columns of one of the two outputs (each CTA
// holding w/2 columns of operand B: A_k or A_v), the whole of K = D in 64-wide
// stages, one tcgen05 pair MMA (cta_group::2, M = 256) per 16 of K.  Per stage
// and CTA the operands are 16 KB of x and w/2 x 64 x 2 bytes of factor: at
// w = 256, 32 KB per 512 cycles of pair MMA, where the single-CTA tile of
// 128 x 256 above streams 48 KB per 512 cycles, more than an SM takes in from
// L2.  Tiles, flattened: for every 256-token block, the key output in
// 256-column tiles (the last one 128 wide when at most 128 columns remain;
// columns past R_k load as zeros and are not stored), then the value output
// likewise.  Pair p takes tiles p, p + P, p + 2P, ... of that list.  Two
// 256-column TMEM accumulators: the epilogue of one tile overlaps the next
// tile's MMAs.
// ---------------------------------------------------------------------------

constexpr int kPStages = 6;
constexpr int kPXBytes = kBM * kBK * 2;      // 16 KB: this CTA's 128 token rows x 64 of K
constexpr int kPBBytes = 2 * kBK * 64 * 2;   // 16 KB: up to 128 factor columns x 64 of K (64-column boxes)
constexpr int kPStageBytes = kPXBytes + kPBBytes;
constexpr int kPThreads = 192;
constexpr int kPRows = 2 * kBM;              // tokens of a pair tile
constexpr uint32_t kPTmemCols = 512;

// Pair tiles of one output of width N (a multiple of 64): 256-column tiles,
// the last one 128 wide when at most 128 columns remain.
__host__ __device__ inline int pt_count(int N) { return (N + 255) / 256; }
__host__ __device__ inline int pt_width(int N, int j) {
  return j + 1 < pt_count(N) || N - 256 * j > 128 ? 256 : 128;
}
struct PairTile {
  int m0;    // first token
  int out;   // 0: key output, 1: value output
  int n0;    // first output column
  int w;     // columns (128 or 256)
};

struct PairPlan {
  int tk, trow;  // key tiles, tiles of a 256-token block
  __device__ PairPlan(int Rk, int rv) : tk(pt_count(Rk)), trow(pt_count(Rk) + pt_count(rv)) {}
  __device__ PairTile tile(int64_t t, int Rk, int rv) const {
    const int64_t mt = t / trow;
    const int j = (int)(t - mt * trow);
    PairTile pt;
    pt.m0 = (int)(mt * kPRows);
    pt.out = j < tk ? 0 : 1;
    const int jj = pt.out ? j - tk : j;
    pt.n0 = 256 * jj;
    pt.w = pt_width(pt.out ? rv : Rk, jj);
    return pt;
  }
};

__global__ void __launch_bounds__(kPThreads, 1)
    append_pair_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_ak,
                       const __grid_constant__ CUtensorMap tm_av, const AppendParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kPStages * kPStageBytes);
  uint64_t* empty = full + kPStages;
  uint64_t* acc_full = empty + kPStages;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hr = (int)cluster_ctarank();  // this CTA's half of every pair tile
  const bool leader = hr == 0;            // the even CTA issues the pair MMAs
  const int P = gridDim.x / 2, pair = blockIdx.x >> 1;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kPStages; ++s) {
      mbar_init(&full[s], 1);   // even CTA: its producer's expect_tx; both CTAs' copies complete on it
      mbar_init(&empty[s], 1);  // the pair MMAs' commit, in both CTAs
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 8);  // even CTA: the four epilogue warps of both CTAs
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, kPTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  pdl_wait();
  pdl_launch_dependents();
  const uint32_t tmem = *tmem_slot;
  auto lead = [](const void* q) { return mapa_shared(smem_u32(q), 0); };
  auto stop_peer = [&]() { st_cluster_u32(mapa_shared(smem_u32((const void*)abort_flag), (uint32_t)(hr ^ 1)), 1u); };

  const PairPlan plan(p.Rk, p.rv);
  const int64_t n_mt = (p.n_tok + kPRows - 1) / kPRows;
  const int64_t n_tiles = n_mt * plan.trow;
  // pair p takes tiles p, p + P, p + 2P, ...: at any time the pairs work on P
  // consecutive tiles, the column tiles of a few token blocks, so a block's x
  // is read from HBM once and from L2 by the pairs of its other column tiles
  // (contiguous ranges per pair re-read x from HBM for every column tile:
  // 76 pairs' x blocks of 2 MB do not stay in L2 together)
  const int64_t t0 = pair, t1 = n_tiles, tstep = P;
  const int kb_n = p.kblocks;

  if (warp == 0) {
    // ---- TMA producer (both CTAs): this CTA's x rows and its half of the factor columns
    if (lane == 0) {
      tma_prefetch_desc(&tm_x);
      tma_prefetch_desc(&tm_ak);
      tma_prefetch_desc(&tm_av);
      uint64_t pol_x, pol_a;
      asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol_x));
      pol_a = policy_evict_last();
      int64_t it = 0;
      bool ok = true;
      for (int64_t t = t0; t < t1 && ok; t += tstep) {
        const PairTile pt = plan.tile(t, p.Rk, p.rv);
        const CUtensorMap* tb = pt.out ? &tm_av : &tm_ak;
        const int half = pt.w / 2, nbx = half / 64;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = (int)(it % kPStages);
          if (it >= kPStages && !(ok = mbar_wait(&empty[s], (uint32_t)(((it / kPStages) - 1) & 1), abort_flag))) break;
          uint8_t* xs = smem + s * kPStageBytes;
          uint8_t* bs = xs + kPXBytes;
          if (leader) mbar_expect_tx(&full[s], 2u * (uint32_t)(kPXBytes + nbx * kBK * 64 * 2));
          tma_load_2d_pair(xs, &tm_x, lead(&full[s]), kb * kBK, pt.m0 + hr * kBM, pol_x);
          for (int bx = 0; bx < nbx; ++bx)
            tma_load_2d_pair(bs + bx * (kBK * 64 * 2), tb, lead(&full[s]), pt.n0 + hr * half + 64 * bx, kb * kBK,
                             pol_a);
        }
      }
      if (!ok) stop_peer();
    }
  } else if (warp == 1) {
    // ---- pair MMAs (even CTA, one thread) -------------------------------------
    if (leader && lane == 0) {
      int64_t it = 0;
      bool ok = true;
      int lt = 0;  // tiles of this pair so far
      for (int64_t t = t0; t < t1 && ok; t += tstep, ++lt) {
        const PairTile pt = plan.tile(t, p.Rk, p.rv);
        const int buf = lt & 1;
        if (lt >= 2 && !(ok = mbar_wait(&acc_empty[buf], (uint32_t)(((lt >> 1) - 1) & 1), abort_flag))) break;
        tc_fence_after();
        const uint32_t idesc = idesc_bf16(kPRows, pt.w, false, true);
        const uint32_t d = tmem + buf * 256;
        for (int kb = 0; kb < kb_n; ++kb, ++it) {
          const int s = (int)(it % kPStages);
          if (!(ok = mbar_wait(&full[s], (uint32_t)((it / kPStages) & 1), abort_flag))) break;
          tc_fence_after();
          const uint32_t xa = smem_u32(smem + s * kPStageBytes);
          const uint32_t ba = xa + kPXBytes;
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k) {
            const uint64_t ad = sdesc(xa + k * 32, 16, 1024, kSw128);
            const uint64_t bd = sdesc(ba + k * 2048, kBK * 64 * 2, 1024, kSw128);
            umma_f16_pair(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          }
          umma_commit_pair(&empty[s]);  // the stage's slots in both CTAs, once these MMAs are done
        }
        if (ok) umma_commit_pair(&acc_full[buf]);
      }
      if (!ok) stop_peer();
    }
    __syncwarp();
  } else {
    // ---- epilogue (warps 2-5, both CTAs): this CTA's 128 rows of each tile -----
    const int quad = warp & 3;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    int lt = 0;
    bool ok = true;
    for (int64_t t = t0; t < t1 && ok; t += tstep, ++lt) {
      const PairTile pt = plan.tile(t, p.Rk, p.rv);
      const int buf = lt & 1;
      ok = mbar_wait(&acc_full[buf], (uint32_t)((lt >> 1) & 1), abort_flag);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const int m = pt.m0 + hr * kBM + quad * 32 + lane;
      int64_t row = -1;
      if (m < p.n_tok) {
        row = p.rows ? p.rows[m] : m;
        if (row < 0 || row >= p.n_rows) {
          atomicOr(p.err, kErrBadRow);
          row = -1;
        }
      }
      const int N = pt.out ? p.rv : p.Rk;
      __nv_bfloat16* dst = pt.out ? p.vc : p.kc;
      for (int c = 0; c < pt.w; c += 32) {
        float v[32];
        tmem_ld32(tmem + lane_base + buf * 256 + c, v);
        tmem_wait_ld();
        if (row >= 0 && pt.n0 + c < N) {  // N and n0 are multiples of 64: a 32-column chunk is all in or all out
          uint4 pk[4];
          __nv_bfloat162* h2 = reinterpret_cast<__nv_bfloat162*>(pk);
#pragma unroll
          for (int i = 0; i < 16; ++i) h2[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
          uint4* o = reinterpret_cast<uint4*>(dst + row * N + pt.n0 + c);
#pragma unroll
          for (int i = 0; i < 4; ++i) o[i] = pk[i];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(&acc_empty[buf]);
        else mbar_arrive_cluster(lead(&acc_empty[buf]));
      }
    }
    if (!ok && lane == 0) stop_peer();
  }
  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // let copies and MMAs already in flight land before the memory is released
    const long long c0 = clock64();
    while (clock64() - c0 < 4000000ll) {
    }
    if (threadIdx.x == 0) atomicOr(p.err, kErrTimeout);
  }
  cluster_sync();  // the peer no longer reads this CTA's operands or arrives on its barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kPTmemCols);
  }
}

// CTA pairs of the pair kernel that fit the device at once (one CTA per SM).
int append_pairs_of_device(size_t smem) {
  static int cache[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (cache[dev]) return cache[dev];
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (sms / 2));
  cfg.blockDim = dim3(kPThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, append_pair_kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 0;
  }
  cache[dev] = std::min(n, sms / 2);
  return cache[dev];
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

// C[M x N] = A[M x K] B[K x N] (bf16 row-major, fp32 accumulation, bf16
// out) on the persistent CTA pairs of the long append, for N a multiple of 64:
// the prefill's value reconstruction V^ = C_v B_v.  Returns
// cudaErrorNotSupported when the pair kernel cannot run on this device.
cudaError_t launch_gemm_pair(const void* A, int64_t M, int K, const void* Bm, int N, void* C, int* err,
                             cudaStream_t s) {
  if (M <= 0 || K <= 0 || N <= 0 || N % 64 || K % 8 || M >= (int64_t(1) << 31)) return cudaErrorInvalidValue;
  AppendParams p;
  std::memset(&p, 0, sizeof(p));
  p.n_tok = (int)M;
  p.D = K;
  p.Rk = N;
  p.rv = 0;
  p.kblocks = (K + kBK - 1) / kBK;
  p.ksplit = 1;
  p.rows = nullptr;  // row m of C is output row m
  p.kc = static_cast<__nv_bfloat16*>(C);
  p.vc = nullptr;
  p.n_rows = M;
  p.err = err;
  CUtensorMap ta, tb;
  if (!make_tmap_2d_bf16(&ta, A, K, M, (uint64_t)K * 2, kBK, kBM, CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_tmap_2d_bf16(&tb, Bm, N, K, (uint64_t)N * 2, 64, kBK, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  const size_t psmem = (size_t)kPStages * kPStageBytes + 1024 + 256;
  cudaError_t e = cudaFuncSetAttribute(append_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)psmem);
  if (e != cudaSuccess) return e;
  const int pairs = append_pairs_of_device(psmem);
  if (pairs <= 0) return cudaErrorNotSupported;
  const int64_t tiles = (M + kPRows - 1) / kPRows * pt_count(N);
  const int P = (int)std::min<int64_t>(pairs, tiles);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * P);
  cfg.blockDim = dim3(kPThreads);
  cfg.dynamicSmemBytes = psmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, append_pair_kernel, ta, tb, tb, p);
}

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
  if (n_tok > kSplitMaxTok && Rk % 64 == 0 && rv % 64 == 0) {
    // long append: persistent CTA pairs over 256-token x 256-column tiles
    const size_t psmem = (size_t)kPStages * kPStageBytes + 1024 + 256;
    cudaError_t e = cudaFuncSetAttribute(append_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)psmem);
    if (e != cudaSuccess) return e;
    const int pairs = append_pairs_of_device(psmem);
    if (pairs > 0) {
      const int64_t n_mt = (n_tok + kPRows - 1) / kPRows;
      const int64_t tiles = n_mt * (pt_count(Rk) + pt_count(rv));
      const int P = (int)std::min<int64_t>(pairs, tiles);
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(2 * P);
      cfg.blockDim = dim3(kPThreads);
      cfg.dynamicSmemBytes = psmem;
      cfg.stream = s;
      cudaLaunchAttribute attr[2];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 2;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
      attr[1].val.programmaticStreamSerializationAllowed = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 2;
      *n_launches = 1;
      return cudaLaunchKernelEx(&cfg, append_pair_kernel, tx, tk, tv, p);
    }
  }
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
