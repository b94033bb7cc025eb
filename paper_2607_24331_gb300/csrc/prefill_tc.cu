// Prefill attention over DynaCalKV latent caches on the tensor cores (bf16).
//
// Prefill is decode with many queries per sequence: the Q_b new tokens of
// sequence b are the last Q_b rows of its cache and the i-th of them, at
// position p_i = L_b - Q_b + i, attends causally to the keys at positions
// 0 .. p_i.  Keys and values are rebuilt from the latents as in decode
// (Sec. III-A x W ~ z R; Sec. III-C one factorisation per head group;
// Sec. III-D one value factorisation for all heads), here once per cache row
// for all of a sequence's queries, as two dense GEMM chains:
//
//  1. recon_kernel: for every 128-row tile of every sequence and every KV
//     head h, K^_h = RoPE(C_g B_g[:, slot(h)]) at the rows' positions and
//     V^_h = C_v B_v[:, h d : (h+1) d] (tcgen05.mma M = 128 rows, N = 128,
//     K = r_g or r_v in TMA-staged pieces, fp32 in TMEM), written as bf16 to
//     the workspace [n_rows][Hkv][d] (keys) and [n_rows][Hkv][d] (values);
//     the values, where the cache rows are mostly in use, instead as one GEMM
//     V^ = C_v B_v over all rows on the pair kernel of append_tc.cu;
//  2. attn_kernel: causal flash attention over them, one CTA per 128 query
//     rows of one KV head (the qpg query heads of a KV head packed into the
//     rows: row r = query index r / qpg, head r % qpg), S = Q^ K^T and
//     O += P V^ on the tensor cores (M = 128 rows, N = 128, K = 128 / 128
//     keys), online softmax in log2 units with a lazy reference max (O in
//     TMEM is rescaled only when a tile's max exceeds it by 8).
//
// Every wait is bounded; on expiry the CTA records kErrTimeout, waits for
// work in flight and still releases TMEM.
#include <algorithm>
#include <cmath>
#include <cstring>

#include "tc_common.cuh"
#include "tmap.h"

namespace dck {

// C[M x N] = A[M x K] B[K x N], bf16 row-major, fp32 accumulation, on the
// persistent CTA pairs of the long latent append (append_tc.cu).
cudaError_t launch_gemm_pair(const void* A, int64_t M, int K, const void* Bm, int N, void* C, int* err,
                             cudaStream_t s);

namespace {

using namespace sm100;
using namespace tc;

constexpr int kPD = 128;               // head dim of the tensor-core prefill
constexpr int kRThreads = 192;         // recon: warp 0 TMA, warp 1 MMA/TMEM, warps 2-5 epilogue
constexpr int kRStages = 4;
constexpr int kRASlot = 16384;         // latent piece [128 rows][<= 64] bf16
constexpr int kRBSlot = 16384;         // factor piece [<= 64 ranks][128 cols] as two 64-column atoms
constexpr int kMaxGroupsP = 16;
constexpr float kTwoPiP = 6.28318530717958647692f;
constexpr float kInvTwoPiP = 0.15915494309189533577f;

// ---------------------------------------------------------------------------
// 1. reconstruction
// ---------------------------------------------------------------------------

struct RMaps {
  CUtensorMap kc64, kc32, kc16;  // key latents: box {w, 128 rows}, 128/64/32B swizzle
  CUtensorMap vc64, vc32, vc16;  // value latents
  CUtensorMap bv;                // B_v [r_v][Hkv d]: box {64 cols, 16 rows}, 128B swizzle
  CUtensorMap bk[kMaxGroupsP];   // B_g [r_g][n_g d]: box {64 cols, 16 rows}, 128B swizzle
};

struct RArgs {
  const int64_t* seq_start;
  const int32_t* seq_len;
  int64_t n_rows;
  int B, Hkv, G, Rk, rv, max_len;
  int grp_roff[kMaxGroupsP], grp_rank[kMaxGroupsP];
  int head_group[128], head_slot[128];
  double om[kPD / 2];
  __nv_bfloat16* kw;  // [n_rows][Hkv][d]
  __nv_bfloat16* vw;  // [n_rows][Hkv][d]
  int* err;
};

struct RSmem {
  uint8_t a[kRStages][kRASlot];
  uint8_t b[kRStages][kRBSlot];
  float beta[kPD / 2], om32[kPD / 2];  // RoPE: (t0 w_i) mod 2 pi of the tile's first row, and w_i
  uint64_t full[kRStages], empty[kRStages], acc;
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ uint32_t swz_w(int w) { return w == 64 ? kSw128 : (w == 32 ? kSw64 : kSw32); }
__device__ __forceinline__ int piece_w(int left) { return left >= 64 ? 64 : (left >= 32 ? 32 : 16); }

// grid (row tiles of the longest sequence, B, 2 Hkv): blockIdx.z < Hkv -> keys of head z, else values of head z - Hkv
__global__ void __launch_bounds__(kRThreads, 1)
    recon_kernel(const __grid_constant__ RMaps maps, const __grid_constant__ RArgs ra) {
  extern __shared__ uint8_t smem_raw[];
  RSmem& sm = *reinterpret_cast<RSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  const int b = blockIdx.y;
  const bool is_v = (int)blockIdx.z >= ra.Hkv;
  const int h = is_v ? blockIdx.z - ra.Hkv : blockIdx.z;
  const int L = valid_len(ra.seq_len, ra.seq_start, b, ra.n_rows);
  const int t0 = blockIdx.x * kTile;  // first position of the tile
  // whole CTA, before any barrier or TMEM is set up; a sequence longer than the
  // launch's bound is left to the attention kernel, which reports it
  if (t0 >= L || L > ra.max_len) return;
  const int64_t row0 = ra.seq_start[b] + t0;
  const int g = ra.head_group[h];
  const int K = is_v ? ra.rv : ra.grp_rank[g];
  const int kcol0 = is_v ? 0 : ra.grp_roff[g];                 // first latent column
  const int bcol0 = is_v ? h * kPD : ra.head_slot[h] * kPD;    // first factor column
  const CUtensorMap* bmap = is_v ? &maps.bv : &maps.bk[g];
  if (tid == 0) {
    for (int s = 0; s < kRStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    mbar_init(&sm.acc, 1);
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  // RoPE angle of row t0 + r and pair i: (t0 w_i reduced mod 2 pi in fp64, once
  // per tile) + r w_i in fp32; the fp64 work stays off the per-row path
  if (!is_v && tid < kPD / 2) {
    const double ang = (double)t0 * ra.om[tid];
    sm.beta[tid] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
    sm.om32[tid] = (float)ra.om[tid];
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 128);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int n = 0;
      for (int k0 = 0; k0 < K; ++n) {
        const int w = piece_w(K - k0), s = n % kRStages;
        if (n >= kRStages && !mbar_wait(&sm.empty[s], ((n / kRStages) - 1) & 1, abort_flag)) break;
        // latent piece [128 rows][w] + factor rows [w][128 columns] (two 64-column atoms, 16-row boxes)
        mbar_expect_tx(&sm.full[s], kTile * w * 2 + w * kPD * 2);
        const CUtensorMap* am = is_v ? (w == 64 ? &maps.vc64 : (w == 32 ? &maps.vc32 : &maps.vc16))
                                     : (w == 64 ? &maps.kc64 : (w == 32 ? &maps.kc32 : &maps.kc16));
        tma_load_2d_hint(sm.a[s], am, &sm.full[s], kcol0 + k0, (int32_t)row0, pol);
        for (int half = 0; half < 2; ++half)
          for (int r = 0; r < w; r += 16)
            tma_load_2d(sm.b[s] + half * (w * 128) + r * 128, bmap, &sm.full[s], bcol0 + 64 * half, k0 + r);
        k0 += w;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, kPD, false, true);
      int n = 0;
      bool ok = true;
      for (int k0 = 0; k0 < K && ok; ++n) {
        const int w = piece_w(K - k0), s = n % kRStages;
        if (!(ok = mbar_wait(&sm.full[s], (n / kRStages) & 1, abort_flag))) break;
        tc_fence_after();
        const uint32_t ab = smem_u32(sm.a[s]), bb = smem_u32(sm.b[s]);
        for (int k = 0; k < w / 16; ++k)
          umma_f16(tmem, sdesc(ab + k * 32, 16, 16 * w, swz_w(w)), sdesc(bb + k * 2048, 128 * w, 1024, kSw128), idesc,
                   (k0 > 0 || k > 0) ? 1u : 0u);
        umma_commit(&sm.empty[s]);
        k0 += w;
      }
      umma_commit(&sm.acc);
    }
  } else {
    // epilogue: thread = row of the tile (TMEM lane); RoPE for keys; bf16 to the workspace
    const int quad = warp & 3, r = quad * 32 + lane;
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.acc, 0, abort_flag));
    const int pos = t0 + r;
    if (ok) {
      tc_fence_after();
      __nv_bfloat16* dst = (is_v ? ra.vw : ra.kw) + ((row0 + r) * ra.Hkv + h) * kPD;
      // frequency pairs (i, i + 64): columns [cc, cc + 32) with [64 + cc, 64 + cc + 32)
#pragma unroll
      for (int cc = 0; cc < kPD / 2; cc += 32) {
        float x[32], y[32];
        tmem_ld32(tmem + ((uint32_t)(quad * 32) << 16) + cc, x);
        tmem_ld32(tmem + ((uint32_t)(quad * 32) << 16) + kPD / 2 + cc, y);
        tmem_wait_ld();
        if (!is_v) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            // angle (t0 w_i mod 2 pi) + r w_i, reduced to [-pi, pi] in fp32
            float ph = fmaf((float)r, sm.om32[cc + i], sm.beta[cc + i]);
            ph = fmaf(-kTwoPiP, rintf(ph * kInvTwoPiP), ph);
            float sn, cs;
            sincosf(ph, &sn, &cs);
            const float xr = x[i] * cs - y[i] * sn, yr = x[i] * sn + y[i] * cs;
            x[i] = xr;
            y[i] = yr;
          }
        }
        if (pos < L)
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            uint4 ox, oy;
            __nv_bfloat162* px = reinterpret_cast<__nv_bfloat162*>(&ox);
            __nv_bfloat162* py = reinterpret_cast<__nv_bfloat162*>(&oy);
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              px[t] = __floats2bfloat162_rn(x[8 * c + 2 * t], x[8 * c + 2 * t + 1]);
              py[t] = __floats2bfloat162_rn(y[8 * c + 2 * t], y[8 * c + 2 * t + 1]);
            }
            *reinterpret_cast<uint4*>(dst + cc + 8 * c) = ox;
            *reinterpret_cast<uint4*>(dst + kPD / 2 + cc + 8 * c) = oy;
          }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (sm.abort_flag) {
    const long long c0 = clock64();
    while (clock64() - c0 < 4000000ll) {
    }
    if (tid == 0) atomicOr(ra.err, kErrTimeout);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 128);
  }
}

// ---------------------------------------------------------------------------
// 2. causal flash attention over the reconstructed keys and values
// ---------------------------------------------------------------------------

constexpr int kAThreadsP = 192;  // warp 0 TMA, warp 1 MMA/TMEM, warps 2-5 softmax (thread = query row)
constexpr int kAtom = 128 * 128;  // one 64-column swizzle atom of 128 rows (16 KB)
constexpr float kThr = 8.f;       // lazy reference max: probabilities stay <= 2^8
constexpr float kLog2eP = 1.4426950408889634f;

struct AMapsP {
  CUtensorMap kw, vw;  // [n_rows][Hkv d] bf16: box {64, 128 rows}, 128B swizzle
};

struct AArgsP {
  const __nv_bfloat16* q;  // [B, Qmax, Hq, d] before RoPE
  const int32_t* q_len;    // [B]
  int qmax, max_len;
  const int64_t* seq_start;
  const int32_t* seq_len;
  int64_t n_rows;
  int B, Hq, Hkv, qpg;
  double om[kPD / 2];
  __nv_bfloat16* out;      // [B, Qmax, Hq, d]
  int* err;
};

struct ASmemP {
  uint8_t q[2][kAtom];      // Q^ [d atom][128 rows][128 B], K-major, 128B-swizzled
  uint8_t k[2][2][kAtom];   // K^ ring [stage][d atom][128 keys][128 B] (TMA)
  uint8_t v[2][2][kAtom];   // V^ ring [stage][d atom][128 keys][128 B] (TMA)
  uint8_t p[2][kAtom];      // P [key atom][128 rows][128 B], K-major, 128B-swizzled
  uint64_t kv_full[2], kv_empty[2], s_full[2], s_free[2], p_ready, o_ready, q_ready;
  float qbeta[kPD / 2], om32[kPD / 2];  // RoPE: (p0 w_i) mod 2 pi of the tile's first query, and w_i
  uint32_t tmem_base;
  int abort_flag;
};

// 16-byte chunk c (0..15 over 128 columns of two atoms) of row r in a K-major
// 128B-swizzled [2 atoms][128 rows][128 B] tile.
__device__ __forceinline__ uint32_t swz_chunk(int r, int c) {
  return (uint32_t)((c >> 3) * kAtom + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// grid (query tiles of 128 rows, B, Hkv)
__global__ void __launch_bounds__(kAThreadsP, 1)
    prefill_attn_kernel(const __grid_constant__ AMapsP maps, const __grid_constant__ AArgsP aa) {
  extern __shared__ uint8_t smem_raw[];
  ASmemP& sm = *reinterpret_cast<ASmemP*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  const int b = blockIdx.y, h = blockIdx.z, qpg = aa.qpg;
  const int64_t Lraw = aa.seq_len[b], st = aa.seq_start[b];
  const int Q = aa.q_len[b];
  const int PP = 128 / qpg;                             // query positions per tile
  const int i0 = (gridDim.x - 1 - blockIdx.x) * PP;    // first query index (longest tiles first)
  if (Q == 0) return;                                   // no new tokens: nothing to write
  if (Q < 0 || Q > Lraw || Q > aa.qmax || Lraw > aa.max_len || st < 0 || st + Lraw > aa.n_rows) {
    // an invalid sequence: recorded, and its output rows of this tile are zero
    if (tid == 0 && blockIdx.x == 0 && h == 0) atomicOr(aa.err, kErrBadSeq);
    for (int e = tid; e < 128 * (kPD / 8); e += blockDim.x) {
      const int r = e / (kPD / 8), qi = i0 + r / qpg;
      if (qi < aa.qmax)
        *reinterpret_cast<uint4*>(aa.out + (((int64_t)b * aa.qmax + qi) * aa.Hq + h * qpg + r % qpg) * kPD +
                                  8 * (e % (kPD / 8))) = make_uint4(0, 0, 0, 0);
    }
    return;
  }
  if (i0 >= Q) return;
  const int L = (int)Lraw;
  const int64_t row0 = aa.seq_start[b];
  const int pmax = L - Q + min(Q - 1, i0 + PP - 1);  // last position of the tile's queries
  const int nkt = pmax / kTile + 1;                   // key tiles it attends to
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.kv_full[i], 1);
      mbar_init(&sm.kv_empty[i], 1);
      mbar_init(&sm.s_full[i], 1);
      mbar_init(&sm.s_free[i], 4);
    }
    mbar_init(&sm.p_ready, 4);
    mbar_init(&sm.o_ready, 1);
    mbar_init(&sm.q_ready, 4);
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  // query RoPE angles: (p0 w_i reduced mod 2 pi in fp64, once per tile) + (row
  // offset) w_i in fp32, p0 the position of the tile's first query
  if (tid < kPD / 2) {
    const double ang = (double)(L - Q + i0) * aa.om[tid];
    sm.qbeta[tid] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
    sm.om32[tid] = (float)aa.om[tid];
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;  // S buffers at columns 0 and 128, O at 256
  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol = policy_evict_last();  // a KV tile is read by several query tiles
      for (int kt = 0; kt < nkt; ++kt) {
        const int sl = kt & 1;
        if (kt >= 2 && !mbar_wait(&sm.kv_empty[sl], ((kt - 2) >> 1) & 1, abort_flag)) break;
        mbar_expect_tx(&sm.kv_full[sl], 4 * kAtom);
        const int32_t y = (int32_t)(row0 + (int64_t)kTile * kt);
        for (int a = 0; a < 2; ++a) {
          tma_load_2d_hint(sm.k[sl][a], &maps.kw, &sm.kv_full[sl], h * kPD + 64 * a, y, pol);
          tma_load_2d_hint(sm.v[sl][a], &maps.vw, &sm.kv_full[sl], h * kPD + 64 * a, y, pol);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16(128, 128, false, false);   // S = Q K^T: both K-major
      const uint32_t id_o = idesc_bf16(128, 128, false, true);    // O += P V: V MN-major
      bool ok = mbar_wait(&sm.q_ready, 0, abort_flag);
      auto pv = [&](int j) -> bool {  // O += P_j V_j
        if (!mbar_wait(&sm.p_ready, j & 1, abort_flag)) return false;
        tc_fence_after();
        const int sl = j & 1;
        for (int k = 0; k < 8; ++k)
          umma_f16(tmem + 256, sdesc(smem_u32(sm.p[k >> 2]) + (k & 3) * 32, 16, 1024, kSw128),
                   sdesc(smem_u32(sm.v[sl][0]) + k * 2048, kAtom, 1024, kSw128), id_o, (j > 0 || k > 0) ? 1u : 0u);
        umma_commit(&sm.kv_empty[sl]);
        umma_commit(&sm.o_ready);
        return true;
      };
      for (int kt = 0; kt < nkt && ok; ++kt) {
        const int sl = kt & 1;
        if (!(ok = mbar_wait(&sm.kv_full[sl], (kt >> 1) & 1, abort_flag))) break;
        if (kt >= 2 && !(ok = mbar_wait(&sm.s_free[sl], ((kt - 2) >> 1) & 1, abort_flag))) break;
        tc_fence_after();
        for (int k = 0; k < 8; ++k)
          umma_f16(tmem + 128 * sl, sdesc(smem_u32(sm.q[k >> 2]) + (k & 3) * 32, 16, 1024, kSw128),
                   sdesc(smem_u32(sm.k[sl][k >> 2]) + (k & 3) * 32, 16, 1024, kSw128), id_s, k > 0 ? 1u : 0u);
        umma_commit(&sm.s_full[sl]);
        if (kt >= 1 && !(ok = pv(kt - 1))) break;
      }
      if (ok) pv(nkt - 1);
    }
  } else {
    // ---- softmax and output: thread = query row r ----------------------------
    const int quad = warp & 3, r = quad * 32 + lane;
    const uint32_t lb = (uint32_t)(quad * 32) << 16;
    const int qi = i0 + r / qpg, j = h * qpg + r % qpg;
    const bool valid = qi < Q;
    const int pos = L - Q + (valid ? qi : 0);
    // Q^ row: RoPE at pos, times log2(e)/sqrt(d) (scores in log2 units), bf16
    {
      const __nv_bfloat16* qr = aa.q + (((int64_t)b * aa.qmax + (valid ? qi : 0)) * aa.Hq + j) * kPD;
      const float sc = kLog2eP * rsqrtf((float)kPD);
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {  // pairs [8 cc, 8 cc + 8): chunks cc (x-halves) and 8 + cc (y-halves)
        const uint4 xr = *reinterpret_cast<const uint4*>(qr + 8 * cc);
        const uint4 yr = *reinterpret_cast<const uint4*>(qr + kPD / 2 + 8 * cc);
        const __nv_bfloat16* xh = reinterpret_cast<const __nv_bfloat16*>(&xr);
        const __nv_bfloat16* yh = reinterpret_cast<const __nv_bfloat16*>(&yr);
        uint4 ox, oy;
        __nv_bfloat162* px = reinterpret_cast<__nv_bfloat162*>(&ox);
        __nv_bfloat162* py = reinterpret_cast<__nv_bfloat162*>(&oy);
#pragma unroll
        for (int t = 0; t < 8; t += 2) {
          float rx[2], ry[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int pi = 8 * cc + t + u;
            float ph = fmaf((float)(valid ? qi - i0 : 0), sm.om32[pi], sm.qbeta[pi]);
            ph = fmaf(-kTwoPiP, rintf(ph * kInvTwoPiP), ph);
            float sn, cs;
            sincosf(ph, &sn, &cs);
            const float x = valid ? __bfloat162float(xh[t + u]) : 0.f, y = valid ? __bfloat162float(yh[t + u]) : 0.f;
            rx[u] = (x * cs - y * sn) * sc;
            ry[u] = (x * sn + y * cs) * sc;
          }
          px[t / 2] = __floats2bfloat162_rn(rx[0], rx[1]);
          py[t / 2] = __floats2bfloat162_rn(ry[0], ry[1]);
        }
        *reinterpret_cast<uint4*>(&sm.q[0][0] + swz_chunk(r, cc)) = ox;
        *reinterpret_cast<uint4*>(&sm.q[0][0] + swz_chunk(r, 8 + cc)) = oy;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.q_ready);
    }
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int kt = 0; kt < nkt && ok; ++kt) {
      const int sl = kt & 1;
      if (!(ok = wwait(&sm.s_full[sl], (kt >> 1) & 1, abort_flag))) break;
      tc_fence_after();
      const uint32_t sb = tmem + lb + 128 * sl;
      const int kbase = kTile * kt;
      const int vis = valid ? min(pos - kbase + 1, kTile) : 0;  // visible keys of this tile: [0, vis)
      // the row's 128 scores in one TMEM round trip, then the tile's max over visible keys
      float sv[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(sb + 32 * c, sv[c]);
      tmem_wait_ld();
      float mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < 4; ++c)
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (32 * c + i < vis) mt = fmaxf(mt, sv[c][i]);
      // the S buffer has been read
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.s_free[sl]);
      // a new reference max for this row when the tile's max passes the old one by kThr;
      // O and l are rescaled where a reference existed.  The TMEM loads and stores are
      // warp-collective, so the whole warp runs them when any row rescales (factor 1
      // for the other rows).
      const bool upd = mt != -INFINITY && (m == -INFINITY || mt > m + kThr);
      const bool resc = upd && m != -INFINITY;
      const float al = resc ? exp2f(m - mt) : 1.f;
      // PV of the previous tile must be done before P is overwritten and before O is rescaled
      if (kt >= 1 && !(ok = wwait(&sm.o_ready, (kt - 1) & 1, abort_flag))) break;
      tc_fence_after();
      if (__any_sync(0xffffffffu, resc)) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(tmem + lb + 256 + 32 * c, v);
          tmem_wait_ld();
          float w16[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) w16[i] = v[i] * al;
          tmem_st16(tmem + lb + 256 + 32 * c, w16);
#pragma unroll
          for (int i = 0; i < 16; ++i) w16[i] = v[16 + i] * al;
          tmem_st16(tmem + lb + 256 + 32 * c + 16, w16);
        }
        tmem_wait_st();
      }
      l *= al;
      if (upd) m = mt;
      // P = 2^(s - m) over visible keys (bf16, the row sum over the rounded values)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float* v = sv[c];
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          uint4 o;
          __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&o);
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const int k0 = 32 * c + 8 * cc + 2 * t;
            const float p0 = k0 < vis ? ex2_approx(v[8 * cc + 2 * t] - m) : 0.f;
            const float p1 = k0 + 1 < vis ? ex2_approx(v[8 * cc + 2 * t + 1] - m) : 0.f;
            po[t] = __floats2bfloat162_rn(p0, p1);
            const float2 pr = __bfloat1622float2(po[t]);
            l += pr.x + pr.y;
          }
          *reinterpret_cast<uint4*>(&sm.p[0][0] + swz_chunk(r, 4 * c + cc)) = o;
        }
      }
      // keys past the sequence in its last tile: exact zeros in V^ (P is zero there)
      if (kbase + r >= L) {
        uint4* z0 = reinterpret_cast<uint4*>(sm.v[sl][0] + r * 128);
        uint4* z1 = reinterpret_cast<uint4*>(sm.v[sl][1] + r * 128);
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          z0[c] = make_uint4(0, 0, 0, 0);
          z1[c] = make_uint4(0, 0, 0, 0);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.p_ready);
    }
    if (ok) ok = wwait(&sm.o_ready, (nkt - 1) & 1, abort_flag);
    if (ok) {
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* orow = aa.out + (((int64_t)b * aa.qmax + qi) * aa.Hq + j) * kPD;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tmem + lb + 256 + 32 * c, v);
        tmem_wait_ld();
        if (valid)
#pragma unroll
          for (int cc = 0; cc < 4; ++cc) {
            uint4 o;
            __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&o);
#pragma unroll
            for (int t = 0; t < 4; ++t) po[t] = __floats2bfloat162_rn(v[8 * cc + 2 * t] * inv, v[8 * cc + 2 * t + 1] * inv);
            *reinterpret_cast<uint4*>(orow + 32 * c + 8 * cc) = o;
          }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (sm.abort_flag) {
    const long long c0 = clock64();
    while (clock64() - c0 < 4000000ll) {
    }
    if (tid == 0) atomicOr(aa.err, kErrTimeout);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

static_assert(sizeof(RSmem) + 1024 <= 232448, "shared memory of the reconstruction kernel");
static_assert(sizeof(ASmemP) + 1024 <= 232448, "shared memory of the prefill attention kernel");

// ---------------------------------------------------------------------------
// host
// ---------------------------------------------------------------------------

bool tc_prefill_supports(const LayerTable& lt, int dtype) {
  if (dtype != DCK_BF16 || lt.d != kPD || lt.G > kMaxGroupsP || lt.Hkv > 128) return false;
  if (lt.qpg != 1 && lt.qpg != 2 && lt.qpg != 4 && lt.qpg != 8) return false;
  if (lt.rv % 16) return false;
  for (int g = 0; g < lt.G; ++g)
    if (lt.grp_rank[g] % 16) return false;
  return true;
}

size_t tc_prefill_workspace(const LayerTable& lt, int64_t n_rows) {
  return 2 * align_up((size_t)std::max<int64_t>(n_rows, 1) * lt.Hkv * kPD * 2, 256);
}

cudaError_t launch_prefill_tc(const LayerTable& lt, const void* q, const int32_t* q_len, int qmax, const void* kc,
                              const void* vc, int64_t n_rows, const void* Bk, const void* Bv,
                              const int64_t* seq_start, const int32_t* seq_len, int B, int max_len, float theta,
                              void* out, void* ws, int* err, LaunchHook* hook, cudaStream_t s) {
  const size_t half = tc_prefill_workspace(lt, n_rows) / 2;
  __nv_bfloat16* kw = static_cast<__nv_bfloat16*>(ws);
  __nv_bfloat16* vw = reinterpret_cast<__nv_bfloat16*>(static_cast<uint8_t*>(ws) + half);
  const uint64_t rows = (uint64_t)std::max<int64_t>(1, n_rows);
  RMaps rm;
  std::memset(&rm, 0, sizeof(rm));
  bool ok = true;
  const int widths[3] = {64, 32, 16};
  const CUtensorMapSwizzle sws[3] = {CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_SWIZZLE_32B};
  CUtensorMap* km[3] = {&rm.kc64, &rm.kc32, &rm.kc16};
  CUtensorMap* vm[3] = {&rm.vc64, &rm.vc32, &rm.vc16};
  for (int i = 0; i < 3 && ok; ++i) {
    ok = make_tmap_2d_bf16(km[i], kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, widths[i], kTile, sws[i]) &&
         make_tmap_2d_bf16(vm[i], vc, lt.rv, rows, (uint64_t)lt.rv * 2, widths[i], kTile, sws[i]);
  }
  ok = ok && make_tmap_2d_bf16(&rm.bv, Bv, (uint64_t)lt.Hkv * kPD, lt.rv, (uint64_t)lt.Hkv * kPD * 2, 64, 16,
                               CU_TENSOR_MAP_SWIZZLE_128B);
  for (int g = 0; g < lt.G && ok; ++g)
    ok = make_tmap_2d_bf16(&rm.bk[g], static_cast<const __nv_bfloat16*>(Bk) + lt.grp_boff[g],
                           (uint64_t)lt.grp_nh[g] * kPD, lt.grp_rank[g], (uint64_t)lt.grp_nh[g] * kPD * 2, 64, 16,
                           CU_TENSOR_MAP_SWIZZLE_128B);
  AMapsP am;
  ok = ok && make_tmap_2d_bf16(&am.kw, kw, (uint64_t)lt.Hkv * kPD, rows, (uint64_t)lt.Hkv * kPD * 2, 64, kTile,
                               CU_TENSOR_MAP_SWIZZLE_128B) &&
       make_tmap_2d_bf16(&am.vw, vw, (uint64_t)lt.Hkv * kPD, rows, (uint64_t)lt.Hkv * kPD * 2, 64, kTile,
                         CU_TENSOR_MAP_SWIZZLE_128B);
  if (!ok) return cudaErrorInvalidValue;
  RArgs ra;
  std::memset(&ra, 0, sizeof(ra));
  ra.seq_start = seq_start;
  ra.seq_len = seq_len;
  ra.n_rows = n_rows;
  ra.max_len = max_len;
  ra.B = B;
  ra.Hkv = lt.Hkv;
  ra.G = lt.G;
  ra.Rk = lt.Rk;
  ra.rv = lt.rv;
  for (int g = 0; g < lt.G; ++g) {
    ra.grp_roff[g] = lt.grp_roff[g];
    ra.grp_rank[g] = lt.grp_rank[g];
  }
  for (int hh = 0; hh < lt.Hkv; ++hh) {
    ra.head_group[hh] = lt.head_group[hh];
    ra.head_slot[hh] = lt.head_slot[hh];
  }
  for (int i = 0; i < kPD / 2; ++i) ra.om[i] = std::exp2(-2.0 * i / kPD * std::log2((double)theta));
  ra.kw = kw;
  ra.vw = vw;
  ra.err = err;
  cudaError_t e = hook_begin(hook, s);
  if (e != cudaSuccess) return e;
  const size_t rsmem = sizeof(RSmem) + 1024, asmem = sizeof(ASmemP) + 1024;
  e = cudaFuncSetAttribute(recon_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)rsmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(prefill_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)asmem);
  if (e != cudaSuccess) return e;
  // Values: V^ = C_v B_v is one dense GEMM over the cache rows (no position
  // enters it), run on the persistent CTA pairs of the long latent append,
  // where the per-head reconstruction CTAs would each stream the whole latent
  // tile for one head; taken when the rows in use can be most of the cache
  // (every row is computed).  Keys (RoPE at each row's position, the head
  // groups' factors) stay with the reconstruction kernel.
  bool v_gemm = n_rows <= 2 * (int64_t)B * max_len && n_rows < (int64_t(1) << 31) - 256;
  if (v_gemm) {
    e = launch_gemm_pair(vc, n_rows, lt.rv, Bv, lt.Hkv * kPD, vw, err, s);
    if (e == cudaErrorNotSupported) {
      cudaGetLastError();
      v_gemm = false;
    } else if (e != cudaSuccess) {
      return e;
    } else if ((e = hook_launched(hook, s)) != cudaSuccess) {
      return e;
    }
  }
  recon_kernel<<<dim3((max_len + kTile - 1) / kTile, B, (v_gemm ? 1 : 2) * lt.Hkv), kRThreads, rsmem, s>>>(rm, ra);
  if ((e = hook_launched(hook, s)) != cudaSuccess) return e;
  AArgsP aa;
  std::memset(&aa, 0, sizeof(aa));
  aa.q = static_cast<const __nv_bfloat16*>(q);
  aa.q_len = q_len;
  aa.qmax = qmax;
  aa.max_len = max_len;
  aa.seq_start = seq_start;
  aa.seq_len = seq_len;
  aa.n_rows = n_rows;
  aa.B = B;
  aa.Hq = lt.Hq;
  aa.Hkv = lt.Hkv;
  aa.qpg = lt.qpg;
  std::memcpy(aa.om, ra.om, sizeof(aa.om));
  aa.out = static_cast<__nv_bfloat16*>(out);
  aa.err = err;
  const int qtiles = (qmax * lt.qpg + 127) / 128;
  prefill_attn_kernel<<<dim3(qtiles, B, lt.Hkv), kAThreadsP, asmem, s>>>(am, aa);
  return hook_launched(hook, s);
}

}  // namespace dck
