// Tensor-core (tcgen05) decode attention over DynaCalKV latent caches, bf16.
//
// One persistent CTA per SM walks its share of 128-token tiles (see
// DecodeArgs).  For every tile and every key group g (Sec. III-C) the group's
// latent tile C_g [128 tokens x r_g] meets, on the tensor cores, one 128-column
// factor per KV head h of the group (tcgen05.mma, M = 128 tokens, N = 128,
// K = r_g, fp32 accumulator in TMEM):
//
//  * key mode (several query heads per KV head): the factor is B_g[:, slot(h)],
//    the product is the reconstructed key K^_h = C_g B_g[:, slot(h)]
//    (Sec. III-A x W ~ z R); the epilogue applies RoPE at the token's position
//    and scores every query head of h against its query rotated to L-1;
//
//  * query-folded mode (one query head per KV head): RoPE is a rotation of
//    each frequency pair, so <R_P q, R_t k> = sum_i cos(t w_i) (a_i x_i + b_i y_i)
//    + sin(t w_i) (b_i x_i - a_i y_i) with (a, b) the halves of q' = R_P q and
//    (x, y) those of k.  With k = c B_g[:, slot] both brackets are linear in the
//    latent c, so a per-sequence factor W (columns 2i and 2i+1:
//    a_i B[:, i] + b_i B[:, i+64] and b_i B[:, i] - a_i B[:, i+64]), prepared by
//    absorb_prep_kernel, gives Y = C_g W on the tensor cores with the same
//    flops, and the score is sum_i cos(t w_i) Y[2i] + sin(t w_i) Y[2i+1]: two
//    FMAs per frequency pair in the epilogue instead of RoPE plus a dot.
//
// Scores are in log2 units; the online softmax keeps a per-head reference max
// that moves only when a tile's max exceeds it by 8 (probabilities <= 256).
// Once per tile the value latents are absorbed in latent space (Sec. III-D,
// x W^(v) ~ z_v R_v applied after the sum):
//   U[:, j] += C_v[tile]^T . P[:, j]     tcgen05.mma, M = 128 rv rows,
//          N = query heads (padded to 16), K = tokens; U stays in TMEM.
// At the end of each sequence segment U, the reference max and the row sum
// are written as a split partial; the combine kernel merges splits and
// applies B_v.
//
// Warp roles (320 threads):
//   warp 0     TMA producer: latent pieces of C_g (ring A), factor slices
//              and C_v pieces (ring S), all through mbarrier rings;
//   warp 1     TMEM owner and tcgen05.mma issuer (one elected lane);
//   warps 2-9  epilogue: each TMEM lane quadrant (32 tokens) is served by two
//              warps that split the 64 RoPE frequency pairs of a head and
//              add their partial scores through shared memory.
// Every wait is bounded (2 s); on expiry the CTA stops issuing work, records
// kErrTimeout, waits for work in flight and still releases TMEM.
//
// Shared-memory layouts (all 128B-swizzled unless noted):
//   A slot  [128 tokens][w ranks] K-major, w in {64, 32, 16} with 128/64/32B
//           swizzle: UMMA operand A of the reconstruction;
//   S slot  two boxes [64 rows][64 cols]: a factor slice (rows = ranks,
//           cols = head dims; MN-major operand B) or a C_v piece (rows =
//           tokens, cols = rv; MN-major operand A of the value absorption);
//   P       [2 token atoms][Hq_pad heads][64 tokens] bf16, K-major operand B.
#include <algorithm>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "sm100.cuh"
#include "tmap.h"

#ifndef DCK_TC_TRACE
#define DCK_TC_TRACE(code) ((void)0)
#endif

namespace dck {
namespace {

using namespace sm100;

constexpr int kD = 128;
#ifndef DCK_TC_NA
#define DCK_TC_NA 5
#endif
#ifndef DCK_TC_NS
#define DCK_TC_NS 5
#endif
constexpr int kNA = DCK_TC_NA;  // latent-piece ring depth (16 KB slots)
constexpr int kNS = DCK_TC_NS;  // factor-slice / value-piece ring depth (16 KB slots)
constexpr int kSlot = 16384;
constexpr int kMaxGroupsTc = 16;
constexpr int kMaxPieces = 5;
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;
constexpr int kMaxHqTc = 32;
constexpr float kRescaleThr = 8.f;  // log2 units: probabilities stay <= 256
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kUCol = 256;     // first TMEM column of the U accumulators
constexpr float kTwoPi = 6.28318530717958647692f;
constexpr float kInvTwoPi = 0.15915494309189533577f;
constexpr float kLog2e = 1.4426950408889634f;

struct Pieces {
  int8_t n[kMaxGroupsTc];
  int8_t w[kMaxGroupsTc][kMaxPieces];
  int16_t k[kMaxGroupsTc][kMaxPieces];
};

struct Maps {
  CUtensorMap kc64, kc32, kc16, vc;
  CUtensorMap bk[kMaxGroupsTc];  // B_g (key mode, 2-D) or the per-sequence W_g (query-folded mode, 3-D)
};

struct TcArgs {
  int hq_pad;
  int n_chunks;                  // rv / 128
  Pieces pc;
  int16_t order[kMaxKvHeads];    // KV head at each (group, slot) position, group-major
};

struct Smem {
  uint8_t a[kNA][kSlot];
  uint8_t s[kNS][kSlot];
  uint8_t p[2][2 * kMaxHqTc * 128];
  float qr[kMaxHqTc * kD];        // key mode: rotated queries * log2(e)/sqrt(d)
  float x[kMaxHqTc * 128];        // scores [head][token]
  float y[4][2][kMaxQPerKv][32];  // partial-score hand-off of a quadrant's warp pair
  double om64[kD / 2];
  float om32[kD / 2];
  float beta[kD / 2];
  float redm[4][kMaxHqTc];
  float redl[4][kMaxHqTc];
  float alpha[kMaxHqTc];
  uint64_t a_full[kNA], a_empty[kNA], s_full[kNS], s_empty[kNS];
  uint64_t k_full[2], k_empty[2], p_full[2], p_empty[2], u_ready, u_free;
  uint64_t epi_bar;
  uint64_t x_full[4][2], x_empty[4][2];
  uint32_t tmem_base;
  int abort_flag;
  int b_first, pre_first, nt_total;
};

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Bounded wait whose outcome is the same in every lane of the warp.
__device__ __forceinline__ bool wwait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  const bool r = mbar_wait(bar, parity, abort_flag);
  return __all_sync(0xffffffffu, r);
}

__device__ __forceinline__ int ntiles_of(const DecodeArgs& a, int b) {
  const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
  return (L + kTile - 1) / kTile;
}

struct Segment {
  int b, L, t_begin, t_end, ntiles;
  int64_t row0;
};

// Walks the sequences overlapping tiles [x, x1) in order.
struct Walker {
  int b, pre, x, x1;
  __device__ bool next(const DecodeArgs& a, Segment& sg) {
    while (x < x1 && b < a.B) {
      const int nt = ntiles_of(a, b);
      if (x >= pre + nt) {
        pre += nt;
        ++b;
        continue;
      }
      const int xe = min(x1, pre + nt);
      sg.b = b;
      sg.L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
      sg.row0 = a.seq_start[b];
      sg.t_begin = (x - pre) * kTile;
      sg.t_end = min(sg.L, (xe - pre) * kTile);
      sg.ntiles = xe - x;
      x = xe;
      return true;
    }
    return false;
  }
};

__device__ __forceinline__ uint32_t swz_of(int w) { return w == 64 ? kSw128 : (w == 32 ? kSw64 : kSw32); }

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Byte offset of P element (head j, token t) inside one P buffer.
__device__ __forceinline__ uint32_t p_off(int j, int t, int hq_pad) {
  const int atom = t >> 6, col = t & 63;
  return atom * (hq_pad * 128) + (j >> 3) * 1024 + (j & 7) * 128 + ((((col >> 3) ^ (j & 7))) << 4) + ((col & 7) << 1);
}

// ---------------------------------------------------------------------------
// producer helper: the C_v pieces of one tile
// ---------------------------------------------------------------------------

__device__ __forceinline__ bool produce_v(Smem& sm, const Maps& maps, int n_chunks, int64_t yrow, int& s_cnt,
                                          uint64_t pol, volatile int* abort_flag) {
  for (int c = 0; c < n_chunks; ++c)
    for (int th = 0; th < 2; ++th) {
      const int sl = s_cnt % kNS;
      if (s_cnt >= kNS && !mbar_wait(&sm.s_empty[sl], ((s_cnt / kNS) - 1) & 1, abort_flag)) return false;
      mbar_expect_tx(&sm.s_full[sl], kSlot);
      tma_load_2d_hint(sm.s[sl], &maps.vc, &sm.s_full[sl], 128 * c, (int32_t)(yrow + 64 * th), pol);
      tma_load_2d_hint(sm.s[sl] + kSlot / 2, &maps.vc, &sm.s_full[sl], 128 * c + 64, (int32_t)(yrow + 64 * th), pol);
      DCK_TC_TRACE(3);
      ++s_cnt;
    }
  return true;
}

// ---------------------------------------------------------------------------
// MMA helper (whole MMA warp; lane 0 issues): value absorption of one tile,
// U[:, c-chunk] += C_v^T P
// ---------------------------------------------------------------------------

__device__ __forceinline__ bool mma_pv(Smem& sm, uint32_t tmem, const TcArgs& ta, int tt, bool first_of_seg,
                                       int nvalid, int sgc, int& s_cnt, int lane, volatile int* abort_flag) {
  const int pb = tt & 1;
  const int hq_pad = ta.hq_pad;
  if (!wwait(&sm.p_full[pb], (tt >> 1) & 1, abort_flag)) return false;
  if (first_of_seg && sgc > 0 && !wwait(&sm.u_free, (sgc - 1) & 1, abort_flag)) return false;
  tc_fence_after();
  DCK_TC_TRACE(12);
  const uint32_t idesc_v = idesc_bf16(128, hq_pad, true, false);
  const uint32_t pbase = smem_u32(sm.p[pb]);
  for (int c = 0; c < ta.n_chunks; ++c)
    for (int th = 0; th < 2; ++th) {
      const int sl = s_cnt % kNS;
      if (!wwait(&sm.s_full[sl], (s_cnt / kNS) & 1, abort_flag)) return false;
      if (nvalid < 128) {  // rows past the sequence end: make them exact zeros
        const int r0 = max(0, nvalid - 64 * th);
        for (int r = r0 + (lane >> 3); r < 64; r += 4) {
          reinterpret_cast<uint4*>(sm.s[sl] + r * 128)[lane & 7] = make_uint4(0, 0, 0, 0);
          reinterpret_cast<uint4*>(sm.s[sl] + kSlot / 2 + r * 128)[lane & 7] = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
        __syncwarp();
      }
      tc_fence_after();
      if (lane == 0) {
        const uint32_t vb = smem_u32(sm.s[sl]);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint64_t ad = sdesc(vb + k * 2048, kSlot / 2, 1024, kSw128);
          const uint64_t bd = sdesc(pbase + th * (hq_pad * 128) + k * 32, 16, 1024, kSw128);
          umma_f16(tmem + kUCol + c * hq_pad, ad, bd, idesc_v, (first_of_seg && th == 0 && k == 0) ? 0u : 1u);
        }
        umma_commit(&sm.s_empty[sl]);
      }
      __syncwarp();
      ++s_cnt;
    }
  if (lane == 0) umma_commit(&sm.p_empty[pb]);
  __syncwarp();
  DCK_TC_TRACE(13);
  return true;
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------

template <bool kFold>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ Maps maps, const LayerTable lt, const DecodeArgs a, const TcArgs ta) {
  extern __shared__ uint8_t smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  const int hq_pad = ta.hq_pad;
  const int Hq = lt.Hq, qpg = lt.qpg;

  // ---- setup -------------------------------------------------------------
  if (tid == 0) {
    for (int i = 0; i < kNA; ++i) {
      mbar_init(&sm.a_full[i], 1);
      mbar_init(&sm.a_empty[i], 1);
    }
    for (int i = 0; i < kNS; ++i) {
      mbar_init(&sm.s_full[i], 1);
      mbar_init(&sm.s_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.k_full[i], 1);
      mbar_init(&sm.k_empty[i], kEpiThreads / 32);
      mbar_init(&sm.p_full[i], kEpiThreads / 32);
      mbar_init(&sm.p_empty[i], 1);
    }
    mbar_init(&sm.u_ready, 1);
    mbar_init(&sm.u_free, kEpiThreads / 32);
    mbar_init(&sm.epi_bar, kEpiThreads / 32);
    for (int q = 0; q < 4; ++q)
      for (int i = 0; i < 2; ++i) {
        mbar_init(&sm.x_full[q][i], 1);
        mbar_init(&sm.x_empty[q][i], 1);
      }
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  {  // P buffers start at zero (padded head rows stay zero)
    uint4* pz = reinterpret_cast<uint4*>(&sm.p[0][0]);
    for (int i = tid; i < (int)(sizeof(sm.p) / 16); i += kThreads) pz[i] = make_uint4(0, 0, 0, 0);
  }
  if (tid < kD / 2) {
    const double om = exp2(-2.0 * tid / kD * log2((double)a.theta));
    sm.om64[tid] = om;
    sm.om32[tid] = (float)om;
  }
  // total tiles and the first sequence of this item (block-wide scan)
  {
    int* scan = reinterpret_cast<int*>(sm.x);
    const int per = (a.B + kThreads - 1) / kThreads;
    const int b0 = tid * per;
    int local = 0;
    for (int b = b0; b < b0 + per && b < a.B; ++b) {
      local += ntiles_of(a, b);
      if (blockIdx.x == 0) {
        const int64_t L = a.seq_len[b], st = a.seq_start[b];
        if (L < 0 || st < 0 || st + L > a.n_rows) atomicOr(a.err, kErrBadSeq);
      }
    }
    scan[tid] = local;
    __syncthreads();
    for (int off = 1; off < kThreads; off <<= 1) {
      const int v = tid >= off ? scan[tid - off] : 0;
      __syncthreads();
      scan[tid] += v;
      __syncthreads();
    }
    const int NT = scan[kThreads - 1];
    const int x0 = item_begin(blockIdx.x, NT, a.n_items);
    int run = tid ? scan[tid - 1] : 0;
    if (tid == 0) {
      sm.nt_total = NT;
      sm.b_first = a.B;
      sm.pre_first = NT;
    }
    __syncthreads();
    for (int b = b0; b < b0 + per && b < a.B; ++b) {
      const int nt = ntiles_of(a, b);
      if (nt > 0 && x0 >= run && x0 < run + nt) {
        sm.b_first = b;
        sm.pre_first = run;
      }
      run += nt;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const int NT = sm.nt_total;
  const int x0 = item_begin(blockIdx.x, NT, a.n_items);
  const int x1 = item_begin(blockIdx.x + 1, NT, a.n_items);
  Walker walk{sm.b_first, sm.pre_first, x0, x1};
  Segment seg;

  if (warp == 0) {
    // ---- TMA producer (one lane) ------------------------------------------
    if (lane == 0 && x0 < x1) {
      const uint64_t pol_stream = policy_evict_first();
      const uint64_t pol_keep = policy_evict_last();
      if (kFold) griddep_wait();  // W is written by the preparation kernel
      int a_cnt = 0, s_cnt = 0;
      bool ok = true;
      while (ok && walk.next(a, seg)) {
        for (int i = 0; i < seg.ntiles && ok; ++i) {
          const int64_t yrow = seg.row0 + seg.t_begin + (int64_t)kTile * i;
          for (int g = 0; g < lt.G && ok; ++g) {
            const int np = ta.pc.n[g];
            for (int p = 0; p < np && ok; ++p) {
              const int sl = a_cnt % kNA;
              if (a_cnt >= kNA && !(ok = mbar_wait(&sm.a_empty[sl], ((a_cnt / kNA) - 1) & 1, abort_flag))) break;
              const int w = ta.pc.w[g][p];
              const CUtensorMap* m = w == 64 ? &maps.kc64 : (w == 32 ? &maps.kc32 : &maps.kc16);
              mbar_expect_tx(&sm.a_full[sl], kTile * w * 2);
              tma_load_2d_hint(sm.a[sl], m, &sm.a_full[sl], lt.grp_roff[g] + ta.pc.k[g][p], (int32_t)yrow,
                               pol_stream);
              DCK_TC_TRACE(1);
              ++a_cnt;
            }
            const int ng = lt.grp_nh[g];
            for (int s = 0; s < ng && ok; ++s)
              for (int p = 0; p < np && ok; ++p) {
                const int sl = s_cnt % kNS;
                if (s_cnt >= kNS && !(ok = mbar_wait(&sm.s_empty[sl], ((s_cnt / kNS) - 1) & 1, abort_flag))) break;
                mbar_expect_tx(&sm.s_full[sl], kSlot);
                if (kFold) {
                  tma_load_3d_hint(sm.s[sl], &maps.bk[g], &sm.s_full[sl], s * kD, ta.pc.k[g][p], seg.b, pol_keep);
                  tma_load_3d_hint(sm.s[sl] + kSlot / 2, &maps.bk[g], &sm.s_full[sl], s * kD + 64, ta.pc.k[g][p],
                                   seg.b, pol_keep);
                } else {
                  tma_load_2d_hint(sm.s[sl], &maps.bk[g], &sm.s_full[sl], s * kD, ta.pc.k[g][p], pol_keep);
                  tma_load_2d_hint(sm.s[sl] + kSlot / 2, &maps.bk[g], &sm.s_full[sl], s * kD + 64, ta.pc.k[g][p],
                                   pol_keep);
                }
                DCK_TC_TRACE(2);
                ++s_cnt;
              }
            if (ok && g == 0 && i > 0)
              ok = produce_v(sm, maps, ta.n_chunks, yrow - kTile, s_cnt, pol_stream, abort_flag);
          }
        }
        if (ok)
          ok = produce_v(sm, maps, ta.n_chunks, seg.row0 + seg.t_begin + (int64_t)kTile * (seg.ntiles - 1), s_cnt,
                         pol_stream, abort_flag);
      }
    }
  } else if (warp == 1) {
    // ---- MMA issuer (whole warp follows, lane 0 issues) ---------------------
    if (x0 < x1) {
      const uint32_t idesc_k = idesc_bf16(128, kD, false, true);
      int a_cnt = 0, s_cnt = 0, kh = 0, tl = 0, sgc = 0;
      bool ok = true;
      while (ok && walk.next(a, seg)) {
        const int tl_first = tl;
        for (int i = 0; i < seg.ntiles && ok; ++i) {
          for (int g = 0; g < lt.G && ok; ++g) {
            const int np = ta.pc.n[g];
            const int a_base = a_cnt;
            const int ng = lt.grp_nh[g];
            for (int s = 0; s < ng && ok; ++s) {
              const int buf = kh & 1;
              if (kh >= 2 && !(ok = wwait(&sm.k_empty[buf], ((kh >> 1) - 1) & 1, abort_flag))) break;
              DCK_TC_TRACE(10);
              for (int p = 0; p < np && ok; ++p) {
                const int asl = (a_base + p) % kNA;
                if (s == 0 && !(ok = wwait(&sm.a_full[asl], ((a_base + p) / kNA) & 1, abort_flag))) break;
                const int ssl = s_cnt % kNS;
                if (!(ok = wwait(&sm.s_full[ssl], (s_cnt / kNS) & 1, abort_flag))) break;
                DCK_TC_TRACE(14);
                tc_fence_after();
                if (lane == 0) {
                  const int w = ta.pc.w[g][p];
                  const uint32_t ab = smem_u32(sm.a[asl]);
                  const uint32_t bb = smem_u32(sm.s[ssl]);
                  const uint32_t swz = swz_of(w);
                  for (int k = 0; k < w / 16; ++k) {
                    const uint64_t ad = sdesc(ab + k * 32, 16, 16 * w, swz);
                    const uint64_t bd = sdesc(bb + k * 2048, kSlot / 2, 1024, kSw128);
                    umma_f16(tmem + buf * kD, ad, bd, idesc_k, (p > 0 || k > 0) ? 1u : 0u);
                  }
                  umma_commit(&sm.s_empty[ssl]);
                }
                __syncwarp();
                ++s_cnt;
              }
              if (ok && lane == 0) umma_commit(&sm.k_full[buf]);
              __syncwarp();
              DCK_TC_TRACE(11);
              ++kh;
            }
            if (ok && lane == 0)
              for (int p = 0; p < np; ++p) umma_commit(&sm.a_empty[(a_base + p) % kNA]);
            __syncwarp();
            a_cnt += np;
            if (ok && g == 0 && i > 0)
              ok = mma_pv(sm, tmem, ta, tl - 1, tl - 1 == tl_first, 128, sgc, s_cnt, lane, abort_flag);
          }
          ++tl;
        }
        if (ok) {
          const int nvalid = seg.t_end - (seg.t_begin + kTile * (seg.ntiles - 1));
          ok = mma_pv(sm, tmem, ta, tl - 1, tl - 1 == tl_first, nvalid, sgc, s_cnt, lane, abort_flag);
        }
        if (ok && lane == 0) umma_commit(&sm.u_ready);
        __syncwarp();
        ++sgc;
      }
    }
  } else {
    // ---- epilogue: RoPE, scores, softmax, P, U readout ----------------------
    const int e = tid - 64;              // 0 .. 255
    const int quad = warp & 3;           // TMEM lane quadrant
    const int hf = (warp - 2) >> 2;      // frequency half, then head half
    const int tau = quad * 32 + lane;    // token row inside the tile
    const int hh = hq_pad / 2;           // heads owned after the hand-off
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    int kh = 0, tl = 0, sgc = 0, round = 0;
    bool ok = true;
    float m_ref[kMaxHqTc / 2];
    float l_acc[kMaxHqTc / 2];
#define EPI_SYNC()                                  \
  do {                                              \
    __syncwarp();                                   \
    if (lane == 0) mbar_arrive(&sm.epi_bar);        \
    ok = wwait(&sm.epi_bar, round & 1, abort_flag); \
    ++round;                                        \
  } while (0)
    while (ok && walk.next(a, seg)) {
      if (!kFold) {
        // rotated queries of this sequence at position L-1, scaled to log2 units
        const double P = (double)(seg.L - 1);
        const float qscale = kLog2e * rsqrtf((float)kD);
        const __nv_bfloat16* qb = static_cast<const __nv_bfloat16*>(a.q) + (int64_t)seg.b * Hq * kD;
        for (int i = e; i < Hq * (kD / 2); i += kEpiThreads) {
          const int j = i / (kD / 2), pi = i % (kD / 2);
          double sn, cs;
          sincos(P * sm.om64[pi], &sn, &cs);
          const double x1v = __bfloat162float(qb[j * kD + pi]), x2v = __bfloat162float(qb[j * kD + pi + kD / 2]);
          sm.qr[j * kD + pi] = (float)(x1v * cs - x2v * sn) * qscale;
          sm.qr[j * kD + pi + kD / 2] = (float)(x1v * sn + x2v * cs) * qscale;
        }
      }
#pragma unroll
      for (int u = 0; u < kMaxHqTc / 2; ++u) {
        m_ref[u] = -INFINITY;
        l_acc[u] = 0.f;
      }
      EPI_SYNC();
      if (!ok) break;
      const int tl_first = tl;
      for (int i = 0; i < seg.ntiles && ok; ++i) {
        const int t0 = seg.t_begin + kTile * i;
        const bool valid = t0 + tau < seg.t_end;
        // RoPE angle of token t0+tau and pair p: (t0*w_p mod 2pi, fp64) + tau*w_p (fp32)
        if (e < kD / 2) {
          const double ang = (double)t0 * sm.om64[e];
          sm.beta[e] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
        }
        EPI_SYNC();
        if (!ok) break;
        float cs[32], sn[32];
#pragma unroll
        for (int ip = 0; ip < 32; ++ip) {
          const int pi = 32 * hf + ip;
          float ph = fmaf((float)tau, sm.om32[pi], sm.beta[pi]);
          ph = fmaf(-kTwoPi, rintf(ph * kInvTwoPi), ph);
          __sincosf(ph, &sn[ip], &cs[ip]);
        }
        // per KV head, in MMA order
        for (int hi = 0; hi < lt.Hkv; ++hi) {
          const int buf = kh & 1;
          if (!(ok = wwait(&sm.k_full[buf], (kh >> 1) & 1, abort_flag))) break;
          tc_fence_after();
          DCK_TC_TRACE(20);
          const int j0 = ta.order[hi] * qpg;
          float part[kMaxQPerKv];
#pragma unroll
          for (int jj = 0; jj < kMaxQPerKv; ++jj) part[jj] = 0.f;
          if (kFold) {
            // Y columns [64 hf, 64 hf + 64): pairs (2i, 2i+1) of my 32 frequencies
#pragma unroll
            for (int ch = 0; ch < 2; ++ch) {
              float yv[32];
              tmem_ld32(tmem + lane_base + buf * kD + 64 * hf + 32 * ch, yv);
              tmem_wait_ld();
#pragma unroll
              for (int i2 = 0; i2 < 16; ++i2)
                part[0] = fmaf(cs[16 * ch + i2], yv[2 * i2], fmaf(sn[16 * ch + i2], yv[2 * i2 + 1], part[0]));
            }
          } else {
#pragma unroll
            for (int ch = 0; ch < 2; ++ch) {
              float k1[16], k2[16];
              tmem_ld16(tmem + lane_base + buf * kD + 32 * hf + 16 * ch, k1);
              tmem_ld16(tmem + lane_base + buf * kD + 64 + 32 * hf + 16 * ch, k2);
              tmem_wait_ld();
#pragma unroll
              for (int i2 = 0; i2 < 16; ++i2) {
                const int ip = 16 * ch + i2;
                const float r1 = fmaf(k1[i2], cs[ip], -k2[i2] * sn[ip]);
                const float r2 = fmaf(k1[i2], sn[ip], k2[i2] * cs[ip]);
                const float* qrow = sm.qr + j0 * kD + 32 * hf + ip;
#pragma unroll
                for (int jj = 0; jj < kMaxQPerKv; ++jj)
                  if (jj < qpg) part[jj] = fmaf(qrow[jj * kD], r1, fmaf(qrow[jj * kD + 64], r2, part[jj]));
              }
            }
          }
          DCK_TC_TRACE(25);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.k_empty[buf]);
          DCK_TC_TRACE(21);
          // the frequency-half-1 warp hands its partial scores to its partner
          const int yb = kh & 1, yn = kh >> 1;
          if (hf == 1) {
            if (yn >= 1 && !(ok = wwait(&sm.x_empty[quad][yb], (yn - 1) & 1, abort_flag))) break;
#pragma unroll
            for (int jj = 0; jj < kMaxQPerKv; ++jj)
              if (jj < qpg) sm.y[quad][yb][jj][lane] = part[jj];
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.x_full[quad][yb]);
          } else {
            if (!(ok = wwait(&sm.x_full[quad][yb], yn & 1, abort_flag))) break;
#pragma unroll
            for (int jj = 0; jj < kMaxQPerKv; ++jj)
              if (jj < qpg) sm.x[(j0 + jj) * 128 + tau] = valid ? part[jj] + sm.y[quad][yb][jj][lane] : -INFINITY;
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.x_empty[quad][yb]);
          }
          DCK_TC_TRACE(26);
          ++kh;
        }
        if (!ok) break;
        // ---- tile end: reference max, optional rescale of U, P -------------
        DCK_TC_TRACE(22);
        EPI_SYNC();
        if (!ok) break;
        float sc[kMaxHqTc / 2];
#pragma unroll
        for (int u = 0; u < kMaxHqTc / 2; ++u) {
          const int j = hf * hh + u;
          sc[u] = (u < hh && j < Hq) ? sm.x[j * 128 + tau] : -INFINITY;
          const float mx = warp_max(sc[u]);
          if (lane == 0 && u < hh && j < Hq) sm.redm[quad][j] = mx;
        }
        EPI_SYNC();
        if (!ok) break;
        float al[kMaxHqTc / 2];
#pragma unroll
        for (int u = 0; u < kMaxHqTc / 2; ++u) {
          const int j = hf * hh + u;
          al[u] = 1.f;
          if (u < hh && j < Hq) {
            const float tmax = fmaxf(fmaxf(sm.redm[0][j], sm.redm[1][j]), fmaxf(sm.redm[2][j], sm.redm[3][j]));
            if (m_ref[u] == -INFINITY || tmax > m_ref[u] + kRescaleThr) {
              al[u] = exp2f(m_ref[u] - tmax);
              m_ref[u] = tmax;
            }
            if (quad == 0 && lane == 0) sm.alpha[j] = al[u];
          }
        }
        EPI_SYNC();
        if (!ok) break;
        bool any = false;
        if (tl != tl_first)
          for (int j = 0; j < Hq; ++j) any |= sm.alpha[j] != 1.f;
        if (any) {
          // rescale U: the previous tile's absorption must have completed
          const int tp = tl - 1;
          if (!(ok = wwait(&sm.p_empty[tp & 1], (tp >> 1) & 1, abort_flag))) break;
          tc_fence_after();
          for (int c = hf; c < ta.n_chunks; c += 2)
            for (int cb = 0; cb < hq_pad / 16; ++cb) {
              float v[16];
              const uint32_t tad = tmem + lane_base + kUCol + c * hq_pad + 16 * cb;
              tmem_ld16(tad, v);
              tmem_wait_ld();
#pragma unroll
              for (int i2 = 0; i2 < 16; ++i2) {
                const int j = 16 * cb + i2;
                v[i2] *= (j < Hq) ? sm.alpha[j] : 1.f;
              }
              tmem_st16(tad, v);
            }
          tmem_wait_st();
          tc_fence_before();
        }
        // probabilities -> P (bf16); row sums use the rounded values
        const int pb = tl & 1;
        if (tl >= 2 && !(ok = wwait(&sm.p_empty[pb], ((tl - 2) >> 1) & 1, abort_flag))) break;
        uint8_t* pbuf = sm.p[pb];
#pragma unroll
        for (int u = 0; u < kMaxHqTc / 2; ++u) {
          const int j = hf * hh + u;
          if (u < hh && j < Hq) {
            l_acc[u] *= al[u];
            const __nv_bfloat16 pv = __float2bfloat16_rn(exp2f(sc[u] - m_ref[u]));
            l_acc[u] += __bfloat162float(pv);
            *reinterpret_cast<__nv_bfloat16*>(pbuf + p_off(j, tau, hq_pad)) = pv;
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sm.p_full[pb]);
        DCK_TC_TRACE(23);
        ++tl;
      }
      if (!ok) break;
      // ---- segment end: U, reference max and row sums -> partial slot c + b ---
      if (!(ok = wwait(&sm.u_ready, sgc & 1, abort_flag))) break;
      tc_fence_after();
      const int64_t slot = (int64_t)blockIdx.x + seg.b;
      for (int c = hf; c < ta.n_chunks; c += 2)
        for (int cb = 0; cb < hq_pad / 16; ++cb) {
          float v[16];
          tmem_ld16(tmem + lane_base + kUCol + c * hq_pad + 16 * cb, v);
          tmem_wait_ld();
          const int r = c * 128 + tau;
#pragma unroll
          for (int i2 = 0; i2 < 16; ++i2) {
            const int j = 16 * cb + i2;
            if (j < Hq) a.part_u[(slot * Hq + j) * lt.rv + r] = v[i2];
          }
        }
      tc_fence_before();
#pragma unroll
      for (int u = 0; u < kMaxHqTc / 2; ++u) {
        const int j = hf * hh + u;
        const float ls = warp_sum(l_acc[u]);
        if (lane == 0 && u < hh && j < Hq) sm.redl[quad][j] = ls;
      }
      EPI_SYNC();
      if (!ok) break;
      if (quad == 0 && lane == 0) {
#pragma unroll
        for (int u = 0; u < kMaxHqTc / 2; ++u) {
          const int j = hf * hh + u;
          if (u < hh && j < Hq) {
            a.part_ml[(slot * Hq + j) * 2] = m_ref[u];
            a.part_ml[(slot * Hq + j) * 2 + 1] = sm.redl[0][j] + sm.redl[1][j] + sm.redl[2][j] + sm.redl[3][j];
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.u_free);
      ++sgc;
    }
#undef EPI_SYNC
  }
  tc_fence_before();
  __syncthreads();
  if (sm.abort_flag) {
    // let copies and MMAs already in flight land before the memory is released
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 2000000ull) {
    }
    if (tid == 0) atomicOr(a.err, kErrTimeout);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Per-sequence query-folded factor of every head (one query head per KV head):
// W_b[g][k][s*128 + 2i]     = a_i B_g[k][s*128 + i] + b_i B_g[k][s*128 + 64 + i]
// W_b[g][k][s*128 + 2i + 1] = b_i B_g[k][s*128 + i] - a_i B_g[k][s*128 + 64 + i]
// with (a, b) the halves of RoPE(q_h, L_b - 1) * log2(e)/sqrt(d) (fp64 angles).
__global__ void __launch_bounds__(256) absorb_prep_kernel(const LayerTable lt, const DecodeArgs a,
                                                          __nv_bfloat16* __restrict__ W, int64_t wtot) {
  griddep_launch();
  const int h = blockIdx.x, b = blockIdx.y;
  const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
  if (L == 0) return;  // no tile of this sequence is ever processed
  __shared__ float qa[kD / 2], qb[kD / 2];
  if (threadIdx.x < kD / 2) {
    const int i = threadIdx.x;
    const double om = exp2(-2.0 * i / kD * log2((double)a.theta));
    double sn, cs;
    sincos((double)(L - 1) * om, &sn, &cs);
    const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(a.q) + ((int64_t)b * lt.Hq + h) * kD;
    const double x1 = __bfloat162float(q[i]), x2 = __bfloat162float(q[i + kD / 2]);
    const float sc = kLog2e * rsqrtf((float)kD);
    qa[i] = (float)(x1 * cs - x2 * sn) * sc;
    qb[i] = (float)(x1 * sn + x2 * cs) * sc;
  }
  __syncthreads();
  const int g = lt.head_group[h], s = lt.head_slot[h];
  const int r = lt.grp_rank[g];
  const int64_t ld = (int64_t)lt.grp_nh[g] * kD;
  const __nv_bfloat16* __restrict__ Bs = static_cast<const __nv_bfloat16*>(a.Bk) + lt.grp_boff[g] + s * kD;
  __nv_bfloat16* __restrict__ Ws = W + (int64_t)b * wtot + lt.grp_boff[g] + s * kD;
  const int total = r * (kD / 2);
  constexpr int kBatch = 8;  // independent loads in flight per thread
  for (int base = threadIdx.x; base < total; base += blockDim.x * kBatch) {
    float x[kBatch], y[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int idx = base + u * blockDim.x;
      x[u] = y[u] = 0.f;
      if (idx < total) {
        const int k = idx / (kD / 2), i = idx % (kD / 2);
        x[u] = __bfloat162float(Bs[k * ld + i]);
        y[u] = __bfloat162float(Bs[k * ld + kD / 2 + i]);
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int idx = base + u * blockDim.x;
      if (idx < total) {
        const int k = idx / (kD / 2), i = idx % (kD / 2);
        const float w0 = fmaf(qa[i], x[u], qb[i] * y[u]);
        const float w1 = fmaf(qb[i], x[u], -qa[i] * y[u]);
        *reinterpret_cast<__nv_bfloat162*>(Ws + k * ld + 2 * i) = __floats2bfloat162_rn(w0, w1);
      }
    }
  }
}

// Split of a group rank into TMA/UMMA pieces of 64, 32 and 16 columns.
int make_pieces(int r, int8_t* w, int16_t* k) {
  int n = 0, off = 0;
  for (const int pw : {64, 32, 16})
    while (r - off >= pw) {
      if (n == kMaxPieces) return kMaxPieces + 1;
      w[n] = (int8_t)pw;
      k[n] = (int16_t)off;
      off += pw;
      ++n;
    }
  return off == r ? n : kMaxPieces + 1;
}

int hq_pad_of(int Hq) { return std::max(16, (Hq + 15) / 16 * 16); }

int64_t bk_elems(const LayerTable& lt) {
  int64_t n = 0;
  for (int g = 0; g < lt.G; ++g) n += (int64_t)lt.grp_rank[g] * lt.grp_nh[g] * kD;
  return n;
}

// Tensor maps depend only on the buffers and the layer: cache the last few.
struct MapsKey {
  const void *kc, *vc, *bk;
  int64_t n_rows;
  int Rk, rv, G, B;
  int64_t sig;
  bool operator==(const MapsKey& o) const {
    return kc == o.kc && vc == o.vc && bk == o.bk && n_rows == o.n_rows && Rk == o.Rk && rv == o.rv && G == o.G &&
           B == o.B && sig == o.sig;
  }
};
constexpr int kMapsCache = 64;
std::mutex g_maps_mu;
MapsKey g_maps_key[kMapsCache];
Maps g_maps_val[kMapsCache];
int g_maps_n = 0, g_maps_next = 0;

bool build_maps(const LayerTable& lt, const DecodeArgs& a, bool fold, Maps& maps) {
  std::memset(&maps, 0, sizeof(maps));
  const uint64_t rows = (uint64_t)std::max<int64_t>(1, a.n_rows);
  bool ok = make_tmap_2d_bf16(&maps.kc64, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 64, kTile, CU_TENSOR_MAP_SWIZZLE_128B) &&
            make_tmap_2d_bf16(&maps.kc32, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 32, kTile, CU_TENSOR_MAP_SWIZZLE_64B) &&
            make_tmap_2d_bf16(&maps.kc16, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 16, kTile, CU_TENSOR_MAP_SWIZZLE_32B) &&
            make_tmap_2d_bf16(&maps.vc, a.vc, lt.rv, rows, (uint64_t)lt.rv * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B);
  const int64_t wtot = bk_elems(lt);
  for (int g = 0; g < lt.G && ok; ++g) {
    const uint64_t cols = (uint64_t)lt.grp_nh[g] * kD;
    if (fold) {
      const __nv_bfloat16* base = static_cast<const __nv_bfloat16*>(a.extra) + lt.grp_boff[g];
      ok = make_tmap_3d_bf16(&maps.bk[g], base, cols, lt.grp_rank[g], a.B, cols * 2, (uint64_t)wtot * 2, 64, 64,
                             CU_TENSOR_MAP_SWIZZLE_128B);
    } else {
      const __nv_bfloat16* base = static_cast<const __nv_bfloat16*>(a.Bk) + lt.grp_boff[g];
      ok = make_tmap_2d_bf16(&maps.bk[g], base, cols, lt.grp_rank[g], cols * 2, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B);
    }
  }
  return ok;
}

}  // namespace

bool tc_decode_supports(const LayerTable& lt, int dtype) {
  if (dtype != DCK_BF16 || lt.d != kD) return false;
  if (lt.Hq > kMaxHqTc || lt.qpg > kMaxQPerKv || lt.G > kMaxGroupsTc) return false;
  if (lt.rv % 128 || (lt.rv / 128) * hq_pad_of(lt.Hq) > 256) return false;
  for (int g = 0; g < lt.G; ++g) {
    int8_t w[kMaxPieces];
    int16_t k[kMaxPieces];
    if (lt.grp_rank[g] > 256 || make_pieces(lt.grp_rank[g], w, k) > kMaxPieces) return false;
  }
  return true;
}

// Extra workspace of the tensor-core path: the per-sequence folded factors.
size_t tc_decode_extra_ws(const LayerTable& lt, int batch) {
  if (lt.qpg != 1 || !tc_decode_supports(lt, DCK_BF16)) return 0;
  return align_up((size_t)batch * bk_elems(lt) * 2, 256);
}

int tc_decode_launches(const LayerTable& lt) { return lt.qpg == 1 ? 2 : 1; }

cudaError_t launch_decode_tc(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  const bool fold = lt.qpg == 1;
  if (fold && !a.extra) return cudaErrorInvalidValue;
  TcArgs ta;
  std::memset(&ta, 0, sizeof(ta));
  ta.hq_pad = hq_pad_of(lt.Hq);
  ta.n_chunks = lt.rv / 128;
  int pos = 0;
  for (int g = 0; g < lt.G; ++g) {
    ta.pc.n[g] = (int8_t)make_pieces(lt.grp_rank[g], ta.pc.w[g], ta.pc.k[g]);
    for (int sl = 0; sl < lt.grp_nh[g]; ++sl)
      for (int h = 0; h < lt.Hkv; ++h)
        if (lt.head_group[h] == g && lt.head_slot[h] == sl) ta.order[pos++] = (int16_t)h;
  }
  int64_t sig = fold ? 1 : 0;
  for (int g = 0; g < lt.G; ++g) sig = sig * 1000003 + lt.grp_rank[g] * 131 + lt.grp_nh[g] * 7 + lt.grp_boff[g];
  const MapsKey key{a.kc, a.vc, fold ? a.extra : a.Bk, a.n_rows, lt.Rk, lt.rv, lt.G, fold ? a.B : 0, sig};
  Maps maps;
  bool have = false;
  {
    std::lock_guard<std::mutex> lk(g_maps_mu);
    for (int i = 0; i < g_maps_n && !have; ++i)
      if (g_maps_key[i] == key) {
        maps = g_maps_val[i];
        have = true;
      }
  }
  if (!have) {
    if (!build_maps(lt, a, fold, maps)) return cudaErrorInvalidValue;
    std::lock_guard<std::mutex> lk(g_maps_mu);
    g_maps_key[g_maps_next] = key;
    g_maps_val[g_maps_next] = maps;
    g_maps_next = (g_maps_next + 1) % kMapsCache;
    g_maps_n = std::min(g_maps_n + 1, kMapsCache);
  }
  const size_t smem = sizeof(Smem) + 1024;
  static int attr_done[64][2] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  const bool dev_ok = dev >= 0 && dev < 64;
  if (!dev_ok || !attr_done[dev][fold]) {
    cudaError_t e = fold ? cudaFuncSetAttribute(decode_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem)
                         : cudaFuncSetAttribute(decode_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem);
    if (e != cudaSuccess) return e;
    if (dev_ok) attr_done[dev][fold] = 1;
  }
  if (a.ev0 && record_timing_event(a.ev0, s) != cudaSuccess)
    return cudaErrorUnknown;
  cudaError_t e;
  if (fold) {
    absorb_prep_kernel<<<dim3(lt.Hq, a.B), 256, 0, s>>>(lt, a, static_cast<__nv_bfloat16*>(a.extra), bk_elems(lt));
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.n_items);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_tc_kernel<true>, maps, lt, a, ta);
  } else {
    decode_tc_kernel<false><<<a.n_items, kThreads, smem, s>>>(maps, lt, a, ta);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess && a.ev1)
    e = record_timing_event(a.ev1, s);
  return e;
}

}  // namespace dck
