// Tensor-core (tcgen05) decode attention over DynaCalKV latent caches, bf16:
// the scores kernel (key reconstruction, RoPE, scores, online softmax).
//
// The kernel runs as persistent CTA pairs: a cluster of two CTAs on the two
// SMs of a TPC issues one tcgen05 pair MMA (cta_group::2) over a pair tile of
// 256 tokens, the even CTA holding the first 128 tokens' latents and the odd
// CTA the rest (the work plan is in tc_common.cuh).  For every pair tile and
// every key group g (Sec. III-C) the group's latent tile C_g [256 tokens x r_g]
// meets the factor columns of the group's KV heads, two heads per MMA where the
// group has them (M = 256 tokens, N = 256 or 128, K = r_g; each CTA holds the
// factor columns of one head, or one half of a lone head, and receives the
// fp32 accumulator rows of its own 128 tokens in its TMEM).  A pair MMA moves
// each SM's share of the factor operand once per 256 tokens instead of once
// per 128, and halves the MMA instructions per token.  Two 256-column
// accumulators (all of TMEM) let the epilogue read one unit while the tensor
// cores compute the next.  Per head:
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
//    a_i B[:, i] + b_i B[:, i+64] and b_i B[:, i] - a_i B[:, i+64]) gives
//    Y = C_g W on the tensor cores with the same flops, and the score is
//    sum_i cos(t w_i) Y[2i] + sin(t w_i) Y[2i+1]: two FMAs per frequency pair.
//
// Factor items (one latent piece's ranks x 128 columns of each head of a
// unit) are prepared once per call by factor_prep_kernel as the exact
// 128B-swizzled shared-memory image of the UMMA B operand (heads * ranks * 256
// bytes each, in consumption order); each CTA of a pair loads its half of an
// item (its head, or its half of a lone head) with one TMA copy.
//
// Scores are in log2 units; the online softmax keeps a per-head reference max
// that moves only when a tile's max exceeds it by 8 (probabilities <= 256).
// Each CTA runs the softmax of its own 128-token halves: their probabilities P
// (bf16, laid out as the B operand of the value absorption) and the reference
// maxima they were computed with go to the workspace per 128-token tile; at
// the end of each segment the reference max and the row sum (over the rounded
// P) are written as the segment's split partial.  The absorption kernel
// (absorb_tc.cu) forms U = C_v^T P from them.
//
// Warp roles (384 threads query-folded, 352 key mode), in both CTAs unless
// noted.  Every TMA instruction costs its issuing thread a long round trip, so
// loads are issued by two producer warps, each putting several copies (one per
// lane) into one instruction; the copies of both CTAs complete on the even
// CTA's barriers, which its MMA threads wait on:
//   warp 0     latent pieces of C_g (ring A)
//   warp 10    factor items (ring W; query-folded mode: one ring per MMA thread)
//   warp 1     TMEM owner; in the even CTA its lane 0 issues pair MMAs.  On this
//              GPU every barrier test, commit or fence costs the issuing thread a
//              dependent round trip of 100-500 cycles, so in query-folded mode
//              lane 0 of the even CTA's warp 11 issues every other unit into the
//              other accumulator and the two threads' bookkeeping overlaps the
//              other's MMAs; the MMA commits arrive on both CTAs' barriers
//   warps 2-9  epilogue: each TMEM lane quadrant (32 tokens) is served by two
//              warps that split the 64 RoPE frequency pairs of a head; their
//              partial scores go to one shared-memory array per frequency
//              half, summed at the tile end.  Both CTAs' epilogues release an
//              accumulator on the even CTA's barrier.
// Every wait is bounded (about 2 s); on expiry the CTA stops issuing work,
// tells its peer to stop, records kErrTimeout, waits for work in flight and
// still releases TMEM.
//
// Shared-memory operand layouts (128B swizzle unless noted), identical in both
// CTAs (a pair MMA reads the same offsets in each):
//   A slot  [128 tokens][w ranks] K-major, w in {64, 32, 16} with 128/64/32B
//           swizzle: this CTA's rows of the UMMA operand A;
//   W slot  [2 halves][w ranks][64 columns] MN-major (one head), or
//           [w ranks][64 columns] (half of a lone head): this CTA's columns of
//           operand B (the 64-column atoms w * 128 bytes apart);
// P ([2 token atoms][Hq_pad heads][64 tokens] bf16, K-major: the absorption's
// operand B) is written straight to the workspace by the tile-end owners.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "tc_common.cuh"
#include "tc_host.h"
#include "tmap.h"

namespace dck {
namespace {

using namespace sm100;
using namespace tc;

constexpr int kD = 128;
constexpr int kSlot = 16384;     // latent slots: 128 tokens x 64 ranks
constexpr int kSlotW = 16384;    // factor slots: one head (2 x 64 ranks x 64 columns) of an item
constexpr int kMaxGroupsTc = 16;
constexpr int kMaxPieces = 5;
constexpr int kMaxHqTc = 32;
constexpr int kMaxItems = 256;
constexpr int kMaxUnits = 32;
constexpr int kEpiThreads = 256;
constexpr int kEpiWarps = kEpiThreads / 32;
// Latent tiles prefetched toward L2 ahead of their loads: two in query-folded
// mode; none in key mode, whose TMA loads keep enough of the latent stream in
// flight themselves and whose prefetches only competed with it (7B GQA layer,
// 0 / 1 / 2 / 4 tiles ahead: 298 / 301 / 306 / 315 us per step)
template <bool kFold>
__host__ __device__ constexpr int prefetch_ahead() { return kFold ? 2 : 0; }
constexpr float kRescaleThr = 8.f;  // log2 units: probabilities stay <= 256
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kKCols = 256;    // TMEM columns of one key accumulator
constexpr float kTwoPi = 6.28318530717958647692f;
constexpr float kInvTwoPi = 0.15915494309189533577f;
constexpr float kLog2e = 1.4426950408889634f;

template <bool kFold>
struct Ring {
  // latent-piece slots (16 KB each) and factor-item slots (half items, 16 KB
  // each).  The latent ring holds the group in use while the next group's
  // pieces arrive from HBM; key mode's B_g items are few and L2-resident, so
  // five of its slots go to the latents (measured on the 7B GQA layer: 4/6
  // latent/factor slots 233 us, 5/5 200 us, 6/4 204 us, 8/2 225 us)
  static constexpr int NA = 5;
  static constexpr int NW = kFold ? 6 : 5;
  // MMA-issuing threads: two in query-folded mode; key mode's units carry up
  // to four items, which one thread streams better
  static constexpr int kMma = kFold ? 2 : 1;
  static constexpr int kThreads = kFold ? 384 : 352;
};

// Latent-piece maps (box 64/32/16 ranks x 128 tokens, 128/64/32B swizzle) and
// factor-image maps (rows of 128 bytes, box 16/32/64/128 rows, no swizzle: the
// images are stored pre-swizzled).
struct Maps {
  CUtensorMap kc64, kc32, kc16;
  CUtensorMap im[4];
};

// Per-group facts the hot loops need; copied to shared memory at kernel start
// (indexing kernel-parameter tables at run time goes through the small constant
// cache, which several warps would share).
struct GroupSm {
  int32_t roff;          // first key-cache column of the group
  int8_t np;             // latent pieces
  int8_t h0, nh;         // MMA position of the group's first head, heads
  int8_t nu;             // units (pairs of heads, the last one single when nh is odd)
  int8_t w[kMaxPieces];  // piece widths (ranks)
  int8_t pad;
  int16_t u0;            // the group's first unit in the tile's unit order
  int16_t k[kMaxPieces]; // first rank of each piece
  int16_t i0;            // the group's first factor item in the tile's item order
  int16_t rank;          // r_g
};

struct TcArgs {
  int hq_pad;
  int n_items;                   // factor items per tile
  int n_pairs;                   // P
  int64_t fimg_seq_bytes;        // factor image bytes per sequence (query-folded mode)
  uint8_t* pglob;                // per-tile P images (workspace)
  float* mglob;                  // per-tile reference maxima (workspace)
  int64_t max_tiles;
  double om[kD / 2];             // RoPE frequencies theta^(-2i/d), fp64
  GroupSm grp[kMaxGroupsTc];
  int16_t order[kMaxHqTc];       // KV head at each MMA position (group-major, slot order)
  int n_units;                   // units per tile
  int16_t uitem[kMaxUnits + 1];  // first factor item of each unit (and the item count)
  int8_t hunit[kMaxHqTc];        // unit of each query head
  uint32_t item[kMaxItems];      // factor item n: byte offset | (bytes / 4096) << 26
};

template <bool kFold>
struct Smem {
  uint8_t a[Ring<kFold>::NA][kSlot];
  uint8_t w[Ring<kFold>::NW][kSlotW];
  // scores [frequency half][query head][token]: each half's partial scores by
  // plain stores, summed at the tile end
  float x[2 * kMaxHqTc * 128];
  // key mode: rotated queries * log2(e)/sqrt(d), bf16 [query head][d] (the
  // B operand of the warps' score MMAs), and per epilogue warp a staging tile
  // of its 32 tokens' rotated keys [token][32] bf16 (the A operand), 16-byte
  // chunks swizzled by (token / 2) % 4
  __nv_bfloat16 qr[kFold ? 2 : kMaxHqTc * kD];
  uint8_t kst[kFold ? 1 : kEpiWarps][kFold ? 16 : 32 * 64];
  double om64[kD / 2];
  float om32[kD / 2];
  float beta[kD / 2];
  float qcs[kFold ? 1 : kD / 2], qsn[kFold ? 1 : kD / 2];  // key mode: RoPE of the query position
  // latent ring: one full/empty pair per group instance; factor rings: one
  // pair per unit (batch of items) of each MMA thread (see SlotFifo)
  uint64_t g_full[kFifoBars], g_empty[kFifoBars];
  uint64_t u_full[kFifoBars], u_empty[kFifoBars];
  uint64_t k_full[2], k_empty[2], epi_bar;
  GroupSm grp[kMaxGroupsTc];
  int16_t order[kMaxHqTc];
  int16_t uitem[kMaxUnits + 1];
  int8_t hunit[kMaxHqTc];
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ uint32_t swz_of(int w) { return w == 64 ? kSw128 : (w == 32 ? kSw64 : kSw32); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return (uint32_t)__bfloat16_as_ushort(h.x) | ((uint32_t)__bfloat16_as_ushort(h.y) << 16);
}
// Four 8x8 b16 matrices from shared memory; lane i gives the row address of row
// i % 8 of matrix i / 8.
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
// d += a b for one 16 x 8 x 16 tile, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Rows (of 128 bytes) of a half item of `bytes` bytes -> factor-image map index.
__device__ __forceinline__ int im_map_of(uint32_t half_rows) {
  return half_rows == 16 ? 0 : (half_rows == 32 ? 1 : (half_rows == 64 ? 2 : 3));
}

// ---------------------------------------------------------------------------
// the scores kernel
// ---------------------------------------------------------------------------

template <bool kFold>
__global__ void __launch_bounds__(Ring<kFold>::kThreads, 1)
    decode_tc_kernel(const __grid_constant__ Maps maps, const LayerTable lt, const DecodeArgs a,
                     const __grid_constant__ TcArgs ta) {
  constexpr int kMma = Ring<kFold>::kMma, NW = Ring<kFold>::NW, kNA = Ring<kFold>::NA;
  constexpr int kThreads = Ring<kFold>::kThreads;
  extern __shared__ uint8_t smem_raw[];
  Smem<kFold>& sm =
      *reinterpret_cast<Smem<kFold>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  const int hq_pad = ta.hq_pad;
  const int Hq = lt.Hq, qpg = lt.qpg;
  const int hr = (int)cluster_ctarank();  // the half of every pair tile this CTA holds
  const bool leader = hr == 0;            // the even CTA issues the pair MMAs
  const int P = ta.n_pairs, pair = blockIdx.x >> 1;

  // ---- setup -------------------------------------------------------------
  if (tid == 0) {
    for (int i = 0; i < kFifoBars; ++i) {
      mbar_init(&sm.g_full[i], 1);      // even CTA: its producer's expect_tx; both CTAs' copies complete on it
      mbar_init(&sm.g_empty[i], kMma);  // released by every MMA thread (arrivals reach both CTAs)
      mbar_init(&sm.u_full[i], 1);
      mbar_init(&sm.u_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.k_full[i], 1);
      mbar_init(&sm.k_empty[i], 2 * kEpiWarps);  // even CTA: both CTAs' epilogue warps
    }
    mbar_init(&sm.epi_bar, kEpiWarps);
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(&sm.tmem_base, kTmemCols);
    tmem_relinquish_pair();
  }
  if (tid < lt.G) sm.grp[tid] = ta.grp[tid];
  if (tid < lt.Hkv) sm.order[tid] = ta.order[tid];
  if (tid <= ta.n_units) sm.uitem[tid] = ta.uitem[tid];
  if (tid < Hq) sm.hunit[tid] = ta.hunit[tid];
  if (tid < kD / 2) {
    sm.om64[tid] = ta.om[tid];
    sm.om32[tid] = (float)ta.om[tid];
  }
  // Work of this pair: main pair tiles [X0, X1) (every unit), then units
  // [u_lo, u_hi) of the flattened (extra tile, unit) list, every extra tile a
  // segment of its own.
  const int U = ta.n_units;
  // block-scan scratch in the latent ring: used only before the first copy is issued
  int* const s256 = reinterpret_cast<int*>(sm.a[0]);
  int* const s128 = s256 + kThreads;
  const int NP = pair_tile_count(a, s256, s128);
  const int NT128 = s128[kThreads - 1];
  const PSplit sp(NP, P);
  // the per-tile stores are sized for non-overlapping sequences; more tiles
  // than that is reported as invalid input and nothing is computed
  const bool fits = NT128 <= ta.max_tiles;
  if (!fits && tid == 0 && blockIdx.x == 0) atomicOr(a.err, kErrBadSeq);
  const int X0 = fits ? sp.main_begin(pair, P) : 0;
  const int X1 = fits ? sp.main_begin(pair + 1, P) : 0;
  const int xu = sp.R * U;
  const int u_lo = fits ? (int)((int64_t)pair * xu / P) : 0;
  const int u_hi = fits ? (int)((int64_t)(pair + 1) * xu / P) : 0;
  const int xe0 = sp.NPm + (u_lo < u_hi ? u_lo / U : 0), xe1 = sp.NPm + (u_lo < u_hi ? (u_hi - 1) / U + 1 : 0);
  const PairWalker walk_m = pair_walker_at(a, s256, s128, X0, X1, false);
  const PairWalker walk_x = pair_walker_at(a, s256, s128, xe0, xe1, true);
  const bool has_work = X0 < X1 || xe0 < xe1;  // the same in both CTAs of the pair
  // units [ua, ub) of flattened pair tile X in phase ph (0: main, 1: extra)
  auto units_of = [&](int ph, int X, int& ua, int& ub) {
    ua = 0;
    ub = U;
    if (ph) {
      const int e = X - sp.NPm;
      ua = max(u_lo - e * U, 0);
      ub = min(u_hi - e * U, U);
    }
  };
  for (int i = tid; i < (int)(sizeof(sm.x) / sizeof(float)); i += kThreads) sm.x[i] = 0.f;
  tc_fence_before();
  cluster_sync();  // both CTAs' barriers initialised and TMEM allocated
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  // shared::cluster addresses: a barrier of the even CTA, or a word of the peer
  auto lead = [](const void* p) { return mapa_shared(smem_u32(p), 0); };
  auto peer = [hr](const void* p) { return mapa_shared(smem_u32(p), (uint32_t)(hr ^ 1)); };
  // a wait that gave up stops the peer too
  auto stop_peer = [&]() { st_cluster_u32(peer(&sm.abort_flag), 1u); };
  PSegment seg;

  // Half items (this CTA's head, or its half of a lone head) of one unit into
  // the factor ring, in batches of at most NW items: each batch is one
  // instance of the ring (one full barrier, which the even CTA's lane 0 arms
  // with the bytes of both CTAs' copies; one TMA copy per lane).  The units of
  // both MMA threads share the ring, in unit order.
  auto put_unit = [&](SlotFifo& f, int n, int np, int64_t img_row0, uint64_t pol) -> bool {
    for (int p0 = 0; p0 < np;) {
      const int nb = min(NW, np - p0);
      if (!f.claim(nb, NW, sm.u_empty, lane, abort_flag)) return false;
      uint64_t* full = &sm.u_full[f.inst % kFifoBars];
      if (leader && lane == 0) {
        uint32_t total = 0;
        for (int q = 0; q < nb; ++q) total += (ta.item[n + p0 + q] >> 26) << 12;
        mbar_expect_tx(full, total);
      }
      __syncwarp();
      if (lane < nb) {
        const int sl = (f.head + lane) % NW;
        const uint32_t it = ta.item[n + p0 + lane];
        const uint32_t hrows = ((it >> 26) << 12) / 256;
        const int64_t y = img_row0 + ((it & 0x03FFFFFFu) >> 7) + hr * hrows;
        tma_load_2d_pair(sm.w[sl], &maps.im[im_map_of(hrows)], lead(full), 0, (int32_t)y, pol);
      }
      __syncwarp();
      f.advance(nb);
      p0 += nb;
    }
    return true;
  };
  const int64_t img_seq_rows = ta.fimg_seq_bytes >> 7;
  // Programmatic dependent launch: every thread lets the absorption kernel
  // launch only after it has seen the preparation kernel complete, so that
  // the absorption's value loads ahead of its own grid-dependency wait find
  // the rows a decode step appends.  The latent producer first moves its
  // first tiles toward L2.
  if (warp != 0) {
    griddep_wait();
    griddep_launch();
  }

  if (warp == 0) {
    // ---- latent pieces (this CTA's 128 rows of each), issued as soon as their
    // slots are free; in query-folded mode also the factor items of MMA thread
    // 1, in the order that thread consumes them (a group's pieces, then its
    // units' items) ---------------------------------------------------------
    if (has_work) {
      const uint64_t pol = policy_evict_first();
      SlotFifo ga;  // the latent ring
      bool ok = true;
      // L2 prefetch of this half's latent rows, prefetch_ahead() tiles ahead of the
      // loads (across segment boundaries): the TMA loads then find them in L2
      PairWalker pwalk[2] = {walk_m, walk_x};
      PSegment pseg;
      int pph = 0, pti = 0;
      bool pvalid = false;
      auto prefetch_next = [&]() {
        if (lane != 0) return;
        while (!pvalid || pti >= pseg.ntiles) {
          while (pph < 2 && !pwalk[pph].next(a, pseg)) ++pph;
          if (pph >= 2) return;
          pvalid = true;
          pti = 0;
        }
        const int64_t r0 = pseg.row0 + pseg.t0(pti++, hr);
        const int64_t nr = a.n_rows - r0 < kTile ? a.n_rows - r0 : (int64_t)kTile;
        if (nr > 0) prefetch_l2(static_cast<const __nv_bfloat16*>(a.kc) + r0 * lt.Rk, (uint32_t)(nr * lt.Rk * 2));
      };
      for (int q = 0; q < prefetch_ahead<kFold>(); ++q) prefetch_next();
      griddep_wait();  // the preparation launch may append the step's own latents
      griddep_launch();
      for (int ph = 0; ph < 2 && ok; ++ph)
        for (PairWalker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
          const int64_t img_row0 = kFold ? (int64_t)seg.b * img_seq_rows : 0;
          for (int i = 0; i < seg.ntiles && ok; ++i) {
            const int64_t yrow = seg.row0 + seg.t0(i, hr);
            prefetch_next();
            int ua, ub;
            units_of(ph, seg.X0 + i, ua, ub);
            for (int g = 0; g < lt.G && ok; ++g) {
              const GroupSm& gs = sm.grp[g];
              const int np = gs.np;
              const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);
              if (lo >= hi) continue;  // none of the group's units in this piece of work
              // the group's pieces: one instance of the latent ring
              if (!(ok = ga.claim(np, kNA, sm.g_empty, lane, abort_flag))) break;
              uint64_t* gfull = &sm.g_full[ga.inst % kFifoBars];
              if (leader && lane == 0) mbar_expect_tx(gfull, 2 * kTile * 2 * gs.rank);
              __syncwarp();
              if (lane < np) {
                const int sl = (ga.head + lane) % kNA;
                const int w = gs.w[lane];
                const CUtensorMap* m = w == 64 ? &maps.kc64 : (w == 32 ? &maps.kc32 : &maps.kc16);
                tma_load_2d_pair(sm.a[sl], m, lead(gfull), gs.roff + gs.k[lane], (int32_t)yrow, pol);
              }
              __syncwarp();
              ga.advance(np);
            }
          }
        }
      if (!ok && lane == 0) stop_peer();
    } else {
      griddep_wait();
      griddep_launch();
    }
  } else if (warp == 10) {
    // ---- factor items: several TMA copies per instruction (query-folded
    // mode: the ring of MMA thread 0 only) --------------------------------------
    if (has_work) {
      const uint64_t pol = policy_evict_last();
      SlotFifo fw;         // the factor ring
      bool ok = true;
      for (int ph = 0; ph < 2 && ok; ++ph)
        for (PairWalker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
          const int64_t img_row0 = kFold ? (int64_t)seg.b * img_seq_rows : 0;
          for (int i = 0; i < seg.ntiles && ok; ++i) {
            int ua, ub;
            units_of(ph, seg.X0 + i, ua, ub);
            for (int g = 0; g < lt.G && ok; ++g) {
              const GroupSm& gs = sm.grp[g];
              const int np = gs.np;
              const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);
              for (int u = lo; u < hi && ok; ++u) ok = put_unit(fw, gs.i0 + u * np, np, img_row0, pol);
            }
          }
        }
      if (!ok && lane == 0) stop_peer();
    }
  } else if (warp == 1 || (kMma == 2 && warp == 11)) {
    // ---- MMA issuers (even CTA only): lane 0 of warp 1 (and of warp 11 in
    // query-folded mode) runs the schedule of every kMma-th unit into its own
    // accumulator, so one thread's barrier waits and commits overlap the
    // other's MMAs.  Each thread owns a factor ring (single consumer).  Per
    // unit: one wait for its items, one for its accumulator, its MMAs, one
    // commit for the items and one for the accumulator; per key group one
    // wait for all its latent pieces and one release (commit, or arrivals in
    // both CTAs when the thread has no unit in the group, after the fill so
    // that no barrier phase is passed early). ---------------------------------
    if (leader && lane == 0 && has_work) {
      const int t = warp == 1 ? 0 : 1;
      int gi = 0, ghead = 0;  // latent-ring instances (groups) and slots handed out so far
      int ui = 0, uhead = 0;  // factor-ring instances (item batches of every unit) and slots
      int kc = 0, own = 0;    // units of the pair so far, units in this thread's accumulator
      bool ok = true;
      for (int ph = 0; ph < 2 && ok; ++ph)
        for (PairWalker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
          for (int i = 0; i < seg.ntiles && ok; ++i) {
            int ua, ub;
            units_of(ph, seg.X0 + i, ua, ub);
            for (int g = 0; g < lt.G && ok; ++g) {
              const GroupSm& gs = sm.grp[g];
              const int np = gs.np;
              const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);  // the group's units here
              if (lo >= hi) continue;
              const int gb = gi % kFifoBars;
              const uint32_t gpar = (gi / kFifoBars) & 1;
              const int uf = lo + (kMma == 2 ? (((kc & 1) == t) ? 0 : 1) : 0);  // this thread's first unit of the group
              // all the group's latent pieces (both CTAs' rows) are there
              if (!(ok = mbar_wait(&sm.g_full[gb], gpar, abort_flag))) break;
              if (uf >= hi) {  // no unit of this thread in the group: release its pieces in both CTAs
                mbar_arrive(&sm.g_empty[gb]);
                mbar_arrive_cluster(peer(&sm.g_empty[gb]));
              }
              for (int u = lo; u < hi && ok; ++u) {
                if (u < uf || (u - uf) % kMma != 0) {  // the other thread's unit: skip its item batches
                  ui += (np + NW - 1) / NW;
                  uhead += np;
                  continue;
                }
                const int nh = min(2, gs.nh - 2 * u);
                const uint32_t idesc_k = idesc_bf16(256, kD * nh, false, true);
                const int kg = kc + (u - lo);                        // unit index of the pair
                const int buf = kMma == 2 ? t : (kg & 1);
                const int use = kMma == 2 ? own : (kg >> 1);         // earlier units in this accumulator
                const uint32_t dcol = tmem + buf * kKCols;
                for (int p0 = 0; p0 < np && ok;) {  // the unit's item batches (ring instances)
                  const int nb = min(NW, np - p0);
                  const int ub_ = ui % kFifoBars;
                  if (!(ok = mbar_wait(&sm.u_full[ub_], (ui / kFifoBars) & 1, abort_flag))) break;
                  if (p0 == 0 && use >= 1) {  // both CTAs' epilogues have read this accumulator's previous unit
                    if (!(ok = mbar_wait(&sm.k_empty[buf], (use - 1) & 1, abort_flag))) break;
                  }
                  tc_fence_after();
                  for (int q = 0; q < nb; ++q) {
                    const int p = p0 + q;
                    const int w = gs.w[p];
                    const uint32_t ab0 = smem_u32(sm.a[(ghead + p) % kNA]);
                    const uint32_t bb = smem_u32(sm.w[(uhead + q) % NW]);
                    const uint32_t swz = swz_of(w);
                    for (int k = 0; k < w / 16; ++k) {
                      const uint64_t ad = sdesc(ab0 + k * 32, 16, 16 * w, swz);
                      const uint64_t bd = sdesc(bb + k * 2048, 128 * w, 1024, kSw128);
                      umma_f16_pair(dcol, ad, bd, idesc_k, (p > 0 || k > 0) ? 1u : 0u);
                    }
                  }
                  umma_commit_pair(&sm.u_empty[ub_]);  // the batch's slots, once its MMAs are done
                  ++ui;
                  uhead += nb;
                  p0 += nb;
                }
                if (!ok) break;
                umma_commit_pair(&sm.k_full[buf]);
                if (u + kMma >= hi) umma_commit_pair(&sm.g_empty[gb]);  // this thread is done with the pieces
                ++own;
              }
              ++gi;
              ghead += np;
              kc += hi - lo;
            }
          }
        }
      if (!ok) stop_peer();
    }
    __syncwarp();
  } else if (warp >= 2 && warp <= 9) {
    // ---- epilogue: RoPE, scores, softmax, P of this CTA's 128-token halves ----
    const int e = tid - 64;              // 0 .. 255
    const int quad = warp & 3;           // TMEM lane quadrant
    const int hf = (warp - 2) >> 2;      // frequency half, then head half
    const int tau = quad * 32 + lane;    // token row inside the half tile
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    // tile and segment ends: thread e owns head jt and the 16 tokens [16 ct, 16 ct + 16)
    // of every half tile; the 8 owners of a head are adjacent lanes of one warp
    const int jt = e >> 3, ct = e & 7;
    int kc = 0, round = 0;
    bool ok = true;
#define EPI_SYNC()                                  \
  do {                                              \
    __syncwarp();                                   \
    if (lane == 0) mbar_arrive(&sm.epi_bar);        \
    ok = wwait(&sm.epi_bar, round & 1, abort_flag); \
    ++round;                                        \
  } while (0)
    // an accumulator has been read by this warp: release it on the even CTA's barrier
    auto release_acc = [&](int buf) {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(&sm.k_empty[buf]);
        else mbar_arrive_cluster(lead(&sm.k_empty[buf]));
      }
    };
    for (int ph = 0; ph < 2 && ok; ++ph)
      for (PairWalker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
        if (!kFold) {
          // rotated queries of this sequence at position L-1, scaled to log2 units
          // (the 64 angles reduced mod 2 pi in fp64 once, sine and cosine in fp32;
          // every query head uses them)
          if (e < kD / 2) {
            const double ang = (double)(seg.L - 1) * sm.om64[e];
            sincosf((float)(ang - 6.283185307179586 * rint(ang * 0.15915494309189535)), &sm.qsn[e], &sm.qcs[e]);
          }
          EPI_SYNC();
          if (!ok) break;
          const float qscale = kLog2e * rsqrtf((float)kD);
          const __nv_bfloat16* qb = static_cast<const __nv_bfloat16*>(a.q) + (int64_t)seg.b * Hq * kD;
          for (int i = e; i < Hq * (kD / 2); i += kEpiThreads) {
            const int j = i / (kD / 2), pi = i % (kD / 2);
            const float sn = sm.qsn[pi], cs = sm.qcs[pi];
            const float x1v = __bfloat162float(qb[j * kD + pi]), x2v = __bfloat162float(qb[j * kD + pi + kD / 2]);
            sm.qr[j * kD + pi] = __float2bfloat16_rn((x1v * cs - x2v * sn) * qscale);
            sm.qr[j * kD + pi + kD / 2] = __float2bfloat16_rn((x1v * sn + x2v * cs) * qscale);
          }
        }
        // RoPE angle of token t0+tau and pair p: (t0*w_p mod 2pi, fp64) + tau*w_p (fp32);
        // the offsets beta of later tiles are written at the previous tile's end
        if (e < kD / 2) {
          const double ang = (double)seg.t0(0, hr) * sm.om64[e];
          sm.beta[e] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
        }
        EPI_SYNC();
        if (!ok) break;
        // head jt's reference max (log2 units; the same in all 8 owners) and this
        // owner's share of its row sum, rescaled whenever the reference moves
        float m_run = -INFINITY, l_part = 0.f;
        int ua = 0, ub = 0;  // units of the current tile
        for (int i = 0; i < seg.ntiles && ok; ++i) {
          const int t0 = seg.t0(i, hr);
          const bool has = seg.has(i, hr);    // this half holds tokens of the sequence
          const int64_t x = seg.x128(i, hr);  // its flattened 128-token tile (when it has)
          units_of(ph, seg.X0 + i, ua, ub);
          float cs[32], sn[32];
#pragma unroll
          for (int ip = 0; ip < 32; ++ip) {
            const int pi = 32 * hf + ip;
            float phs = fmaf((float)tau, sm.om32[pi], sm.beta[pi]);
            phs = fmaf(-kTwoPi, rintf(phs * kInvTwoPi), phs);
            __sincosf(phs, &sn[ip], &cs[ip]);
          }
          // per unit (one or two KV heads), in MMA order: partial scores of this frequency half
          for (int g = 0; g < lt.G && ok; ++g) {
            const GroupSm& gs = sm.grp[g];
            const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);
            for (int u = lo; u < hi; ++u) {
              const int nh = min(2, gs.nh - 2 * u);
              const int buf = kc & 1;
              if (!(ok = wwait(&sm.k_full[buf], (kc >> 1) & 1, abort_flag))) break;
              tc_fence_after();
              if (kFold) {
                // Y columns [64 hf, 64 hf + 64) of both heads: pairs (2i, 2i+1) of my 32
                // frequencies, in two passes of 16 pairs; each pass loads both heads
                // before its one wait, so a unit costs two TMEM round trips
                const uint32_t cb = tmem + lane_base + buf * kKCols + 64 * hf;
                float pa[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};  // independent chains
#pragma unroll
                for (int ps = 0; ps < 2; ++ps) {
                  float y0[32], y1[32];
                  tmem_ld32(cb + 32 * ps, y0);
                  if (nh == 2) tmem_ld32(cb + kD + 32 * ps, y1);
                  tmem_wait_ld();
                  if (ps == 1) release_acc(buf);
#pragma unroll
                  for (int i2 = 0; i2 < 16; ++i2)
                    pa[0][i2 & 3] =
                        fmaf(cs[16 * ps + i2], y0[2 * i2], fmaf(sn[16 * ps + i2], y0[2 * i2 + 1], pa[0][i2 & 3]));
                  if (nh == 2)
#pragma unroll
                    for (int i2 = 0; i2 < 16; ++i2)
                      pa[1][i2 & 3] =
                          fmaf(cs[16 * ps + i2], y1[2 * i2], fmaf(sn[16 * ps + i2], y1[2 * i2 + 1], pa[1][i2 & 3]));
                }
                float* xh = sm.x + hf * (kMaxHqTc * 128);  // this frequency half's scores
                xh[sm.order[gs.h0 + 2 * u] * 128 + tau] = (pa[0][0] + pa[0][1]) + (pa[0][2] + pa[0][3]);
                if (nh == 2)
                  xh[sm.order[gs.h0 + 2 * u + 1] * 128 + tau] = (pa[1][0] + pa[1][1]) + (pa[1][2] + pa[1][3]);
              } else {
                // per head: rotate the key's 32 frequency pairs of this half (two
                // passes of 16), stage them as bf16, and form the scores of the
                // head's qpg query heads with mma m16n8k16 (rows: the warp's 32
                // tokens in two m-tiles; k: 16 rotated x-halves, then 16 y-halves
                // per pass; n: query heads, padded to 8)
                const int gid = lane >> 2, tig = lane & 3;
                uint8_t* st = sm.kst[warp - 2];
                const uint32_t st_addr = smem_u32(st);
                for (int hh = 0; hh < nh; ++hh) {
                  const int j0 = sm.order[gs.h0 + 2 * u + hh] * qpg;
                  const uint32_t cb = tmem + lane_base + buf * kKCols + hh * kD;
                  const bool last = hh == nh - 1;
                  float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
                  for (int ps = 0; ps < 2; ++ps) {
                    float k1v[16], k2v[16];
                    tmem_ld16(cb + 32 * hf + 16 * ps, k1v);
                    tmem_ld16(cb + 64 + 32 * hf + 16 * ps, k2v);
                    tmem_wait_ld();
                    if (last && ps == 1) release_acc(buf);
                    // this lane's token: rotated x-halves (chunks 0, 1) and y-halves (2, 3)
                    uint32_t rw[16];
#pragma unroll
                    for (int w = 0; w < 8; ++w) {
                      const int ip = 16 * ps + 2 * w;
                      const float a0 = fmaf(k1v[2 * w], cs[ip], -k2v[2 * w] * sn[ip]);
                      const float a1 = fmaf(k1v[2 * w + 1], cs[ip + 1], -k2v[2 * w + 1] * sn[ip + 1]);
                      const float b0 = fmaf(k1v[2 * w], sn[ip], k2v[2 * w] * cs[ip]);
                      const float b1 = fmaf(k1v[2 * w + 1], sn[ip + 1], k2v[2 * w + 1] * cs[ip + 1]);
                      rw[w] = pack_bf16x2(a0, a1);
                      rw[8 + w] = pack_bf16x2(b0, b1);
                    }
                    __syncwarp();  // the previous pass's fragments have been read
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                      *reinterpret_cast<uint4*>(st + lane * 64 + ((c ^ ((lane >> 1) & 3)) << 4)) =
                          make_uint4(rw[4 * c], rw[4 * c + 1], rw[4 * c + 2], rw[4 * c + 3]);
                    __syncwarp();
#pragma unroll
                    for (int ks = 0; ks < 2; ++ks) {  // x-halves, then y-halves
                      // B: query head n = gid (zero past qpg), k = 2 tig .. and 2 tig + 8 ..
                      uint32_t bq0 = 0u, bq1 = 0u;
                      if (gid < qpg) {
                        const __nv_bfloat16* qrow = sm.qr + (j0 + gid) * kD + 64 * ks + 32 * hf + 16 * ps;
                        bq0 = *reinterpret_cast<const uint32_t*>(qrow + 2 * tig);
                        bq1 = *reinterpret_cast<const uint32_t*>(qrow + 2 * tig + 8);
                      }
#pragma unroll
                      for (int mt = 0; mt < 2; ++mt) {
                        // A: tokens 16 mt .. +15, k chunks 2 ks and 2 ks + 1 of the staged rows
                        const int r = 16 * mt + (lane & 7) + 8 * ((lane >> 3) & 1), ch = 2 * ks + (lane >> 4);
                        uint32_t af[4];
                        ldmatrix_x4(af, st_addr + r * 64 + ((ch ^ ((r >> 1) & 3)) << 4));
                        mma_bf16_16816(acc[mt], af, bq0, bq1);
                      }
                    }
                  }
                  // scores: token (16 mt + gid [+ 8]) of this quadrant, query heads 2 tig, 2 tig + 1
                  float* xh = sm.x + hf * (kMaxHqTc * 128);  // this frequency half's scores
#pragma unroll
                  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                      const int jj = 2 * tig + (q & 1), tt = quad * 32 + 16 * mt + gid + 8 * (q >> 1);
                      if (jj < qpg) xh[(j0 + jj) * 128 + tt] = acc[mt][q];
                    }
                }
              }
              ++kc;
            }
          }
          if (!ok) break;
          // ---- tile end: reference max, P ------------------------------------
          EPI_SYNC();  // every partial score of the tile is in x
          if (!ok) break;
          {
            const bool own = jt < Hq && sm.hunit[jt] >= ua && sm.hunit[jt] < ub;  // head computed here
            const int tb = 16 * ct;  // first token of this owner
            float sc[16];
            const float4* xr = reinterpret_cast<const float4*>(&sm.x[jt * 128 + tb]);
            const float4* xr2 = reinterpret_cast<const float4*>(&sm.x[kMaxHqTc * 128 + jt * 128 + tb]);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float4 v = own ? xr[q] : make_float4(0.f, 0.f, 0.f, 0.f);
              if (own) {  // plus the other frequency half (every score is stored each tile)
                const float4 w = xr2[q];
                v = make_float4(v.x + w.x, v.y + w.y, v.z + w.z, v.w + w.w);
              }
              sc[4 * q] = v.x;
              sc[4 * q + 1] = v.y;
              sc[4 * q + 2] = v.z;
              sc[4 * q + 3] = v.w;
            }
            const int nv = max(0, min(16, seg.L - (t0 + tb)));  // tokens inside the sequence
            float mx = -INFINITY;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              if (k >= nv || !own) sc[k] = -INFINITY;
              mx = fmaxf(mx, sc[k]);
            }
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
            // the reference moves only when the tile's max exceeds it by the threshold
            if (own && (m_run == -INFINITY || mx > m_run + kRescaleThr)) {
              l_part *= exp2f(m_run - mx);
              m_run = mx;
            }
            if (has && own && ct == 0) ta.mglob[x * Hq + jt] = m_run;
            // probabilities (bf16, the absorption's operand) straight into this tile's
            // P image; the row sum uses the rounded values
            uint32_t pk[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const __nv_bfloat162 pv = __floats2bfloat162_rn(own ? ex2_approx(sc[2 * k] - m_run) : 0.f,
                                                              own ? ex2_approx(sc[2 * k + 1] - m_run) : 0.f);
              const float2 pf = __bfloat1622float2(pv);
              l_part += pf.x + pf.y;
              pk[k] = *reinterpret_cast<const uint32_t*>(&pv);
            }
            if (has && (own || (jt >= Hq && jt < hq_pad && ua == 0))) {  // padded heads get zero rows
              // image: [token atom (64)][head row][64 tokens], 128B rows, 16-byte chunks swizzled by row % 8
              uint8_t* img = ta.pglob + x * (hq_pad * 256) + (tb >> 6) * (hq_pad * 128) + (jt >> 3) * 1024 +
                             (jt & 7) * 128;
              const int ch = (tb & 63) >> 3;
              *reinterpret_cast<uint4*>(img + ((ch ^ (jt & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
              *reinterpret_cast<uint4*>(img + (((ch + 1) ^ (jt & 7)) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
            }
          }
          if (e < kD / 2 && i + 1 < seg.ntiles) {  // RoPE phase offsets of the next pair tile
            const double ang = (double)(t0 + kPTile) * sm.om64[e];
            sm.beta[e] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
          }
          EPI_SYNC();  // x is clear and the next tile's phase offsets are in place
          if (!ok) break;
        }
        if (!ok) break;
        // ---- segment end: reference max and row sum -> this half's partial slot ----
        l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
        l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
        l_part += __shfl_xor_sync(0xffffffffu, l_part, 4);
        if (jt < Hq && ct == 0 && sm.hunit[jt] >= ua && sm.hunit[jt] < ub) {
          const int64_t slot = ph ? pair_xslot(P, a.B, seg.X0 - sp.NPm, hr) : pair_slot(pair, seg.b, hr);
          a.part_ml[(slot * Hq + jt) * 2] = m_run;
          a.part_ml[(slot * Hq + jt) * 2 + 1] = l_part;
        }
      }
#undef EPI_SYNC
    if (!ok && lane == 0) stop_peer();
  }
  tc_fence_before();
  __syncthreads();
  if (sm.abort_flag) {
    // let copies and MMAs already in flight land before the memory is released
    const long long c0 = clock64();
    while (clock64() - c0 < 4000000ll) {
    }
    if (tid == 0) atomicOr(a.err, kErrTimeout);
  }
  cluster_sync();  // the peer no longer reads this CTA's operands or arrives on its barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// factor images
// ---------------------------------------------------------------------------

struct PrepItem {
  int8_t g, s0, nh, ws;  // group, first head slot, heads, ranks
  int16_t k0;            // first rank
  int8_t kv[2];          // KV head of each of the item's heads
  int32_t off;           // byte offset in a sequence's image
};

// The decode step's latent append, done by extra blocks of the preparation
// launch: z_b = x_b [A_k | A_v] for the batch's new tokens, written to cache
// row rows[b] (Sec. III-A z = x L; Sec. III-C L_g side by side; Sec. III-D L_v).
struct StepAppend {
  const __nv_bfloat16* x;   // [B, D]
  const __nv_bfloat16* Ak;  // [D, Rk]
  const __nv_bfloat16* Av;  // [D, rv]
  const int64_t* rows;      // [B]
  int D;
  int n_blocks;             // GEMV blocks: one per 16 output columns
};

struct PrepArgs {
  int n_items;
  int64_t seq_bytes;
  double om[kD / 2];  // RoPE frequencies, fp64
  PrepItem item[kMaxItems];
  StepAppend app;
};

constexpr int kAppCols = 16;     // output columns of one GEMV block
constexpr int kAppMaxTok = 64;   // tokens of a fused append
constexpr int kAppWarps = 8;     // warps of a GEMV block, each a K range of D / 8

// d += a b for one 16 x 8 x 16 tile, bf16 inputs, fp32 accumulators (row.col).
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Four 8x8 b16 matrices from shared memory, transposed.
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// 16-byte global -> shared copies tracked per thread (cp.async groups).
__device__ __forceinline__ void cp_async16_cg(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit_group() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Four 8x8 b16 matrices from shared memory.
__device__ __forceinline__ void ldmatrix_x4_plain(uint32_t (&r)[4], uint32_t addr) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

constexpr int kAppStages = 6;    // k-steps of a warp in flight
// Dynamic shared memory of the append blocks: per warp kAppStages stages of a
// factor tile (512 B) and an x tile (16 tokens x 16 k per token m-tile), then
// the warps' partial sums.
__host__ __device__ inline int app_stage_bytes(int batch) { return 512 + ((batch + 15) / 16) * 512; }
__host__ __device__ inline size_t app_smem_bytes(int batch) {
  return (size_t)kAppWarps * kAppStages * app_stage_bytes(batch) + (size_t)kAppWarps * batch * kAppCols * 4;
}

// One GEMV block: output columns [c0, c0 + 16) of [A_k | A_v] for B <= 64
// tokens.  Warp w accumulates K range [w D / 8, (w + 1) D / 8) with mma
// m16n8k16 (tokens x K) . (K x 16 columns).  Each k-step's factor tile
// [16 k][16 columns] and x tile [tokens][16 k] go through a per-warp ring of
// cp.async stages, kAppStages k-steps ahead, so the factor stream (read once)
// keeps enough bytes in flight; ldmatrix reads the operands (.trans for the
// column-major factor).  The eight warps' partial sums are added in shared
// memory, rounded to bf16 and written to the cache rows.
__device__ __forceinline__ void step_append_block(const LayerTable& lt, const DecodeArgs& a, const StepAppend& ap,
                                                  int blk) {
  extern __shared__ __align__(128) uint8_t app_dyn[];
  const int sb = app_stage_bytes(a.B);
  float* red = reinterpret_cast<float*>(app_dyn + (size_t)kAppWarps * kAppStages * sb);  // [warp][B * 16]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;
  const int c0 = blk * kAppCols;
  const bool is_k = c0 < lt.Rk;
  const int N = is_k ? lt.Rk : lt.rv;
  const __nv_bfloat16* A = (is_k ? ap.Ak : ap.Av) + (is_k ? c0 : c0 - lt.Rk);
  const int B = a.B, D = ap.D;
  const int mt = (B + 15) / 16;  // token m-tiles
  const int kr = D / kAppWarps, kbeg = warp * kr, nks = kr / 16;
  float acc[kAppMaxTok / 16][2][4];
#pragma unroll
  for (int m = 0; m < kAppMaxTok / 16; ++m)
#pragma unroll
    for (int n = 0; n < 2; ++n)
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[m][n][q] = 0.f;
  const uint32_t rbase = smem_u32(app_dyn + (size_t)warp * kAppStages * sb);
  // stage kk: factor rows k (lane / 2), columns 8 (lane & 1) ..; x rows t, 16-byte halves h (two per row)
  auto issue = [&](int kk) {
    const uint32_t st = rbase + (uint32_t)((kk % kAppStages) * sb);
    if (kk < nks) {
      const int k0 = kbeg + 16 * kk;
      cp_async16_cg(st + (uint32_t)(((lane >> 1) * 16 + 8 * (lane & 1)) * 2),
                    A + (int64_t)(k0 + (lane >> 1)) * N + 8 * (lane & 1));
      for (int e = lane; e < 2 * 16 * mt; e += 32) {  // x rows of the token m-tiles (zero rows past B)
        const int t = e >> 1, h = e & 1;
        const uint32_t dst = st + 512 + (uint32_t)((t * 16 + 8 * h) * 2);
        if (t < B) cp_async16_cg(dst, ap.x + (int64_t)t * D + k0 + 8 * h);
        else asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" ::"r"(dst), "r"(0u) : "memory");
      }
    }
    cp_async_commit_group();
  };
#pragma unroll
  for (int q = 0; q < kAppStages - 1; ++q) issue(q);
  for (int kk = 0; kk < nks; ++kk) {
    issue(kk + kAppStages - 1);
    cp_async_wait_group<kAppStages - 1>();  // stage kk has landed (this thread's copies)
    __syncwarp();
    const uint32_t st = rbase + (uint32_t)((kk % kAppStages) * sb);
    // B fragments: matrix m = lane / 8 covers k rows 8 (m & 1) .., n columns 8 (m >> 1) ..
    uint32_t bf[4];
    const int m8 = lane >> 3, r8 = lane & 7;
    ldmatrix_x4_trans(bf, st + (uint32_t)(((8 * (m8 & 1) + r8) * 16 + 8 * (m8 >> 1)) * 2));
#pragma unroll
    for (int m = 0; m < kAppMaxTok / 16; ++m) {
      if (m >= mt) break;
      // A fragments (tokens 16 m .., k 0..15): matrix q = lane / 8 covers rows 8 (q & 1) .., k 8 (q >> 1) ..
      uint32_t af[4];
      ldmatrix_x4_plain(af, st + 512 + (uint32_t)(((16 * m + 8 * (m8 & 1) + r8) * 16 + 8 * (m8 >> 1)) * 2));
      mma_16816(acc[m][0], af[0], af[1], af[2], af[3], bf[0], bf[1]);
      mma_16816(acc[m][1], af[0], af[1], af[2], af[3], bf[2], bf[3]);
    }
    __syncwarp();  // every lane is done with the stage before it is refilled
  }
  cp_async_wait_group<0>();
  // partial sums -> shared memory: token 16 m + gid (+8), column 8 n + 2 tig (+1)
#pragma unroll
  for (int m = 0; m < kAppMaxTok / 16; ++m)
#pragma unroll
    for (int n = 0; n < 2; ++n)
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int t = 16 * m + gid + 8 * (q >> 1), c = 8 * n + 2 * tig + (q & 1);
        if (t < B) red[warp * B * kAppCols + t * kAppCols + c] = acc[m][n][q];
      }
  __syncthreads();
  __nv_bfloat16* cache = static_cast<__nv_bfloat16*>(const_cast<void*>(is_k ? a.kc : a.vc));
  for (int e = threadIdx.x; e < B * kAppCols; e += blockDim.x) {
    const int t = e / kAppCols, c = e % kAppCols;
    float v = 0.f;
#pragma unroll
    for (int w = 0; w < kAppWarps; ++w) v += red[w * B * kAppCols + e];
    const int64_t row = ap.rows[t];
    if (row < 0 || row >= a.n_rows) {
      if (c == 0) atomicOr(a.err, kErrBadRow);
      continue;
    }
    cache[row * N + (is_k ? c0 : c0 - lt.Rk) + c] = __float2bfloat16_rn(v);
  }
}

// One block writes one factor item: [nh heads][2 halves][ws rank rows]
// [64 columns] bf16, 128B-swizzled (16-byte chunk c of row r stored at chunk
// c ^ (r % 8); every half starts on a 1024-byte swizzle atom).
// Key mode: columns of B_g[:, slot].  Query-folded mode (the block's row of
// the grid covers kPrepSeqs sequences b): columns 2i and 2i+1 are
//   a_i B[:, i] + b_i B[:, i+64]  and  b_i B[:, i] - a_i B[:, i+64]
// with (a, b) the halves of RoPE(q_{b,h}, L_b - 1) * log2(e)/sqrt(d); each
// thread loads its B_g values once and writes them folded for every sequence.
// Blocks in rows after the preparation rows do the decode step's latent
// append (step_append_block), when the call has one.
constexpr int kPrepSeqs = 4;
template <bool kFold>
__global__ void __launch_bounds__(256) factor_prep_kernel(const LayerTable lt, const DecodeArgs a, const PrepArgs pa,
                                                          uint8_t* __restrict__ img) {
  griddep_launch();
  const int prep_rows = kFold ? (a.B + kPrepSeqs - 1) / kPrepSeqs : 1;
  if ((int)blockIdx.y >= prep_rows) {  // a block of the fused decode-step append
    const int blk = (blockIdx.y - prep_rows) * gridDim.x + blockIdx.x;
    if (blk < pa.app.n_blocks) step_append_block(lt, a, pa.app, blk);
    return;
  }
  const int n = blockIdx.x, bs0 = blockIdx.y * kPrepSeqs;
  const int nbs = kFold ? min(kPrepSeqs, a.B - bs0) : 1;
  const PrepItem it = pa.item[n];
  const int g = it.g, ws = it.ws, nh = it.nh;
  __shared__ float qa[kPrepSeqs][2][kD / 2], qb[kPrepSeqs][2][kD / 2];
  __shared__ int live[kPrepSeqs];
  if (kFold) {
    for (int e = threadIdx.x; e < nbs * nh * (kD / 2); e += blockDim.x) {
      const int sb = e / (nh * (kD / 2)), hh = (e / (kD / 2)) % nh, i = e % (kD / 2);
      const int b = bs0 + sb;
      const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
      if (hh == 0 && i == 0) live[sb] = L > 0;  // no tile of an empty sequence is ever processed
      const int kv = it.kv[hh];
      // angle (L-1) w_i reduced mod 2 pi in fp64, sine and cosine in fp32
      const double ang = (double)max(L - 1, 0) * pa.om[i];
      float sn, cs;
      sincosf((float)(ang - 6.283185307179586 * rint(ang * 0.15915494309189535)), &sn, &cs);
      const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(a.q) + ((int64_t)b * lt.Hq + kv) * kD;
      const float x1 = __bfloat162float(q[i]), x2 = __bfloat162float(q[i + kD / 2]);
      const float sc = kLog2e * rsqrtf((float)kD);
      qa[sb][hh][i] = (x1 * cs - x2 * sn) * sc;
      qb[sb][hh][i] = (x1 * sn + x2 * cs) * sc;
    }
    __syncthreads();
  }
  const int64_t ld = (int64_t)lt.grp_nh[g] * kD;
  // thread -> (head, row, 8-column chunk): nh x ws rows x 16 chunks (2 halves x 8)
  for (int idx = threadIdx.x; idx < nh * ws * 16; idx += blockDim.x) {
    const int hh = idx / (ws * 16), r = (idx >> 4) % ws, ch = idx & 15;
    const int half = ch >> 3, c8 = ch & 7;
    const __nv_bfloat16* __restrict__ Bs =
        static_cast<const __nv_bfloat16*>(a.Bk) + lt.grp_boff[g] + (it.s0 + hh) * kD + (int64_t)(it.k0 + r) * ld;
    const int64_t doff = it.off + (hh * 2 + half) * (ws * 128) + r * 128 + ((c8 ^ (r & 7)) << 4);
    if (kFold) {
      // output columns col = 64*half + 8*c8 + t, t even/odd -> pair i = col/2 = 32*half + 4*c8 + t/2:
      // the x-halves B[:, i] and y-halves B[:, i+64] of four pairs, one 8-byte load each
      const int i0 = 32 * half + 4 * c8;
      const uint2 xr = *reinterpret_cast<const uint2*>(Bs + i0);
      const uint2 yr = *reinterpret_cast<const uint2*>(Bs + kD / 2 + i0);
      const __nv_bfloat16* xh = reinterpret_cast<const __nv_bfloat16*>(&xr);
      const __nv_bfloat16* yh = reinterpret_cast<const __nv_bfloat16*>(&yr);
      float x[4], y[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        x[t] = __bfloat162float(xh[t]);
        y[t] = __bfloat162float(yh[t]);
      }
      for (int sb = 0; sb < nbs; ++sb) {
        if (!live[sb]) continue;
        uint4 out;
        __nv_bfloat162* o2 = reinterpret_cast<__nv_bfloat162*>(&out);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float qa_ = qa[sb][hh][i0 + t], qb_ = qb[sb][hh][i0 + t];
          o2[t] = __floats2bfloat162_rn(fmaf(qa_, x[t], qb_ * y[t]), fmaf(qb_, x[t], -qa_ * y[t]));
        }
        *reinterpret_cast<uint4*>(img + (int64_t)(bs0 + sb) * pa.seq_bytes + doff) = out;
      }
    } else {
      *reinterpret_cast<uint4*>(img + doff) = *reinterpret_cast<const uint4*>(Bs + 64 * half + 8 * c8);
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

// Bytes of one copy of all factor images: sum over heads of r_g * 128 columns * 2.
size_t image_bytes_of(const LayerTable& lt) {
  size_t n = 0;
  for (int g = 0; g < lt.G; ++g) n += (size_t)lt.grp_nh[g] * lt.grp_rank[g] * 256;
  return n;
}

// Tensor maps depend only on the buffers and the layer: cache the last few.
struct MapsKey {
  const void* kc;
  int64_t n_rows;
  int Rk;
  const void* img;
  int64_t img_rows;
  bool operator==(const MapsKey& o) const {
    return kc == o.kc && n_rows == o.n_rows && Rk == o.Rk && img == o.img && img_rows == o.img_rows;
  }
};
constexpr int kMapsCache = 64;
std::mutex g_maps_mu;
MapsKey g_maps_key[kMapsCache];
Maps g_maps_val[kMapsCache];
int g_maps_n = 0, g_maps_next = 0;

bool build_maps(const LayerTable& lt, const DecodeArgs& a, const void* img, int64_t img_rows, Maps& maps) {
  std::memset(&maps, 0, sizeof(maps));
  const uint64_t rows = (uint64_t)std::max<int64_t>(1, a.n_rows);
  if (!(make_tmap_2d_bf16(&maps.kc64, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 64, kTile, CU_TENSOR_MAP_SWIZZLE_128B) &&
        make_tmap_2d_bf16(&maps.kc32, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 32, kTile, CU_TENSOR_MAP_SWIZZLE_64B) &&
        make_tmap_2d_bf16(&maps.kc16, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 16, kTile, CU_TENSOR_MAP_SWIZZLE_32B)))
    return false;
  // the factor images as rows of 128 bytes (64 bf16), boxes of 16 .. 128 rows
  const uint32_t box_rows[4] = {16, 32, 64, 128};
  for (int i = 0; i < 4; ++i)
    if (!make_tmap_2d_bf16(&maps.im[i], img, 64, (uint64_t)std::max<int64_t>(img_rows, 128), 128, 64, box_rows[i],
                           CU_TENSOR_MAP_SWIZZLE_NONE))
      return false;
  return true;
}

static_assert(sizeof(Smem<true>) + 1024 <= 232448, "shared memory of the query-folded kernel");
static_assert(sizeof(Smem<false>) + 1024 <= 232448, "shared memory of the key-mode kernel");

template <bool kFold>
cudaError_t set_smem_attr() {
  static int attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  const bool dev_ok = dev >= 0 && dev < 64;
  if (dev_ok && attr_done[dev]) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(decode_tc_kernel<kFold>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)(sizeof(Smem<kFold>) + 1024));
  if (e == cudaSuccess && dev_ok) attr_done[dev] = 1;
  return e;
}

// CTA pairs that can be resident at once (at most half the SMs): the scores
// kernel is persistent, so its grid is exactly that many pairs.
template <bool kFold>
int pairs_of_device() {
  static int pairs[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (pairs[dev]) return pairs[dev];
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (set_smem_attr<kFold>() != cudaSuccess) return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (sms / 2));
  cfg.blockDim = dim3(Ring<kFold>::kThreads);
  cfg.dynamicSmemBytes = sizeof(Smem<kFold>) + 1024;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, decode_tc_kernel<kFold>, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 0;
  }
  pairs[dev] = std::min(n, sms / 2);
  return pairs[dev];
}

template <bool kFold>
cudaError_t launch_mode(const LayerTable& lt, const DecodeArgs& a, const Maps& maps, const TcArgs& ta,
                        const PrepArgs& pa, cudaStream_t s) {
  cudaError_t e = set_smem_attr<kFold>();
  if (e != cudaSuccess) return e;
  const int prep_rows = kFold ? (a.B + kPrepSeqs - 1) / kPrepSeqs : 1;
  const int app_rows = (pa.app.n_blocks + pa.n_items - 1) / pa.n_items;
  const size_t app_smem = pa.app.n_blocks ? app_smem_bytes(a.B) : 0;
  if (app_smem) {
    e = cudaFuncSetAttribute(factor_prep_kernel<kFold>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)app_smem);
    if (e != cudaSuccess) return e;
  }
  factor_prep_kernel<kFold><<<dim3(pa.n_items, prep_rows + app_rows), 256, app_smem, s>>>(
      lt, a, pa, static_cast<uint8_t*>(a.extra));
  e = hook_launched(a.hook, s);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * ta.n_pairs);
  cfg.blockDim = dim3(Ring<kFold>::kThreads);
  cfg.dynamicSmemBytes = sizeof(Smem<kFold>) + 1024;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, decode_tc_kernel<kFold>, maps, lt, a, ta);
  return e != cudaSuccess ? e : hook_launched(a.hook, s);
}

// Order in which a tile's key groups are processed: the latent ring holds the
// pieces of the group in use while it fills with the next group's, so groups
// with many pieces are interleaved with groups with few (largest first, then
// smallest, ...), which keeps the piece counts of neighbours (cyclically: the
// last group is followed by the next tile's first) within the ring.
void group_order(const LayerTable& lt, int* order) {
  int idx[kMaxGroupsTc];
  int8_t w[kMaxPieces];
  int16_t k[kMaxPieces];
  int np[kMaxGroupsTc];
  for (int g = 0; g < lt.G; ++g) {
    idx[g] = g;
    np[g] = make_pieces(lt.grp_rank[g], w, k);
  }
  std::stable_sort(idx, idx + lt.G, [&](int x, int y) { return np[x] > np[y]; });
  for (int i = 0, lo = 0, hi = lt.G - 1; lo <= hi; ++i) order[i] = (i & 1) ? idx[hi--] : idx[lo++];
}

// Units, items and per-group tables of a layer (groups in processing order).
// Returns false when the layer does not fit the tables.
bool build_tables(const LayerTable& lt, TcArgs& ta, PrepArgs& pa) {
  std::memset(&ta, 0, sizeof(ta));
  std::memset(&pa, 0, sizeof(pa));
  ta.hq_pad = hq_pad_of(lt.Hq);
  if (lt.G > kMaxGroupsTc) return false;
  int gorder[kMaxGroupsTc];
  group_order(lt, gorder);
  int pos = 0, item = 0, off = 0, unit = 0;
  for (int gi = 0; gi < lt.G; ++gi) {
    const int g = gorder[gi];
    GroupSm& gs = ta.grp[gi];
    gs.roff = lt.grp_roff[g];
    gs.rank = (int16_t)lt.grp_rank[g];
    int16_t kk[kMaxPieces];
    gs.np = (int8_t)make_pieces(lt.grp_rank[g], gs.w, kk);
    if (gs.np > kMaxPieces || gs.np > std::min(Ring<true>::NA, Ring<false>::NA)) return false;
    for (int p = 0; p < gs.np; ++p) gs.k[p] = kk[p];
    gs.h0 = (int8_t)pos;
    gs.nh = (int8_t)lt.grp_nh[g];
    gs.nu = (int8_t)((lt.grp_nh[g] + 1) / 2);
    gs.u0 = (int16_t)unit;
    gs.i0 = (int16_t)item;
    for (int sl = 0; sl < lt.grp_nh[g]; ++sl)
      for (int h = 0; h < lt.Hkv; ++h)
        if (lt.head_group[h] == g && lt.head_slot[h] == sl) {
          if (pos >= kMaxHqTc) return false;
          ta.order[pos++] = (int16_t)h;
          for (int jj = 0; jj < lt.qpg; ++jj) ta.hunit[h * lt.qpg + jj] = (int8_t)(unit + sl / 2);
        }
    for (int s0 = 0; s0 < lt.grp_nh[g]; s0 += 2) {
      const int nh = std::min(2, lt.grp_nh[g] - s0);
      if (unit >= kMaxUnits) return false;
      ta.uitem[unit++] = (int16_t)item;
      for (int p = 0; p < gs.np; ++p) {
        if (item >= kMaxItems) return false;
        const int w = gs.w[p], bytes = nh * w * 256;
        PrepItem& pi = pa.item[item];
        pi.g = (int8_t)g;
        pi.s0 = (int8_t)s0;
        for (int hh = 0; hh < nh; ++hh)
          for (int h = 0; h < lt.Hkv; ++h)
            if (lt.head_group[h] == g && lt.head_slot[h] == s0 + hh) pi.kv[hh] = (int8_t)h;
        pi.nh = (int8_t)nh;
        pi.ws = (int8_t)w;
        pi.k0 = gs.k[p];
        pi.off = off;
        ta.item[item] = (uint32_t)off | ((uint32_t)(bytes >> 12) << 26);
        off += bytes;
        ++item;
      }
    }
  }
  ta.n_units = unit;
  ta.uitem[unit] = (int16_t)item;
  ta.n_items = item;
  pa.n_items = item;
  pa.seq_bytes = off;
  ta.fimg_seq_bytes = off;
  return true;
}

// RoPE frequencies w_i = theta^(-2i/d) in fp64 (positions reach 1e5 and more,
// so the angle t w_i needs the extra precision before its reduction mod 2 pi).
void rope_freqs(float theta, double* om) {
  for (int i = 0; i < kD / 2; ++i) om[i] = std::exp2(-2.0 * i / kD * std::log2((double)theta));
}

// Workspace layout of the tensor-core path (after the split partials):
// factor images, then the per-tile P images, then the per-tile reference maxima.
struct ExtraLayout {
  size_t img, p, m, total;
};

ExtraLayout extra_layout(const LayerTable& lt, int batch, int64_t n_rows) {
  ExtraLayout x;
  const int64_t nt = max_tiles(n_rows, batch);
  x.img = align_up(lt.qpg == 1 ? image_bytes_of(lt) * std::max(batch, 1) : image_bytes_of(lt), 256);
  x.p = align_up((size_t)nt * hq_pad_of(lt.Hq) * 256, 256);
  x.m = align_up((size_t)nt * lt.Hq * sizeof(float), 256);
  x.total = x.img + x.p + x.m;
  return x;
}

}  // namespace

bool tc_decode_supports(const LayerTable& lt, int dtype) {
  if (dtype != DCK_BF16 || lt.d != kD) return false;
  if (lt.Hq > kMaxHqTc || lt.qpg > kMaxQPerKv || lt.G > kMaxGroupsTc) return false;
  if (lt.rv % 128 || (lt.rv / 128) * hq_pad_of(lt.Hq) > 512) return false;
  for (int g = 0; g < lt.G; ++g)
    if (lt.grp_rank[g] > 256 || lt.grp_rank[g] % 16) return false;
  static thread_local TcArgs ta;
  static thread_local PrepArgs pa;
  return build_tables(lt, ta, pa);
}

// Extra workspace of the tensor-core path.
size_t tc_decode_extra_ws(const LayerTable& lt, int batch, int64_t n_rows) {
  if (!tc_decode_supports(lt, DCK_BF16)) return 0;
  return extra_layout(lt, batch, n_rows).total;
}

// The fused decode-step append takes up to 64 tokens and widths D that split
// into eight warp ranges of 16-wide k-steps.
bool tc_step_append_supports(const LayerTable& lt, int D, int batch) {
  return batch >= 1 && batch <= kAppMaxTok && D % (kAppWarps * 16) == 0 && lt.Rk % kAppCols == 0 &&
         lt.rv % kAppCols == 0;
}

// CTA pairs of the tensor-core path on the current device (0 if it cannot run).
int tc_decode_pairs(const LayerTable& lt) { return lt.qpg == 1 ? pairs_of_device<true>() : pairs_of_device<false>(); }

cudaError_t launch_decode_tc(const LayerTable& lt, const DecodeArgs& a, const TcStepAppend* app, cudaStream_t s) {
  const bool fold = lt.qpg == 1;
  if (!a.extra || a.n_items < 2 || (a.n_items & 1)) return cudaErrorInvalidValue;
  static thread_local TcArgs ta;
  static thread_local PrepArgs pa;
  if (!build_tables(lt, ta, pa)) return cudaErrorInvalidValue;
  if (app) {
    if (!tc_step_append_supports(lt, app->D, a.B)) return cudaErrorInvalidValue;
    pa.app.x = static_cast<const __nv_bfloat16*>(app->x);
    pa.app.Ak = static_cast<const __nv_bfloat16*>(app->A_k);
    pa.app.Av = static_cast<const __nv_bfloat16*>(app->A_v);
    pa.app.rows = app->rows;
    pa.app.D = app->D;
    pa.app.n_blocks = (lt.Rk + lt.rv) / kAppCols;
  }
  rope_freqs(a.theta, ta.om);
  std::memcpy(pa.om, ta.om, sizeof(ta.om));
  const ExtraLayout xl = extra_layout(lt, a.B, a.n_rows);
  uint8_t* base = static_cast<uint8_t*>(a.extra);
  ta.n_pairs = a.n_items / 2;
  ta.pglob = base + xl.img;
  ta.mglob = reinterpret_cast<float*>(base + xl.img + xl.p);
  ta.max_tiles = max_tiles(a.n_rows, a.B);
  const int64_t img_rows = (int64_t)(xl.img >> 7);
  const MapsKey key{a.kc, a.n_rows, lt.Rk, base, img_rows};
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
    if (!build_maps(lt, a, base, img_rows, maps)) return cudaErrorInvalidValue;
    std::lock_guard<std::mutex> lk(g_maps_mu);
    g_maps_key[g_maps_next] = key;
    g_maps_val[g_maps_next] = maps;
    g_maps_next = (g_maps_next + 1) % kMapsCache;
    g_maps_n = std::min(g_maps_n + 1, kMapsCache);
  }
  cudaError_t e = hook_begin(a.hook, s);
  if (e != cudaSuccess) return e;
  e = fold ? launch_mode<true>(lt, a, maps, ta, pa, s) : launch_mode<false>(lt, a, maps, ta, pa, s);
  if (e != cudaSuccess) return e;
  TcRegions r;
  r.pglob = ta.pglob;
  r.mglob = ta.mglob;
  r.max_tiles = ta.max_tiles;
  r.hq_pad = ta.hq_pad;
  r.early_values = true;
  e = launch_absorb_tc(lt, a, r, s);
  return e != cudaSuccess ? e : hook_launched(a.hook, s);
}

}  // namespace dck
