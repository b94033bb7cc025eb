// Tensor-core (tcgen05) decode attention over DynaCalKV latent caches, bf16:
// the scores kernel (key reconstruction, RoPE, scores, online softmax).
//
// One persistent CTA per SM walks its share of 128-token tiles (see
// DecodeArgs).  For every tile and every key group g (Sec. III-C) the group's
// latent tile C_g [128 tokens x r_g] meets, on the tensor cores, the factor
// columns of the group's KV heads, two heads per MMA where the group has them
// (tcgen05.mma, M = 128 tokens, N = 256 or 128, K = r_g, fp32 accumulator in
// TMEM).  A pair shares every read of the latent operand: one-head MMAs that
// read fresh shared-memory operands run the tensor pipe at about half rate.
// Two 256-column accumulators (all of TMEM) let the epilogue read one unit
// while the tensor core computes the next.  Per head:
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
// bytes each, in consumption order), so each item arrives with one 1-D bulk copy.
//
// Scores are in log2 units; the online softmax keeps a per-head reference max
// that moves only when a tile's max exceeds it by 8 (probabilities <= 256).
// Each tile's probabilities P (bf16, laid out as the B operand of the value
// absorption) and the reference maxima they were computed with go to the
// workspace; at the end of each sequence segment the reference max and the
// row sum (over the rounded P) are written as the segment's split partial.
// The absorption kernel (absorb_tc.cu) forms U = C_v^T P from them.
//
// Warp roles (384 threads query-folded, 352 key mode).  Every TMA or
// bulk-copy instruction costs its issuing thread a long round trip, so loads
// are issued by two producer warps, each putting several copies (one per lane)
// into one instruction:
//   warp 0     latent pieces of C_g (ring A)
//   warp 10    factor items (ring W; query-folded mode: one ring per MMA thread)
//   warp 1     TMEM owner; its lane 0 issues MMAs.  On this GPU every barrier
//              test, commit or fence costs the issuing thread a dependent round
//              trip of 100-500 cycles, longer than the MMAs of a factor item, so
//              in query-folded mode lane 0 of warp 11 issues every other unit
//              into the other accumulator and the two threads' bookkeeping
//              overlaps the other's MMAs
//   warps 2-9  epilogue: each TMEM lane quadrant (32 tokens) is served by two
//              warps that split the 64 RoPE frequency pairs of a head; their
//              partial scores go to one shared-memory array per frequency
//              half, summed at the tile end.
// Every wait is bounded (about 2 s); on expiry the CTA stops issuing work,
// records kErrTimeout, waits for work in flight and still releases TMEM.
//
// Shared-memory operand layouts (128B swizzle unless noted):
//   A slot  [128 tokens][w ranks] K-major, w in {64, 32, 16} with 128/64/32B
//           swizzle: UMMA operand A of the reconstruction;
//   W slot  [nh heads][2 halves][w ranks][64 columns] MN-major: operand B
//           (N = 128 nh, the 64-column atoms w * 128 bytes apart);
// P ([2 token atoms][Hq_pad heads][64 tokens] bf16, K-major: the absorption's
// operand B) is written straight to the workspace by the tile-end owners.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "tc_common.cuh"
#include "tc_host.h"
#include "tmap.h"

#ifndef DCK_TC_TRACE
#define DCK_TC_TRACE(code) ((void)0)
#endif
#ifndef DCK_TC_TRACE_FLUSH
#define DCK_TC_TRACE_FLUSH() ((void)0)
#endif

namespace dck {
namespace {

using namespace sm100;
using namespace tc;

constexpr int kD = 128;
constexpr int kSlot = 16384;     // latent slots
constexpr int kSlotW = 32768;    // factor slots: up to 2 heads x 64 ranks x 128 columns
constexpr int kNA = 4;           // latent-piece ring depth
constexpr int kMaxGroupsTc = 16;
constexpr int kMaxPieces = 5;
constexpr int kMaxHqTc = 32;
constexpr int kMaxItems = 256;
constexpr int kMaxUnits = 32;
constexpr int kEpiThreads = 256;
constexpr float kRescaleThr = 8.f;  // log2 units: probabilities stay <= 256
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kKCols = 256;    // TMEM columns of one key accumulator
constexpr float kTwoPi = 6.28318530717958647692f;
constexpr float kInvTwoPi = 0.15915494309189533577f;
constexpr float kLog2e = 1.4426950408889634f;

template <bool kFold>
struct Ring {
  static constexpr int NW = kFold ? 4 : 3;    // factor-item slots (key mode keeps 16 KB for queries)
  // MMA-issuing threads, each with its own factor ring: two in query-folded
  // mode; key mode's units carry up to four items, which one thread's ring of
  // all four slots streams better
  static constexpr int kMma = kFold ? 2 : 1;
  static constexpr int NWt = NW / kMma;       // slots of one MMA thread's ring
  static constexpr int kThreads = kFold ? 384 : 352;
};

struct Maps {
  CUtensorMap kc64, kc32, kc16;
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
};

struct TcArgs {
  int hq_pad;
  int n_items;                   // factor items per tile
  int64_t fimg_seq_bytes;        // factor image bytes per sequence (query-folded mode)
  const uint8_t* fimg;           // factor images (workspace)
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
  uint8_t a[kNA][kSlot];
  uint8_t w[Ring<kFold>::NW][kSlotW];
  // scores [frequency half][query head][token]: each half's partial scores by
  // plain stores, summed at the tile end
  float x[2 * kMaxHqTc * 128];
  // key mode: rotated queries * log2(e)/sqrt(d), bf16 [query head][d] (the
  // B operand of the warps' score MMAs), and per epilogue warp a staging tile
  // of its 32 tokens' rotated keys [token][32] bf16 (the A operand), 16-byte
  // chunks swizzled by (token / 2) % 4
  __nv_bfloat16 qr[kFold ? 2 : kMaxHqTc * kD];
  uint8_t kst[kFold ? 1 : kEpiThreads / 32][kFold ? 16 : 32 * 64];
  double om64[kD / 2];
  float om32[kD / 2];
  float beta[kD / 2];
  uint64_t a_full[kNA], a_empty[kNA];
  uint64_t w_full[Ring<kFold>::NW], w_empty[Ring<kFold>::NW];
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

// ---------------------------------------------------------------------------
// the scores kernel
// ---------------------------------------------------------------------------

template <bool kFold>
__global__ void __launch_bounds__(Ring<kFold>::kThreads, 1)
    decode_tc_kernel(const __grid_constant__ Maps maps, const LayerTable lt, const DecodeArgs a,
                     const __grid_constant__ TcArgs ta) {
  constexpr int NW = Ring<kFold>::NW, kMma = Ring<kFold>::kMma, NWt = Ring<kFold>::NWt;
  constexpr int kThreads = Ring<kFold>::kThreads;
  extern __shared__ uint8_t smem_raw[];
  Smem<kFold>& sm =
      *reinterpret_cast<Smem<kFold>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  const int hq_pad = ta.hq_pad;
  const int Hq = lt.Hq, qpg = lt.qpg;
  griddep_launch();  // the absorption kernel may start streaming values as CTAs finish

  // ---- setup -------------------------------------------------------------
  if (tid == 0) {
    for (int i = 0; i < kNA; ++i) {
      mbar_init(&sm.a_full[i], 1);
      mbar_init(&sm.a_empty[i], kMma);  // released by every MMA thread
    }
    for (int i = 0; i < NW; ++i) {
      mbar_init(&sm.w_full[i], 1);
      mbar_init(&sm.w_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.k_full[i], 1);
      mbar_init(&sm.k_empty[i], kEpiThreads / 32);
    }
    mbar_init(&sm.epi_bar, kEpiThreads / 32);
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (tid < lt.G) sm.grp[tid] = ta.grp[tid];
  if (tid < lt.Hkv) sm.order[tid] = ta.order[tid];
  if (tid <= ta.n_units) sm.uitem[tid] = ta.uitem[tid];
  if (tid < Hq) sm.hunit[tid] = ta.hunit[tid];
  if (tid < kD / 2) {
    sm.om64[tid] = ta.om[tid];
    sm.om32[tid] = (float)ta.om[tid];
  }
  // Work of this CTA: main tiles [x0, x1) (every unit), then units [u_lo, u_hi)
  // of the flattened (extra tile, unit) list, every extra tile a segment of its own.
  const int U = ta.n_units;
  const int NT = tile_count(a, reinterpret_cast<int*>(sm.x));
  const Split sp(NT, a.n_items, a.split_extra != 0);
  // the per-tile stores are sized for non-overlapping sequences; more tiles
  // than that is reported as invalid input and nothing is computed
  const bool fits = NT <= ta.max_tiles;
  if (!fits && tid == 0 && blockIdx.x == 0) atomicOr(a.err, kErrBadSeq);
  const int x0 = fits ? sp.main_begin(blockIdx.x, a.n_items) : 0;
  const int x1 = fits ? sp.main_begin(blockIdx.x + 1, a.n_items) : 0;
  const int xu = sp.R * U;
  const int u_lo = fits ? (int)((int64_t)blockIdx.x * xu / a.n_items) : 0;
  const int u_hi = fits ? (int)((int64_t)(blockIdx.x + 1) * xu / a.n_items) : 0;
  const int xe0 = sp.NTm + (u_lo < u_hi ? u_lo / U : 0), xe1 = sp.NTm + (u_lo < u_hi ? (u_hi - 1) / U + 1 : 0);
  int bm, pm, bx, px;
  tile_find(a, reinterpret_cast<const int*>(sm.x), x0, bm, pm);
  tile_find(a, reinterpret_cast<const int*>(sm.x), xe0, bx, px);
  const Walker walk_m{bm, pm, x0, x1, false}, walk_x{bx, px, xe0, xe1, true};
  const bool has_work = x0 < x1 || xe0 < xe1;
  const int64_t xbase = extra_slot_base(a.n_items, a.B);
  // units [ua, ub) of flattened tile x in phase ph (0: main, 1: extra)
  auto units_of = [&](int ph, int x, int& ua, int& ub) {
    ua = 0;
    ub = U;
    if (ph) {
      const int e = x - sp.NTm;
      ua = max(u_lo - e * U, 0);
      ub = min(u_hi - e * U, U);
    }
  };
  for (int i = tid; i < (int)(sizeof(sm.x) / sizeof(float)); i += kThreads) sm.x[i] = 0.f;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  Segment seg;
  DCK_TC_TRACE(0);

  // Factor items of one unit into MMA thread rw's ring (query-folded mode): up to
  // NWt bulk copies per instruction, one per lane, as their slots come free.
  auto put_unit_items = [&](int rw, int& wc, int n, int np, const uint8_t* img, uint64_t pol) -> bool {
    for (int p0 = 0; p0 < np;) {
      const int nb = claim_slots(sm.w_empty + rw * NWt, NWt, wc, np - p0, lane, abort_flag);
      if (nb == 0) return false;
      DCK_TC_TRACE(30 + nb);
      if (lane < nb) {
        const int sl = rw * NWt + (wc + lane) % NWt;
        const uint32_t it = ta.item[n + p0 + lane];
        const uint32_t bytes = (it >> 26) << 12;
        mbar_expect_tx(&sm.w_full[sl], bytes);
        bulk_load(sm.w[sl], img + (it & 0x03FFFFFFu), bytes, &sm.w_full[sl], pol);
      }
      __syncwarp();
      wc += nb;
      p0 += nb;
    }
    return true;
  };

  if (warp == 0) {
    // ---- latent pieces, issued as soon as their slots are free; in
    // query-folded mode also the factor items of MMA thread 1, in the order
    // that thread consumes them (a group's pieces, then its units' items) ------
    if (has_work) {
      const uint64_t pol = policy_evict_first();
      const uint64_t pol_w = policy_evict_last();
      int a_cnt = 0, wc = 0, kc = 0;
      bool ok = true, images_ready = false;
      for (int ph = 0; ph < 2 && ok; ++ph)
        for (Walker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
          const uint8_t* img = ta.fimg + (kFold ? (int64_t)seg.b * ta.fimg_seq_bytes : 0);
          for (int i = 0; i < seg.ntiles && ok; ++i) {
            const int64_t yrow = seg.row0 + seg.t_begin + (int64_t)kTile * i;
            if (lane == 0 && i + 1 < seg.ntiles) {  // next tile's latent rows toward L2
              const int64_t r0 = yrow + kTile, nr = a.n_rows - r0 < kTile ? a.n_rows - r0 : (int64_t)kTile;
              if (nr > 0)
                prefetch_l2(static_cast<const __nv_bfloat16*>(a.kc) + r0 * lt.Rk, (uint32_t)(nr * lt.Rk * 2));
            }
            int ua, ub;
            units_of(ph, seg.x0 + i, ua, ub);
            for (int g = 0; g < lt.G && ok; ++g) {
              const GroupSm& gs = sm.grp[g];
              const int np = gs.np;
              const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);
              if (lo >= hi) continue;  // none of the group's units in this piece of work
              for (int p0 = 0; p0 < np && ok;) {
                const int nb = claim_slots(sm.a_empty, kNA, a_cnt, np - p0, lane, abort_flag);
                ok = nb > 0;
                if (!ok) break;
                if (lane < nb) {
                  const int sl = (a_cnt + lane) % kNA;
                  const int w = gs.w[p0 + lane];
                  const CUtensorMap* m = w == 64 ? &maps.kc64 : (w == 32 ? &maps.kc32 : &maps.kc16);
                  mbar_expect_tx(&sm.a_full[sl], kTile * w * 2);
                  tma_load_2d_hint(sm.a[sl], m, &sm.a_full[sl], gs.roff + gs.k[p0 + lane], (int32_t)yrow, pol);
                }
                __syncwarp();
                a_cnt += nb;
                p0 += nb;
              }
              if (kMma == 2)
                for (int u = lo; u < hi && ok; ++u, ++kc) {
                  if ((kc & 1) != 1) continue;  // MMA thread 0's unit
                  if (!images_ready) {          // the images are written by the preparation kernel
                    griddep_wait();
                    images_ready = true;
                  }
                  ok = put_unit_items(1, wc, gs.i0 + u * np, np, img, pol_w);
                }
            }
          }
        }
    }
  } else if (warp == 10) {
    // ---- factor items: several bulk copies per instruction (query-folded
    // mode: the ring of MMA thread 0 only) --------------------------------------
    if (has_work) {
      const uint64_t pol = policy_evict_last();
      griddep_wait();  // the images are written by the preparation kernel
      int w_cnt = 0;
      bool ok = true;
      int wc = 0, kc = 0;  // items put into MMA thread 0's ring, units so far
      for (int ph = 0; ph < 2 && ok; ++ph)
        for (Walker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
          const uint8_t* img = ta.fimg + (kFold ? (int64_t)seg.b * ta.fimg_seq_bytes : 0);
          for (int i = 0; i < seg.ntiles && ok; ++i) {
            int ua, ub;
            units_of(ph, seg.x0 + i, ua, ub);
            if (kMma == 1) {  // one ring: claims may span units (the units' items are contiguous)
              const int n_end = sm.uitem[ub];
              for (int n0 = sm.uitem[ua]; n0 < n_end && ok;) {
                const int nb = claim_slots(sm.w_empty, NW, w_cnt, min(NW, n_end - n0), lane, abort_flag);
                ok = nb > 0;
                if (!ok) break;
                if (lane < nb) {
                  const int sl = (w_cnt + lane) % NW;
                  const uint32_t it = ta.item[n0 + lane];
                  const uint32_t bytes = (it >> 26) << 12;
                  mbar_expect_tx(&sm.w_full[sl], bytes);
                  bulk_load(sm.w[sl], img + (it & 0x03FFFFFFu), bytes, &sm.w_full[sl], pol);
                }
                __syncwarp();
                w_cnt += nb;
                n0 += nb;
              }
              continue;
            }
            for (int g = 0; g < lt.G && ok; ++g) {
              const GroupSm& gs = sm.grp[g];
              const int np = gs.np;
              const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);
              for (int u = lo; u < hi && ok; ++u, ++kc)
                if ((kc & 1) == 0) ok = put_unit_items(0, wc, gs.i0 + u * np, np, img, pol);
            }
          }
        }
    }
  } else if (warp == 1 || (kMma == 2 && warp == 11)) {
    // ---- MMA issuers: lane 0 of warp 1 (and of warp 11 in query-folded mode)
    // runs the schedule of every kMma-th unit into its own accumulator, so one
    // thread's barrier tests and commits overlap the other's MMAs.  Each thread
    // owns a factor ring (single consumer) and observes every latent piece's
    // fill in order, releasing the pieces of groups it has no unit in, so no
    // parity test can see a stale phase. ---------------------------------------
    if (lane == 0 && has_work) {
      const int t = warp == 1 ? 0 : 1;
      uint64_t* wfull = sm.w_full + t * NWt;
      uint64_t* wempty = sm.w_empty + t * NWt;
      int a_cnt = 0, w_cnt = 0, kc = 0, own = 0;
      bool ok = true;
      for (int ph = 0; ph < 2 && ok; ++ph)
      for (Walker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
        for (int i = 0; i < seg.ntiles && ok; ++i) {
          int ua, ub;
          units_of(ph, seg.x0 + i, ua, ub);
          for (int g = 0; g < lt.G && ok; ++g) {
            const GroupSm& gs = sm.grp[g];
            const int np = gs.np;
            const int lo = max(ua - gs.u0, 0), hi = min(ub - gs.u0, (int)gs.nu);  // the group's units here
            if (lo >= hi) continue;
            const int a_base = a_cnt;
            const int uf = lo + (kMma == 2 ? (((kc & 1) == t) ? 0 : 1) : 0);  // this thread's first unit of the group
            if (uf >= hi)  // none: observe the group's pieces, then release them
              for (int p = 0; p < np && ok; ++p) {
                const int sl = (a_base + p) % kNA;
                if ((ok = mbar_wait(&sm.a_full[sl], ((a_base + p) / kNA) & 1, abort_flag))) mbar_arrive(&sm.a_empty[sl]);
              }
            for (int u = uf; u < hi && ok; u += kMma) {
              const int nh = min(2, gs.nh - 2 * u);
              const uint32_t idesc_k = idesc_bf16(128, kD * nh, false, true);
              const int kg = kc + (u - lo);                        // unit index of the CTA
              const int buf = kMma == 2 ? t : (kg & 1);
              const int use = kMma == 2 ? own : (kg >> 1);         // earlier units in this accumulator
              // readiness of this unit's factor items (and, at this thread's first
              // unit of the group, latent pieces): independent tests whose latencies
              // overlap; blocking waits, in ring order, only for what is not there
              // yet.  Only items within one turn of the ring are tested: the previous
              // use of their slot has been consumed, so the parity test cannot see a
              // stale phase.
              uint32_t miss = 0;
#pragma unroll
              for (int p = 0; p < kMaxPieces; ++p)
                if (p < np) {
                  const int c = w_cnt + p;
                  if (p >= NWt || !mbar_test(&wfull[c % NWt], (c / NWt) & 1)) miss |= 1u << p;
                  if (u == uf && !mbar_test(&sm.a_full[(a_base + p) % kNA], ((a_base + p) / kNA) & 1))
                    miss |= 0x100u << p;
                }
              // the first piece and item before the accumulator: the operand streams do
              // not depend on the epilogue, so the MMAs can start as soon as it is free
              if ((miss & 0x100u) && !(ok = mbar_wait(&sm.a_full[a_base % kNA], (a_base / kNA) & 1, abort_flag))) break;
              if ((miss & 1u) && !(ok = mbar_wait(&wfull[w_cnt % NWt], (w_cnt / NWt) & 1, abort_flag))) break;
              miss &= ~0x101u;
              DCK_TC_TRACE(12);
              if (use >= 1) {  // the epilogue has read this accumulator's previous unit
                if (!(ok = mbar_wait(&sm.k_empty[buf], (use - 1) & 1, abort_flag))) break;
                tc_fence_after();
              }
              DCK_TC_TRACE(10);
              const uint32_t dcol = tmem + buf * kKCols;
              const bool last = u + kMma >= hi;  // this thread's last unit of the group
              for (int p = 0; p < np; ++p) {
                const int asl = (a_base + p) % kNA;
                const int wsl = w_cnt % NWt;
                if (((miss >> (8 + p)) & 1) && !(ok = mbar_wait(&sm.a_full[asl], ((a_base + p) / kNA) & 1, abort_flag)))
                  break;
                if (((miss >> p) & 1) && !(ok = mbar_wait(&wfull[wsl], (w_cnt / NWt) & 1, abort_flag))) break;
                DCK_TC_TRACE(13);
                const int w = gs.w[p];
                const uint32_t ab0 = smem_u32(sm.a[asl]);
                const uint32_t bb = smem_u32(sm.w[t * NWt + wsl]);
                const uint32_t swz = swz_of(w);
                for (int k = 0; k < w / 16; ++k) {
                  const uint64_t ad = sdesc(ab0 + k * 32, 16, 16 * w, swz);
                  const uint64_t bd = sdesc(bb + k * 2048, 128 * w, 1024, kSw128);
                  umma_f16(dcol, ad, bd, idesc_k, (p > 0 || k > 0) ? 1u : 0u);
                }
                umma_commit(&wempty[wsl]);
                if (last) umma_commit(&sm.a_empty[asl]);  // this thread is done with the piece
                DCK_TC_TRACE(14);
                ++w_cnt;
              }
              if (!ok) break;
              umma_commit(&sm.k_full[buf]);
              DCK_TC_TRACE(11);
              ++own;
            }
            a_cnt += np;
            kc += hi - lo;
          }
        }
      }
    }
    __syncwarp();
  } else if (warp >= 2 && warp <= 9) {
    // ---- epilogue: RoPE, scores, softmax, P -------------------------------
    const int e = tid - 64;              // 0 .. 255
    const int quad = warp & 3;           // TMEM lane quadrant
    const int hf = (warp - 2) >> 2;      // frequency half, then head half
    const int tau = quad * 32 + lane;    // token row inside the tile
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    // tile and segment ends: thread e owns head jt and the 16 tokens [16 ct, 16 ct + 16)
    // of every tile; the 8 owners of a head are adjacent lanes of one warp
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
    for (int ph = 0; ph < 2 && ok; ++ph)
    for (Walker walk = ph ? walk_x : walk_m; ok && walk.next(a, seg);) {
      if (!kFold) {
        // rotated queries of this sequence at position L-1, scaled to log2 units
        // (angle reduced mod 2 pi in fp64, sine and cosine in fp32)
        const double P = (double)(seg.L - 1);
        const float qscale = kLog2e * rsqrtf((float)kD);
        const __nv_bfloat16* qb = static_cast<const __nv_bfloat16*>(a.q) + (int64_t)seg.b * Hq * kD;
        for (int i = e; i < Hq * (kD / 2); i += kEpiThreads) {
          const int j = i / (kD / 2), pi = i % (kD / 2);
          const double ang = P * sm.om64[pi];
          float sn, cs;
          sincosf((float)(ang - 6.283185307179586 * rint(ang * 0.15915494309189535)), &sn, &cs);
          const float x1v = __bfloat162float(qb[j * kD + pi]), x2v = __bfloat162float(qb[j * kD + pi + kD / 2]);
          sm.qr[j * kD + pi] = __float2bfloat16_rn((x1v * cs - x2v * sn) * qscale);
          sm.qr[j * kD + pi + kD / 2] = __float2bfloat16_rn((x1v * sn + x2v * cs) * qscale);
        }
      }
      // RoPE angle of token t0+tau and pair p: (t0*w_p mod 2pi, fp64) + tau*w_p (fp32);
      // the offsets beta of later tiles are written at the previous tile's end
      if (e < kD / 2) {
        const double ang = (double)seg.t_begin * sm.om64[e];
        sm.beta[e] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
      }
      EPI_SYNC();
      if (!ok) break;
      // head jt's reference max (log2 units; the same in all 8 owners) and this
      // owner's share of its row sum, rescaled whenever the reference moves
      float m_run = -INFINITY, l_part = 0.f;
      int ua = 0, ub = 0;  // units of the current tile
      for (int i = 0; i < seg.ntiles && ok; ++i) {
        const int t0 = seg.t_begin + kTile * i;
        const int64_t x = seg.x0 + i;  // flattened tile index
        units_of(ph, (int)x, ua, ub);
        float cs[32], sn[32];
#pragma unroll
        for (int ip = 0; ip < 32; ++ip) {
          const int pi = 32 * hf + ip;
          float ph = fmaf((float)tau, sm.om32[pi], sm.beta[pi]);
          ph = fmaf(-kTwoPi, rintf(ph * kInvTwoPi), ph);
          __sincosf(ph, &sn[ip], &cs[ip]);
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
            DCK_TC_TRACE(20);
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
                DCK_TC_TRACE(43 + ps);
                if (ps == 1) {
                  tc_fence_before();
                  __syncwarp();
                  if (lane == 0) mbar_arrive(&sm.k_empty[buf]);
                }
#pragma unroll
                for (int i2 = 0; i2 < 16; ++i2)
                  pa[0][i2 & 3] = fmaf(cs[16 * ps + i2], y0[2 * i2], fmaf(sn[16 * ps + i2], y0[2 * i2 + 1], pa[0][i2 & 3]));
                if (nh == 2)
#pragma unroll
                  for (int i2 = 0; i2 < 16; ++i2)
                    pa[1][i2 & 3] =
                        fmaf(cs[16 * ps + i2], y1[2 * i2], fmaf(sn[16 * ps + i2], y1[2 * i2 + 1], pa[1][i2 & 3]));
              }
              float* xh = sm.x + hf * (kMaxHqTc * 128);  // this frequency half's scores
              xh[sm.order[gs.h0 + 2 * u] * 128 + tau] = (pa[0][0] + pa[0][1]) + (pa[0][2] + pa[0][3]);
              if (nh == 2) xh[sm.order[gs.h0 + 2 * u + 1] * 128 + tau] = (pa[1][0] + pa[1][1]) + (pa[1][2] + pa[1][3]);
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
                  if (last && ps == 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sm.k_empty[buf]);
                  }
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
                    const int jj = 2 * tig + (q & 1), t = quad * 32 + 16 * mt + gid + 8 * (q >> 1);
                    if (jj < qpg) xh[(j0 + jj) * 128 + t] = acc[mt][q];
                  }
              }
            }
            DCK_TC_TRACE(21);
            ++kc;
          }
        }
        if (!ok) break;
        // ---- tile end: reference max, P ------------------------------------
        DCK_TC_TRACE(22);
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
          const int nv = max(0, min(16, seg.t_end - (t0 + tb)));  // tokens inside the sequence
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
          if (own && ct == 0) ta.mglob[x * Hq + jt] = m_run;
          // probabilities (bf16, the absorption's operand) straight into this tile's
          // P image; the row sum uses the rounded values
          uint32_t pk[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const __nv_bfloat162 pv = __floats2bfloat162_rn(own ? exp2f(sc[2 * k] - m_run) : 0.f,
                                                            own ? exp2f(sc[2 * k + 1] - m_run) : 0.f);
            const float2 pf = __bfloat1622float2(pv);
            l_part += pf.x + pf.y;
            pk[k] = *reinterpret_cast<const uint32_t*>(&pv);
          }
          if (own || (jt >= Hq && jt < hq_pad && ua == 0)) {  // padded heads get zero rows
            // image: [token atom (64)][head row][64 tokens], 128B rows, 16-byte chunks swizzled by row % 8
            uint8_t* img = ta.pglob + x * (hq_pad * 256) + (tb >> 6) * (hq_pad * 128) + (jt >> 3) * 1024 +
                           (jt & 7) * 128;
            const int ch = (tb & 63) >> 3;
            *reinterpret_cast<uint4*>(img + ((ch ^ (jt & 7)) << 4)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            *reinterpret_cast<uint4*>(img + (((ch + 1) ^ (jt & 7)) << 4)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          }
        }
        if (e < kD / 2 && i + 1 < seg.ntiles) {  // RoPE phase offsets of the next tile
          const double ang = (double)(t0 + kTile) * sm.om64[e];
          sm.beta[e] = (float)(ang - 6.283185307179586 * floor(ang * 0.15915494309189535));
        }
        DCK_TC_TRACE(23);
        EPI_SYNC();  // x is clear and the next tile's phase offsets are in place
        if (!ok) break;
      }
      if (!ok) break;
      // ---- segment end: reference max and row sum -> partial slot c + b -------
      l_part += __shfl_xor_sync(0xffffffffu, l_part, 1);
      l_part += __shfl_xor_sync(0xffffffffu, l_part, 2);
      l_part += __shfl_xor_sync(0xffffffffu, l_part, 4);
      if (jt < Hq && ct == 0 && sm.hunit[jt] >= ua && sm.hunit[jt] < ub) {
        const int64_t slot = ph ? xbase + (seg.x0 - sp.NTm) : (int64_t)blockIdx.x + seg.b;
        a.part_ml[(slot * Hq + jt) * 2] = m_run;
        a.part_ml[(slot * Hq + jt) * 2 + 1] = l_part;
      }
    }
#undef EPI_SYNC
  }
  tc_fence_before();
  __syncthreads();
  DCK_TC_TRACE_FLUSH();
  if (sm.abort_flag) {
    // let copies and MMAs already in flight land before the memory is released
    const long long c0 = clock64();
    while (clock64() - c0 < 4000000ll) {
    }
    if (tid == 0) atomicOr(a.err, kErrTimeout);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
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

struct PrepArgs {
  int n_items;
  int64_t seq_bytes;
  double om[kD / 2];  // RoPE frequencies, fp64
  PrepItem item[kMaxItems];
};

// One block writes one factor item: [nh heads][2 halves][ws rank rows]
// [64 columns] bf16, 128B-swizzled (16-byte chunk c of row r stored at chunk
// c ^ (r % 8); every half starts on a 1024-byte swizzle atom).
// Key mode: columns of B_g[:, slot].  Query-folded mode (one block row per
// sequence b): columns 2i and 2i+1 are
//   a_i B[:, i] + b_i B[:, i+64]  and  b_i B[:, i] - a_i B[:, i+64]
// with (a, b) the halves of RoPE(q_{b,h}, L_b - 1) * log2(e)/sqrt(d).
template <bool kFold>
__global__ void __launch_bounds__(256) factor_prep_kernel(const LayerTable lt, const DecodeArgs a, const PrepArgs pa,
                                                          uint8_t* __restrict__ img) {
  griddep_launch();
  const int n = blockIdx.x, b = blockIdx.y;
  const PrepItem it = pa.item[n];
  const int g = it.g, ws = it.ws, nh = it.nh;
  __shared__ float qa[2][kD / 2], qb[2][kD / 2];
  if (kFold) {
    const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
    if (L == 0) return;  // no tile of this sequence is ever processed
    if (threadIdx.x < nh * (kD / 2)) {
      const int hh = threadIdx.x / (kD / 2), i = threadIdx.x % (kD / 2);
      const int kv = it.kv[hh];
      // angle (L-1) w_i reduced mod 2 pi in fp64, sine and cosine in fp32
      const double ang = (double)(L - 1) * pa.om[i];
      float sn, cs;
      sincosf((float)(ang - 6.283185307179586 * rint(ang * 0.15915494309189535)), &sn, &cs);
      const __nv_bfloat16* q = static_cast<const __nv_bfloat16*>(a.q) + ((int64_t)b * lt.Hq + kv) * kD;
      const float x1 = __bfloat162float(q[i]), x2 = __bfloat162float(q[i + kD / 2]);
      const float sc = kLog2e * rsqrtf((float)kD);
      qa[hh][i] = (x1 * cs - x2 * sn) * sc;
      qb[hh][i] = (x1 * sn + x2 * cs) * sc;
    }
    __syncthreads();
  }
  const int64_t ld = (int64_t)lt.grp_nh[g] * kD;
  uint8_t* dst = img + (kFold ? (int64_t)b * pa.seq_bytes : 0) + it.off;
  // thread -> (head, row, 8-column chunk): nh x ws rows x 16 chunks (2 halves x 8)
  for (int idx = threadIdx.x; idx < nh * ws * 16; idx += blockDim.x) {
    const int hh = idx / (ws * 16), r = (idx >> 4) % ws, ch = idx & 15;
    const int half = ch >> 3, c8 = ch & 7;
    const __nv_bfloat16* __restrict__ Bs =
        static_cast<const __nv_bfloat16*>(a.Bk) + lt.grp_boff[g] + (it.s0 + hh) * kD;
    const int k = it.k0 + r;
    float v[8];
    if (kFold) {
      // output columns col = 64*half + 8*c8 + t, t even/odd -> pair i = col/2
#pragma unroll
      for (int t = 0; t < 8; t += 2) {
        const int i = (64 * half + 8 * c8 + t) >> 1;
        const float x = __bfloat162float(Bs[k * ld + i]);
        const float y = __bfloat162float(Bs[k * ld + kD / 2 + i]);
        v[t] = fmaf(qa[hh][i], x, qb[hh][i] * y);
        v[t + 1] = fmaf(qb[hh][i], x, -qa[hh][i] * y);
      }
    } else {
      const uint4 raw = *reinterpret_cast<const uint4*>(Bs + k * ld + 64 * half + 8 * c8);
      const __nv_bfloat16* h8 = reinterpret_cast<const __nv_bfloat16*>(&raw);
#pragma unroll
      for (int t = 0; t < 8; ++t) v[t] = __bfloat162float(h8[t]);
    }
    uint4 out;
    __nv_bfloat162* o2 = reinterpret_cast<__nv_bfloat162*>(&out);
#pragma unroll
    for (int t = 0; t < 4; ++t) o2[t] = __floats2bfloat162_rn(v[2 * t], v[2 * t + 1]);
    *reinterpret_cast<uint4*>(dst + (hh * 2 + half) * (ws * 128) + r * 128 + ((c8 ^ (r & 7)) << 4)) = out;
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
  bool operator==(const MapsKey& o) const { return kc == o.kc && n_rows == o.n_rows && Rk == o.Rk; }
};
constexpr int kMapsCache = 64;
std::mutex g_maps_mu;
MapsKey g_maps_key[kMapsCache];
Maps g_maps_val[kMapsCache];
int g_maps_n = 0, g_maps_next = 0;

bool build_maps(const LayerTable& lt, const DecodeArgs& a, Maps& maps) {
  std::memset(&maps, 0, sizeof(maps));
  const uint64_t rows = (uint64_t)std::max<int64_t>(1, a.n_rows);
  return make_tmap_2d_bf16(&maps.kc64, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 64, kTile, CU_TENSOR_MAP_SWIZZLE_128B) &&
         make_tmap_2d_bf16(&maps.kc32, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 32, kTile, CU_TENSOR_MAP_SWIZZLE_64B) &&
         make_tmap_2d_bf16(&maps.kc16, a.kc, lt.Rk, rows, (uint64_t)lt.Rk * 2, 16, kTile, CU_TENSOR_MAP_SWIZZLE_32B);
}

static_assert(sizeof(Smem<true>) + 1024 <= 232448, "shared memory of the query-folded kernel");
static_assert(sizeof(Smem<false>) + 1024 <= 232448, "shared memory of the key-mode kernel");

template <bool kFold>
cudaError_t launch_mode(const LayerTable& lt, const DecodeArgs& a, const Maps& maps, const TcArgs& ta,
                        const PrepArgs& pa, cudaStream_t s) {
  const size_t smem = sizeof(Smem<kFold>) + 1024;
  static int attr_done[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  const bool dev_ok = dev >= 0 && dev < 64;
  if (!dev_ok || !attr_done[dev]) {
    cudaError_t e = cudaFuncSetAttribute(decode_tc_kernel<kFold>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    if (dev_ok) attr_done[dev] = 1;
  }
  factor_prep_kernel<kFold><<<dim3(pa.n_items, kFold ? a.B : 1), 256, 0, s>>>(lt, a, pa,
                                                                                static_cast<uint8_t*>(a.extra));
  cudaError_t e = hook_launched(a.hook, s);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_items);
  cfg.blockDim = dim3(Ring<kFold>::kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decode_tc_kernel<kFold>, maps, lt, a, ta);
  return e != cudaSuccess ? e : hook_launched(a.hook, s);
}

// Units, items and per-group tables of a layer.  Returns false when the layer
// does not fit the tables.
bool build_tables(const LayerTable& lt, TcArgs& ta, PrepArgs& pa) {
  std::memset(&ta, 0, sizeof(ta));
  std::memset(&pa, 0, sizeof(pa));
  ta.hq_pad = hq_pad_of(lt.Hq);
  int pos = 0, item = 0, off = 0, unit = 0;
  for (int g = 0; g < lt.G; ++g) {
    GroupSm& gs = ta.grp[g];
    gs.roff = lt.grp_roff[g];
    int16_t kk[kMaxPieces];
    gs.np = (int8_t)make_pieces(lt.grp_rank[g], gs.w, kk);
    if (gs.np > kMaxPieces || gs.np > kNA) return false;
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

cudaError_t launch_decode_tc(const LayerTable& lt, const DecodeArgs& a, cudaStream_t s) {
  const bool fold = lt.qpg == 1;
  if (!a.extra) return cudaErrorInvalidValue;
  static thread_local TcArgs ta;
  static thread_local PrepArgs pa;
  if (!build_tables(lt, ta, pa)) return cudaErrorInvalidValue;
  rope_freqs(a.theta, ta.om);
  std::memcpy(pa.om, ta.om, sizeof(ta.om));
  const ExtraLayout xl = extra_layout(lt, a.B, a.n_rows);
  uint8_t* base = static_cast<uint8_t*>(a.extra);
  ta.fimg = base;
  ta.pglob = base + xl.img;
  ta.mglob = reinterpret_cast<float*>(base + xl.img + xl.p);
  ta.max_tiles = max_tiles(a.n_rows, a.B);
  const MapsKey key{a.kc, a.n_rows, lt.Rk};
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
    if (!build_maps(lt, a, maps)) return cudaErrorInvalidValue;
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
  e = launch_absorb_tc(lt, a, r, s);
  return e != cudaSuccess ? e : hook_launched(a.hook, s);
}

}  // namespace dck
