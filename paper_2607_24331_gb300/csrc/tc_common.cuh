// Pieces shared by the tensor-core decode kernels (scores and absorption):
// bulk copies, bounded waits usable by one thread or a whole warp, ring-slot
// claims, the tile walk over sequence segments and the block-wide tile scan.
#pragma once

#include "common.cuh"
#include "sm100.cuh"

namespace dck {
namespace tc {

using namespace sm100;

__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Global -> shared bulk copy completing on `bar` (16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}

// Shared -> global bulk copy tracked by the issuing thread's bulk groups.
__device__ __forceinline__ void bulk_store(void* dst, const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_u32(src)), "r"(bytes)
               : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// The issuing thread's bulk stores have finished reading shared memory.
__device__ __forceinline__ void bulk_store_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and their writes are complete.
__device__ __forceinline__ void bulk_store_wait() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Moves [src, src + bytes) toward L2 ahead of its TMA loads (16-byte multiples).
__device__ __forceinline__ void prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// Bounded wait whose outcome is the same in every lane of the warp.
__device__ __forceinline__ bool wwait(uint64_t* bar, uint32_t parity, volatile int* abort_flag) {
  const bool r = mbar_wait(bar, parity, abort_flag);
  return __all_sync(0xffffffffu, r);
}

// Lane 0 waits for the `n` ring slots starting at ring position `cnt` (depth
// `depth`) to be released; the result is shared with the warp.
__device__ __forceinline__ bool wait_slots(uint64_t* empty, int depth, int cnt, int n, int lane,
                                           volatile int* abort_flag) {
  bool ok = true;
  if (lane == 0)
    for (int i = 0; i < n && ok; ++i) {
      const int c = cnt + i;
      if (c >= depth) ok = mbar_wait(&empty[c % depth], ((c / depth) - 1) & 1, abort_flag);
    }
  return __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
}

// Lane 0 waits for ring position `cnt` to be free, then counts how many of the
// following positions (up to `max_n` in all, at most one ring turn) are free
// already, without waiting.  Returns that count to the whole warp, 0 if the
// wait gave up.  (A position within one turn is at most one use ahead of its
// release, so the parity test cannot see a stale phase.)
__device__ __forceinline__ int claim_slots(uint64_t* empty, int depth, int cnt, int max_n, int lane,
                                           volatile int* abort_flag) {
  int n = 0;
  if (lane == 0 && (cnt < depth || mbar_wait(&empty[cnt % depth], ((cnt / depth) - 1) & 1, abort_flag))) {
    n = 1;
    while (n < max_n && n < depth) {
      const int c = cnt + n;
      if (c >= depth && !mbar_test(&empty[c % depth], ((c / depth) - 1) & 1)) break;
      ++n;
    }
  }
  return __shfl_sync(0xffffffffu, n, 0);
}

// A ring of `depth` shared-memory slots handed out in FIFO order to
// instances of variable size (a key group's latent pieces, a unit's factor
// items), each instance with one full and one empty mbarrier (index
// instance % kFifoBars; phase (instance / kFifoBars) & 1).  One warp fills the
// ring; its lanes all keep the same state.  Since every instance holds at
// least one slot and depth <= kFifoBars, an instance is allocated only after
// the one kFifoBars before it (same barriers) has been released, so no
// barrier phase can be confused with another.
constexpr int kFifoBars = 8;
struct SlotFifo {
  int head = 0;       // slots handed out so far (the next instance starts at head % depth)
  int used = 0;       // slots held by instances not yet released
  int tail = 0;       // oldest instance not yet released
  int inst = 0;       // instances handed out so far
  uint32_t hist = 0;  // slot counts of the last kFifoBars instances, 4 bits each
  // Waits (lane 0) for the oldest instances' empty barriers until n slots are
  // free, then records the next instance; false (in every lane) if a wait gave up.
  __device__ bool claim(int n, int depth, uint64_t* empty, int lane, volatile int* abort_flag) {
    while (depth - used < n) {
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&empty[tail % kFifoBars], (tail / kFifoBars) & 1, abort_flag);
      if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) return false;
      used -= (hist >> (4 * (tail % kFifoBars))) & 0xFu;
      ++tail;
    }
    const int sh = 4 * (inst % kFifoBars);
    hist = (hist & ~(0xFu << sh)) | ((uint32_t)n << sh);
    used += n;
    return true;
  }
  __device__ void advance(int n) {
    head += n;
    ++inst;
  }
};

// ---------------------------------------------------------------------------
// Work plan of the tensor-core decode path.
//
// The scores kernel runs as P CTA pairs (clusters of two CTAs, one tcgen05
// pair MMA of M = 256 tokens): every sequence is cut into pair tiles of 256
// tokens, whose first 128 tokens belong to the pair's even CTA (half 0) and
// the rest to its odd CTA (half 1).  The flattened pair-tile list (sequences in
// order) is split over the pairs: pair p takes the contiguous range
// [floor(p NPm / P), floor((p+1) NPm / P)) of the first NPm tiles; with fewer
// than kFineSplitBelow tiles per pair the R = NP - NPm left over are shared
// out by units (groups of heads) instead, pair p taking units
// [floor(p R U / P), floor((p+1) R U / P)) of the flattened (extra tile, unit)
// list.  The absorption kernel's CTA c = 2p + h follows half h of pair p's
// tiles (its extra tiles it splits by r_v chunks instead).
//
// Softmax segments and their partial slots: half h of pair p over sequence b's
// tiles in p's main range writes slot 2 (p + b) + h; half h of extra tile e is
// a segment of its own, slot 2 (P + B - 1) + 2 e + h.  A slot is live when its
// half has at least one token (the odd half of a sequence's last pair tile can
// be empty); only live slots are read.
// ---------------------------------------------------------------------------

constexpr int kPTile = 256;  // tokens of a pair tile

__device__ __forceinline__ int n128_of(const DecodeArgs& a, int b) {
  return (valid_len(a.seq_len, a.seq_start, b, a.n_rows) + kTile - 1) / kTile;
}
__device__ __forceinline__ int n256_of(const DecodeArgs& a, int b) {
  return (valid_len(a.seq_len, a.seq_start, b, a.n_rows) + kPTile - 1) / kPTile;
}

__host__ __device__ inline int64_t pair_slot(int p, int b, int h) { return 2 * ((int64_t)p + b) + h; }
__host__ __device__ inline int64_t pair_xslot(int P, int B, int e, int h) {
  return 2 * ((int64_t)P + B - 1) + 2 * (int64_t)e + h;
}
// Partial slots of a call over caches of n_rows rows: main slots, then the
// extra tiles (fewer than P, and no more than the call's pair tiles,
// ceil(n_rows / 256) + B with non-overlapping sequences).
__host__ __device__ inline int64_t pair_slot_count(int P, int B, int64_t n_rows) {
  const int64_t tiles = (n_rows + kPTile - 1) / kPTile + B;
  const int64_t extra = P > 1 ? (P - 1 < tiles ? P - 1 : tiles) : 0;
  return 2 * ((int64_t)P + (B > 0 ? B - 1 : 0)) + 2 * extra;
}

// Split of NP pair tiles over P pairs (see above).
struct PSplit {
  int NP, NPm, R;
  __host__ __device__ PSplit(int np, int P) : NP(np), NPm(np / P < kFineSplitBelow ? np / P * P : np), R(np - NPm) {}
  __host__ __device__ int main_begin(int p, int P) const { return item_begin(p, NPm, P); }
};

// A run of consecutive pair tiles of one sequence.
struct PSegment {
  int b, L;
  int i0;        // local index (within the sequence) of the run's first pair tile
  int ntiles;    // pair tiles in the run
  int X0;        // flattened index of the run's first pair tile
  int pre128;    // flattened index of the sequence's first 128-token tile
  int n128;      // 128-token tiles of the sequence
  int64_t row0;  // first cache row of the sequence
  // 128-token tile of local pair tile i0 + i, half h, and whether it exists
  __device__ int x128(int i, int h) const { return pre128 + 2 * (i0 + i) + h; }
  __device__ bool has(int i, int h) const { return 2 * (i0 + i) + h < n128; }
  __device__ int t0(int i, int h) const { return kPTile * (i0 + i) + kTile * h; }  // first token position
};

// Walks the sequences overlapping flattened pair tiles [X, X1) in order; with
// `single`, every pair tile is a run of its own.
struct PairWalker {
  int b, pre256, pre128, X, X1;
  bool single;
  __device__ bool next(const DecodeArgs& a, PSegment& sg) {
    while (X < X1 && b < a.B) {
      const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
      const int nt = (L + kPTile - 1) / kPTile;
      if (X >= pre256 + nt) {
        pre256 += nt;
        pre128 += (L + kTile - 1) / kTile;
        ++b;
        continue;
      }
      const int Xe = single ? X + 1 : min(X1, pre256 + nt);
      sg.b = b;
      sg.L = L;
      sg.i0 = X - pre256;
      sg.ntiles = Xe - X;
      sg.X0 = X;
      sg.pre128 = pre128;
      sg.n128 = (L + kTile - 1) / kTile;
      sg.row0 = a.seq_start[b];
      X = Xe;
      return true;
    }
    return false;
  }
};

// Block-wide count of pair tiles over the batch (every thread of the block
// calls it; s256 and s128 are shared scratch of blockDim.x ints each and keep
// every thread's inclusive prefixes of pair tiles and of 128-token tiles for
// pair_tile_find).  Block 0 of the grid reports sequences whose rows fall
// outside the cache.  Returns NP.
__device__ __forceinline__ int pair_tile_count(const DecodeArgs& a, int* s256, int* s128) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int per = (a.B + nthr - 1) / nthr;
  const int b0 = tid * per;
  int l256 = 0, l128 = 0;
  for (int b = b0; b < b0 + per && b < a.B; ++b) {
    l256 += n256_of(a, b);
    l128 += n128_of(a, b);
    if (blockIdx.x == 0) {
      const int64_t L = a.seq_len[b], st = a.seq_start[b];
      if (L < 0 || st < 0 || st + L > a.n_rows) atomicOr(a.err, kErrBadSeq);
    }
  }
  s256[tid] = l256;
  s128[tid] = l128;
  __syncthreads();
  for (int off = 1; off < nthr; off <<= 1) {
    const int v = tid >= off ? s256[tid - off] : 0;
    const int w = tid >= off ? s128[tid - off] : 0;
    __syncthreads();
    s256[tid] += v;
    s128[tid] += w;
    __syncthreads();
  }
  return s256[nthr - 1];
}

// Block-wide lookup (after pair_tile_count, same scratch): a walker positioned
// at flattened pair tile X over [X, X1).
__device__ __forceinline__ PairWalker pair_walker_at(const DecodeArgs& a, const int* s256, const int* s128, int X,
                                                     int X1, bool single) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int per = (a.B + nthr - 1) / nthr;
  const int b0 = tid * per;
  __shared__ int s_b, s_p256, s_p128;
  if (tid == 0) {
    s_b = a.B;
    s_p256 = s256[nthr - 1];
    s_p128 = s128[nthr - 1];
  }
  __syncthreads();
  int r256 = tid ? s256[tid - 1] : 0, r128 = tid ? s128[tid - 1] : 0;
  if (per == 1) {  // this thread's sequence (if any): its tile counts are the prefix steps
    const int nt = s256[tid] - r256;
    if (b0 < a.B && nt > 0 && X >= r256 && X < r256 + nt) {
      s_b = b0;
      s_p256 = r256;
      s_p128 = r128;
    }
  } else {
    for (int b = b0; b < b0 + per && b < a.B; ++b) {
      const int nt = n256_of(a, b);
      if (nt > 0 && X >= r256 && X < r256 + nt) {
        s_b = b;
        s_p256 = r256;
        s_p128 = r128;
      }
      r256 += nt;
      r128 += n128_of(a, b);
    }
  }
  __syncthreads();
  PairWalker w{s_b, s_p256, s_p128, X, X1, single};
  __syncthreads();
  return w;
}

// Most 128-token tiles a call can have with non-overlapping sequences: the
// per-tile probability and reference-max stores of the tensor-core path are
// sized for this many.
__host__ __device__ inline int64_t max_tiles(int64_t n_rows, int batch) { return (n_rows + kTile - 1) / kTile + batch; }

}  // namespace tc
}  // namespace dck
