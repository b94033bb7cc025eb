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

__device__ __forceinline__ int ntiles_of(const DecodeArgs& a, int b) {
  const int L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
  return (L + kTile - 1) / kTile;
}

struct Segment {
  int b, L, t_begin, t_end, ntiles;
  int x0;        // flattened index of the segment's first tile
  int64_t row0;  // first cache row of the sequence
};

// Walks the sequences overlapping flattened tiles [x, x1) in order; with
// `single`, every tile is a segment of its own.
struct Walker {
  int b, pre, x, x1;
  bool single;
  __device__ bool next(const DecodeArgs& a, Segment& sg) {
    while (x < x1 && b < a.B) {
      const int nt = ntiles_of(a, b);
      if (x >= pre + nt) {
        pre += nt;
        ++b;
        continue;
      }
      const int xe = single ? x + 1 : min(x1, pre + nt);
      sg.b = b;
      sg.L = valid_len(a.seq_len, a.seq_start, b, a.n_rows);
      sg.row0 = a.seq_start[b];
      sg.t_begin = (x - pre) * kTile;
      sg.t_end = min(sg.L, (xe - pre) * kTile);
      sg.ntiles = xe - x;
      sg.x0 = x;
      x = xe;
      return true;
    }
    return false;
  }
};

// Block-wide tile count over the batch (every thread of the block calls it;
// `scan` is shared scratch of blockDim.x ints and keeps each thread's
// inclusive prefix for tile_find).  Block 0 of the grid reports sequences
// whose rows fall outside the cache.
__device__ __forceinline__ int tile_count(const DecodeArgs& a, int* scan) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int per = (a.B + nthr - 1) / nthr;
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
  for (int off = 1; off < nthr; off <<= 1) {
    const int v = tid >= off ? scan[tid - off] : 0;
    __syncthreads();
    scan[tid] += v;
    __syncthreads();
  }
  return scan[nthr - 1];
}

// Block-wide lookup (after tile_count, same scan): the sequence owning
// flattened tile x and its first tile; (B, NT) when no sequence does.
__device__ __forceinline__ void tile_find(const DecodeArgs& a, const int* scan, int x, int& b_out, int& pre_out) {
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int per = (a.B + nthr - 1) / nthr;
  const int b0 = tid * per;
  __shared__ int s_bf, s_pf;
  if (tid == 0) {
    s_bf = a.B;
    s_pf = scan[nthr - 1];
  }
  __syncthreads();
  int run = tid ? scan[tid - 1] : 0;
  for (int b = b0; b < b0 + per && b < a.B; ++b) {
    const int nt = ntiles_of(a, b);
    if (nt > 0 && x >= run && x < run + nt) {
      s_bf = b;
      s_pf = run;
    }
    run += nt;
  }
  __syncthreads();
  b_out = s_bf;
  pre_out = s_pf;
  __syncthreads();
}

// Work split of the tensor-core kernels.  With n CTAs and NT tiles, fewer than
// kFineSplitBelow per CTA, every CTA takes floor(NT / n) whole tiles (the main
// tiles [0, NTm), in contiguous ranges) and the R = NT - NTm extra tiles are
// shared out more finely, so that no CTA carries a whole tile more than
// another (with more tiles per CTA, that imbalance is small and NTm = NT): the scores kernel splits them
// into their units (CTA c: units [c XU / n, (c+1) XU / n) of the flattened
// (extra tile, unit) list, XU = R U), the absorption kernel hands out whole
// extra tiles.  Every extra tile is a segment of its own (its own partial slot
// extra_base + e, e = x - NTm), so its heads' softmax state never spans CTAs.
struct Split {
  int NT, NTm, R;
  __device__ Split(int nt, int n, bool extra) : NT(nt), NTm(main_tiles(nt, n, extra)), R(NT - NTm) {}
  __device__ int main_begin(int c, int n) const { return item_begin(c, NTm, n); }
};

// First partial slot of the extra tiles: after the main slots c + b.
__host__ __device__ inline int64_t extra_slot_base(int n_items, int batch) { return (int64_t)n_items + batch - 1; }

// Most 128-token tiles a call can have with non-overlapping sequences: the
// per-tile probability and reference-max stores of the tensor-core path are
// sized for this many.
__host__ __device__ inline int64_t max_tiles(int64_t n_rows, int batch) { return (n_rows + kTile - 1) / kTile + batch; }

}  // namespace tc
}  // namespace dck
