// Internal declarations shared by the libdck translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/dck.h"

namespace dck {

constexpr int kMaxKvHeads = 128;
constexpr int kMaxGroups = 128;
constexpr int kMaxQPerKv = 8;     // query heads per KV head handled by the kernels
constexpr int kMaxRankV = 2048;
constexpr int kMaxBatch = 4096;
constexpr int kMaxPrefillLen = 1 << 24;  // bound on a prefill call's q_max and max_seq_len
constexpr int kTile = 128;        // tokens per work tile (one UMMA M block)

// Device error word values (bit flags).
constexpr int kErrBadSeq = 1;     // a sequence's rows fall outside the cache
constexpr int kErrBadRow = 2;     // an append destination row is outside the cache
constexpr int kErrTimeout = 4;    // a bounded wait gave up

// Group table and shapes of one layer, passed by value to the kernels.
struct LayerTable {
  int32_t Hq, Hkv, d, G, Rk, rv, qpg;
  int32_t head_group[kMaxKvHeads];  // KV head -> group
  int32_t head_slot[kMaxKvHeads];   // KV head -> column-block slot in its group
  int32_t grp_rank[kMaxGroups];     // r_g
  int32_t grp_roff[kMaxGroups];     // first key-cache column of group g
  int32_t grp_nh[kMaxGroups];       // n_g
  int64_t grp_boff[kMaxGroups];     // element offset of B_g in the packed B_k
};

// Work decomposition of a decode call: every sequence is cut into 128-token
// tiles; the flattened tile list is split into n_items contiguous ranges
// (item c: tiles [floor(c*NT/n), floor((c+1)*NT/n))).  Item c writes one
// partial per sequence b it touches, in slot c + b.
struct DecodeArgs {
  const void* q;
  const void* kc;
  const void* vc;
  const void* Bk;
  const void* Bv;
  const int64_t* seq_start;
  const int32_t* seq_len;
  int64_t n_rows;
  int32_t B;
  int32_t n_items;
  int32_t split_extra;  // tensor-core path: the pair-tile plan of tc_common.cuh (n_items = 2 x CTA pairs)
  float theta;
  float* part_u;   // [n_slots, Hq, rv]
  float* part_ml;  // [n_slots, Hq, 2]  (running max in log2 units, sum)
  void* out;       // [B, Hq, d]
  int* err;
  struct LaunchHook* hook;  // host-side launch count and optional timing events (never read by kernels)
  void* extra;     // workspace region of the tensor-core path (per-sequence folded factors)
};

// Host-side record of the kernels one entry-point call puts on its stream.
// When `n_ev` > 0, ev[0] (a cudaEvent_t) is recorded before the call's first
// kernel, ev[k] after its k-th kernel for k < n_ev - 1 and ev[n_ev - 1] after
// its last kernel, so that a caller can time the whole call (n_ev = 2, nothing
// recorded between the kernels) or every kernel of it (n_ev = kernels + 1).
struct LaunchHook {
  void* const* ev = nullptr;
  int n_ev = 0;
  int count = 0;
};
inline cudaError_t hook_begin(LaunchHook* h, cudaStream_t s);     // before the first kernel
inline cudaError_t hook_launched(LaunchHook* h, cudaStream_t s);  // after each kernel launch
inline cudaError_t hook_end(LaunchHook* h, cudaStream_t s);       // after the call's last kernel

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Host launchers (each defined in its own translation unit).
cudaError_t launch_decode_simt(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s);
cudaError_t launch_combine(const LayerTable& lt, const DecodeArgs& a, int dtype, cudaStream_t s);
cudaError_t launch_append_simt(const void* x, int n_tok, int D, const void* A_k, const void* A_v, int Rk,
                               int rv, const int64_t* rows, void* kc, void* vc, int64_t n_rows, int dtype,
                               int* err, cudaStream_t s);
cudaError_t launch_synth_gaussian(void* dst, int64_t n, uint64_t key, int64_t start, float scale, int dtype,
                                  cudaStream_t s);
// Host-side argument checks shared by the decode entry points (no CUDA call).
dck_status decode_precheck(const dck_layer_desc* desc, const void* q, const void* kcache, const void* vcache,
                           int64_t n_rows, const void* B_k, const void* B_v, const int64_t* d_seq_start,
                           const int32_t* d_seq_len, int32_t batch, float rope_theta, const void* out);

// ---------------------------------------------------------------------------
// device helpers
// ---------------------------------------------------------------------------

template <typename T>
__device__ __forceinline__ float to_f32(T v);
template <>
__device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// Number of `tile`-token tiles of every sequence, as an exclusive prefix in
// shared memory prefix[0..B].  Sequences whose rows fall outside the cache
// count as empty and raise kErrBadSeq.  Must be called by the whole block.
// Returns the total tile count NT.
__device__ __forceinline__ int build_tile_prefix(const int32_t* __restrict__ seq_len,
                                                 const int64_t* __restrict__ seq_start, int B,
                                                 int64_t n_rows, int* prefix, int* scratch, int* err,
                                                 bool report, int tile = kTile) {
  const int nt = blockDim.x;
  const int per = (B + nt - 1) / nt;
  const int b0 = threadIdx.x * per;
  int local = 0;
  for (int b = b0; b < b0 + per && b < B; ++b) {
    int64_t L = seq_len[b];
    int64_t st = seq_start[b];
    if (L < 0 || st < 0 || st + L > n_rows) {
      if (report) atomicOr(err, kErrBadSeq);
      L = 0;
    }
    local += (int)((L + tile - 1) / tile);
  }
  scratch[threadIdx.x] = local;
  __syncthreads();
  // Hillis-Steele inclusive scan over the per-thread sums
  for (int off = 1; off < nt; off <<= 1) {
    int v = threadIdx.x >= off ? scratch[threadIdx.x - off] : 0;
    __syncthreads();
    scratch[threadIdx.x] += v;
    __syncthreads();
  }
  int run = threadIdx.x ? scratch[threadIdx.x - 1] : 0;
  for (int b = b0; b < b0 + per && b < B; ++b) {
    prefix[b] = run;
    int64_t L = seq_len[b];
    int64_t st = seq_start[b];
    if (L < 0 || st < 0 || st + L > n_rows) L = 0;
    run += (int)((L + tile - 1) / tile);
  }
  int total = scratch[nt - 1];
  if (threadIdx.x == 0) prefix[B] = total;
  __syncthreads();
  return total;
}

// Length of sequence b as used by the kernels (0 when its rows are invalid).
__device__ __forceinline__ int valid_len(const int32_t* seq_len, const int64_t* seq_start, int b,
                                         int64_t n_rows) {
  int64_t L = seq_len[b];
  int64_t st = seq_start[b];
  if (L < 0 || st < 0 || st + L > n_rows) return 0;
  return (int)L;
}

__host__ __device__ __forceinline__ int item_begin(int c, int NT, int n_items) {
  return (int)(((int64_t)c * NT) / n_items);
}

// Programmatic dependent launch: a kernel launched with launch_pdl may start
// while the previous kernel on the stream finishes; pdl_wait() returns once
// that kernel is complete and its memory visible (a no-op without PDL), and
// pdl_launch_dependents() lets the next kernel launch early in turn.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Tiles [0, main_tiles) are split in contiguous whole-tile ranges over the
// n_items work items; with `split_extra` (tensor-core path) and fewer than
// kFineSplitBelow tiles per item, only n_items * floor(NT / n_items) of them,
// the rest ("extra tiles") being shared out more finely (see tc_common.cuh).
constexpr int kFineSplitBelow = 8;
__host__ __device__ __forceinline__ int main_tiles(int NT, int n_items, bool split_extra) {
  return split_extra && NT / n_items < kFineSplitBelow ? NT / n_items * n_items : NT;
}

// The item whose tile range contains tile x (0 <= x < NT).
__device__ __forceinline__ int item_of_tile(int x, int NT, int n_items) {
  return (int)((((int64_t)(x + 1) * n_items) + NT - 1) / NT) - 1;
}

// Sequence owning flattened tile x: largest b with prefix[b] <= x and a
// non-empty tile range.
__device__ __forceinline__ int seq_of_tile(const int* prefix, int B, int x) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (prefix[mid] <= x) lo = mid; else hi = mid - 1;
  }
  return lo;
}

}  // namespace dck

namespace dck {
// Records a caller's timing event on `s`; inside stream capture it becomes an
// external event node, so that it can be timed after each graph replay.
inline cudaError_t record_timing_event(void* ev, cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &st) != cudaSuccess) return cudaErrorUnknown;
  if (st == cudaStreamCaptureStatusActive)
    return cudaEventRecordWithFlags(static_cast<cudaEvent_t>(ev), s, cudaEventRecordExternal);
  return cudaEventRecord(static_cast<cudaEvent_t>(ev), s);
}

inline cudaError_t hook_begin(LaunchHook* h, cudaStream_t s) {
  if (!h || h->n_ev <= 0) return cudaSuccess;
  return record_timing_event(h->ev[0], s);
}

// Events between kernels stop programmatic dependent launch from starting the
// next kernel early, so only the brackets a caller asked for are recorded:
// ev[k] after the k-th kernel for k < n_ev - 1, and ev[n_ev - 1] once, after
// the call's last kernel (hook_end).
inline cudaError_t hook_launched(LaunchHook* h, cudaStream_t s) {
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || !h) return e;
  ++h->count;
  if (h->count >= h->n_ev - 1) return cudaSuccess;
  return record_timing_event(h->ev[h->count], s);
}

inline cudaError_t hook_end(LaunchHook* h, cudaStream_t s) {
  if (!h || h->n_ev <= 0) return cudaSuccess;
  return record_timing_event(h->ev[h->n_ev - 1], s);
}
}  // namespace dck
