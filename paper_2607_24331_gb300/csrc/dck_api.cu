// C ABI of libdck: argument validation, work planning and kernel dispatch.
// The formulas and conventions are documented in include/dck.h.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "common.cuh"
#include "tc_common.cuh"
#include "tc_host.h"

namespace dck {
bool simt_supports(const LayerTable& lt);
bool combine_supports(const LayerTable& lt);
bool tc_decode_supports(const LayerTable& lt, int dtype);
size_t tc_decode_extra_ws(const LayerTable& lt, int batch, int64_t n_rows);
int tc_decode_pairs(const LayerTable& lt);
cudaError_t launch_decode_tc(const LayerTable& lt, const DecodeArgs& a, const TcStepAppend* app, cudaStream_t s);
bool tc_step_append_supports(const LayerTable& lt, int D, int batch);
bool tc_append_supports(int D, int Rk, int rv, int dtype);
size_t tc_append_workspace(int n_tok, int Rk, int rv);
bool tc_prefill_supports(const LayerTable& lt, int dtype);
size_t tc_prefill_workspace(const LayerTable& lt, int64_t n_rows);
cudaError_t launch_prefill_tc(const LayerTable& lt, const void* q, const int32_t* q_len, int qmax, const void* kc,
                              const void* vc, int64_t n_rows, const void* Bk, const void* Bv,
                              const int64_t* seq_start, const int32_t* seq_len, int B, int max_len, float theta,
                              void* out, void* ws, int* err, LaunchHook* hook, cudaStream_t s);
cudaError_t launch_bounded_wait_selftest(long long limit_cycles, int* err, cudaStream_t s);
cudaError_t launch_append_tc(const void* x, int n_tok, int D, const void* A_k, const void* A_v, int Rk, int rv,
                             const int64_t* rows, void* kc, void* vc, int64_t n_rows, void* ws, size_t ws_bytes,
                             int* err, cudaStream_t s, int* n_launches);
}  // namespace dck

using namespace dck;

namespace {

// Sticky device error word; its device address is looked up per device.
__device__ int g_dck_error_word;

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int* g_err_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
// Test and measurement hooks: per calling thread, so that a hook set by one
// thread never acts on a call made by another.
constexpr int kMaxHookEvents = 16;
thread_local int t_decode_kernel = 0;
thread_local int t_last_launches = 0;
thread_local void* t_events[kMaxHookEvents] = {};
thread_local int t_n_events = 0;

bool device_state(int** err, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_err_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_dck_error_word) != cudaSuccess) return false;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return false;
    g_err_ptr[dev] = static_cast<int*>(p);
    g_sm_count[dev] = n;
  }
  if (err) *err = g_err_ptr[dev];
  if (sms) *sms = g_sm_count[dev];
  return true;
}

dck_status check_desc(const dck_layer_desc* d) {
  if (!d) return DCK_ERR_INVALID;
  if (d->hidden <= 0 || d->n_q_heads <= 0 || d->n_kv_heads <= 0 || d->head_dim <= 0 || d->n_groups <= 0 ||
      d->rank_v <= 0)
    return DCK_ERR_INVALID;
  if (d->dtype != DCK_BF16 && d->dtype != DCK_F32) return DCK_ERR_INVALID;
  if (d->n_q_heads % d->n_kv_heads != 0 || (d->head_dim & 1)) return DCK_ERR_INVALID;
  if (!d->group_offsets || !d->group_heads || !d->ranks) return DCK_ERR_INVALID;
  if (d->n_kv_heads > kMaxKvHeads || d->n_groups > kMaxGroups) return DCK_ERR_UNSUPPORTED;
  if (d->group_offsets[0] != 0 || d->group_offsets[d->n_groups] != d->n_kv_heads) return DCK_ERR_INVALID;
  for (int g = 0; g < d->n_groups; ++g) {
    if (d->group_offsets[g + 1] <= d->group_offsets[g]) return DCK_ERR_INVALID;
    if (d->ranks[g] <= 0) return DCK_ERR_INVALID;
  }
  bool seen[kMaxKvHeads] = {};
  for (int i = 0; i < d->n_kv_heads; ++i) {
    const int h = d->group_heads[i];
    if (h < 0 || h >= d->n_kv_heads || seen[h]) return DCK_ERR_INVALID;
    seen[h] = true;
  }
  if (d->head_dim != 64 && d->head_dim != 128) return DCK_ERR_UNSUPPORTED;
  if (d->n_q_heads / d->n_kv_heads > kMaxQPerKv) return DCK_ERR_UNSUPPORTED;
  if (d->rank_v % 16 || d->rank_v > kMaxRankV) return DCK_ERR_UNSUPPORTED;
  for (int g = 0; g < d->n_groups; ++g)
    if (d->ranks[g] % 16) return DCK_ERR_UNSUPPORTED;
  return DCK_OK;
}

LayerTable make_table(const dck_layer_desc* d) {
  LayerTable lt;
  std::memset(&lt, 0, sizeof(lt));
  lt.Hq = d->n_q_heads;
  lt.Hkv = d->n_kv_heads;
  lt.d = d->head_dim;
  lt.G = d->n_groups;
  lt.rv = d->rank_v;
  lt.qpg = d->n_q_heads / d->n_kv_heads;
  int roff = 0;
  int64_t boff = 0;
  for (int g = 0; g < d->n_groups; ++g) {
    const int n = d->group_offsets[g + 1] - d->group_offsets[g];
    lt.grp_rank[g] = d->ranks[g];
    lt.grp_roff[g] = roff;
    lt.grp_nh[g] = n;
    lt.grp_boff[g] = boff;
    for (int s = 0; s < n; ++s) {
      const int h = d->group_heads[d->group_offsets[g] + s];
      lt.head_group[h] = g;
      lt.head_slot[h] = s;
    }
    roff += d->ranks[g];
    boff += (int64_t)d->ranks[g] * n * d->head_dim;
  }
  lt.Rk = roff;
  return lt;
}

// Partial slots: CUDA-core path, c + b for work item c (one per SM) and
// sequence b it touched; tensor-core path, two per (CTA pair, sequence) and two
// per extra pair tile (tc::pair_slot_count, at most SMs / 2 pairs).  The
// workspace holds the larger count, so one size query serves both paths.
size_t n_partial_slots(int batch, int sms, int64_t n_rows) {
  const int64_t simt = (int64_t)sms + (batch > 0 ? batch - 1 : 0);
  const int64_t tc = tc::pair_slot_count(sms / 2, batch, n_rows);
  return (size_t)std::max(simt, tc);
}

size_t decode_ws_parts(const LayerTable& lt, int batch, int n_items, int64_t n_rows) {
  const size_t slots = n_partial_slots(batch, n_items, n_rows);
  return align_up(slots * lt.Hq * lt.rv * sizeof(float), 256) + align_up(slots * lt.Hq * 2 * sizeof(float), 256);
}

// Workspace: split partials U and (m, l), then the tensor-core path's extra region.
size_t decode_ws_bytes(const LayerTable& lt, int batch, int n_items, int dtype, int64_t n_rows) {
  return decode_ws_parts(lt, batch, n_items, n_rows) + (dtype == DCK_BF16 ? tc_decode_extra_ws(lt, batch, n_rows) : 0);
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" {

const char* dck_status_string(int32_t s) {
  switch (s) {
    case DCK_OK: return "ok";
    case DCK_ERR_INVALID: return "invalid argument";
    case DCK_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case DCK_ERR_WORKSPACE: return "workspace missing or too small";
    case DCK_ERR_CUDA: return "CUDA error";
    case DCK_ERR_TIMEOUT: return "device-side wait timed out";
    default: return "unknown status";
  }
}

dck_status dck_validate_desc(const dck_layer_desc* desc) { return check_desc(desc); }

int32_t dck_set_decode_kernel(int32_t which) {
  const int prev = t_decode_kernel;
  t_decode_kernel = which;
  return prev;
}

int32_t dck_last_launch_count(void) { return t_last_launches; }

dck_status dck_set_timing_events(void* const* events, int32_t n) {
  if (n == 0) {
    t_n_events = 0;
    return DCK_OK;
  }
  if (!events || n < 2 || n > kMaxHookEvents) return DCK_ERR_INVALID;
  for (int i = 0; i < n; ++i)
    if (!events[i]) return DCK_ERR_INVALID;
  for (int i = 0; i < n; ++i) t_events[i] = events[i];
  t_n_events = n;
  return DCK_OK;
}

size_t dck_decode_workspace_size(const dck_layer_desc* desc, int32_t batch, int64_t n_rows) {
  if (check_desc(desc) != DCK_OK || batch < 0 || n_rows < 0) return 0;
  int sms = 0;
  if (!device_state(nullptr, &sms)) return 0;
  return decode_ws_bytes(make_table(desc), batch, sms, desc->dtype, n_rows);
}

}  // extern "C"

namespace dck {
// Host-side argument checks of a decode call, in the order every decode entry
// point applies them, before any CUDA call.
dck_status decode_precheck(const dck_layer_desc* desc, const void* q, const void* kcache, const void* vcache,
                           int64_t n_rows, const void* B_k, const void* B_v, const int64_t* d_seq_start,
                           const int32_t* d_seq_len, int32_t batch, float rope_theta, const void* out) {
  dck_status st = check_desc(desc);
  if (st != DCK_OK) return st;
  if (batch < 0 || batch > kMaxBatch || n_rows < 0) return DCK_ERR_INVALID;
  if (!(rope_theta > 0.f) || !std::isfinite(rope_theta)) return DCK_ERR_INVALID;
  if (batch == 0) return DCK_OK;
  if (!q || !kcache || !vcache || !B_k || !B_v || !d_seq_start || !d_seq_len || !out) return DCK_ERR_INVALID;
  const size_t el = desc->dtype == DCK_F32 ? 4 : 2;
  if (!aligned(q, el) || !aligned(out, el) || !aligned(kcache, 16) || !aligned(vcache, 16) || !aligned(B_k, 16) ||
      !aligned(B_v, 16))
    return DCK_ERR_INVALID;
  return DCK_OK;
}
}  // namespace dck

extern "C" {

size_t dck_prefill_workspace_size(const dck_layer_desc* desc, int64_t n_rows) {
  if (check_desc(desc) != DCK_OK || n_rows < 0) return 0;
  const LayerTable lt = make_table(desc);
  if (!tc_prefill_supports(lt, desc->dtype)) return 0;
  return tc_prefill_workspace(lt, n_rows);
}

dck_status dck_prefill_attention(const dck_layer_desc* desc, const void* q, const int32_t* d_q_len, int32_t q_max,
                                 const void* kcache, const void* vcache, int64_t n_rows, const void* B_k,
                                 const void* B_v, const int64_t* d_seq_start, const int32_t* d_seq_len,
                                 int32_t batch, int32_t max_seq_len, float rope_theta, void* out, void* workspace,
                                 size_t ws_bytes, void* stream) {
  t_last_launches = 0;
  dck_status st =
      decode_precheck(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta, out);
  if (st != DCK_OK) return st;
  if (q_max < 1 || q_max > kMaxPrefillLen || max_seq_len < 1 || max_seq_len > kMaxPrefillLen) return DCK_ERR_INVALID;
  if (batch == 0) return DCK_OK;
  if (!d_q_len || !aligned(q, 16) || !aligned(out, 16)) return DCK_ERR_INVALID;
  const LayerTable lt = make_table(desc);
  if (!tc_prefill_supports(lt, desc->dtype) || n_rows >= (int64_t(1) << 31) - 256) return DCK_ERR_UNSUPPORTED;
  if (!workspace || ws_bytes < tc_prefill_workspace(lt, n_rows) || !aligned(workspace, 256)) return DCK_ERR_WORKSPACE;
  int* err = nullptr;
  if (!device_state(&err, nullptr)) return DCK_ERR_CUDA;
  LaunchHook hook;
  hook.ev = t_events;
  hook.n_ev = t_n_events;
  cudaError_t e = launch_prefill_tc(lt, q, d_q_len, q_max, kcache, vcache, n_rows, B_k, B_v, d_seq_start,
                                    d_seq_len, batch, max_seq_len, rope_theta, out, workspace, err, &hook,
                                    static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) e = hook_end(&hook, static_cast<cudaStream_t>(stream));
  t_last_launches = hook.count;
  return e == cudaSuccess ? DCK_OK : DCK_ERR_CUDA;
}

}  // extern "C"

namespace {
// The decode call, optionally with the decode step's latent append fused into
// its first launch (app != nullptr: the caller has checked that the fused
// append applies).
dck_status decode_call(const dck_layer_desc* desc, const void* q, const void* kcache, const void* vcache,
                       int64_t n_rows, const void* B_k, const void* B_v, const int64_t* d_seq_start,
                       const int32_t* d_seq_len, int32_t batch, float rope_theta, void* out, void* workspace,
                       size_t ws_bytes, const TcStepAppend* app, void* stream) {
  t_last_launches = 0;
  const dck_status st =
      decode_precheck(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta, out);
  if (st != DCK_OK || batch == 0) return st;
  int* err = nullptr;
  int sms = 0;
  if (!device_state(&err, &sms)) return DCK_ERR_CUDA;
  const LayerTable lt = make_table(desc);
  const size_t need = decode_ws_bytes(lt, batch, sms, desc->dtype, n_rows);
  if (!workspace || ws_bytes < need || !aligned(workspace, 256)) return DCK_ERR_WORKSPACE;
  if (!simt_supports(lt) || !combine_supports(lt)) return DCK_ERR_UNSUPPORTED;

  DecodeArgs a;
  a.q = q;
  a.kc = kcache;
  a.vc = vcache;
  a.Bk = B_k;
  a.Bv = B_v;
  a.seq_start = d_seq_start;
  a.seq_len = d_seq_len;
  a.n_rows = n_rows;
  a.B = batch;
  a.n_items = sms;
  a.theta = rope_theta;
  const size_t slots = n_partial_slots(batch, sms, n_rows);
  a.part_u = static_cast<float*>(workspace);
  a.part_ml = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                       align_up(slots * lt.Hq * lt.rv * sizeof(float), 256));
  a.out = out;
  a.err = err;
  a.extra = static_cast<char*>(workspace) + decode_ws_parts(lt, batch, sms, n_rows);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  const int pairs = t_decode_kernel == 0 && n_rows < (int64_t(1) << 31) - 256 && tc_decode_supports(lt, desc->dtype)
                        ? std::min(tc_decode_pairs(lt), sms / 2)
                        : 0;
  const bool use_tc = pairs > 0;
  if (app && !use_tc) return DCK_ERR_UNSUPPORTED;
  LaunchHook hook;
  hook.ev = t_events;
  hook.n_ev = t_n_events;
  a.hook = &hook;
  a.split_extra = use_tc ? 1 : 0;
  if (use_tc) a.n_items = 2 * pairs;  // the tensor-core kernels run on the pairs' SMs
  if (use_tc) e = launch_decode_tc(lt, a, app, s);
  else e = launch_decode_simt(lt, a, desc->dtype, s);
  if (e != cudaSuccess) return DCK_ERR_CUDA;
  e = launch_combine(lt, a, desc->dtype, s);
  if (e == cudaSuccess) e = hook_end(&hook, s);
  t_last_launches = hook.count;
  if (e != cudaSuccess) return DCK_ERR_CUDA;
  return DCK_OK;
}

// Whether dck_decode_step can fuse the append into the decode call.
bool step_fuses(const dck_layer_desc* desc, int32_t batch, int64_t n_rows) {
  if (check_desc(desc) != DCK_OK || desc->dtype != DCK_BF16 || batch < 1) return false;
  const LayerTable lt = make_table(desc);
  int sms = 0;
  if (!device_state(nullptr, &sms)) return false;
  return t_decode_kernel == 0 && n_rows < (int64_t(1) << 31) - 256 && tc_decode_supports(lt, desc->dtype) &&
         tc_step_append_supports(lt, desc->hidden, batch) && std::min(tc_decode_pairs(lt), sms / 2) > 0;
}
}  // namespace

extern "C" {

dck_status dck_decode_attention(const dck_layer_desc* desc, const void* q, const void* kcache, const void* vcache,
                                int64_t n_rows, const void* B_k, const void* B_v, const int64_t* d_seq_start,
                                const int32_t* d_seq_len, int32_t batch, float rope_theta, void* out,
                                void* workspace, size_t ws_bytes, void* stream) {
  return decode_call(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta, out,
                     workspace, ws_bytes, nullptr, stream);
}

size_t dck_decode_step_workspace_size(const dck_layer_desc* desc, int32_t batch, int64_t n_rows) {
  const size_t dw = dck_decode_workspace_size(desc, batch, n_rows);
  if (dw == 0) return 0;
  // the separate append (when the fused one does not apply) uses the space after the decode workspace
  return align_up(dw, 256) + align_up(dck_latent_append_workspace_size(desc, batch), 256);
}

dck_status dck_decode_step(const dck_layer_desc* desc, const void* x, const void* A_k, const void* A_v,
                           const int64_t* d_rows, const void* q, void* kcache, void* vcache, int64_t n_rows,
                           const void* B_k, const void* B_v, const int64_t* d_seq_start, const int32_t* d_seq_len,
                           int32_t batch, float rope_theta, void* out, void* workspace, size_t ws_bytes,
                           void* stream) {
  t_last_launches = 0;
  const dck_status st =
      decode_precheck(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta, out);
  if (st != DCK_OK || batch == 0) return st;
  if (!x || !A_k || !A_v || !d_rows || !aligned(x, 16) || !aligned(A_k, 16) || !aligned(A_v, 16))
    return DCK_ERR_INVALID;
  if (step_fuses(desc, batch, n_rows)) {
    TcStepAppend app;
    app.x = x;
    app.A_k = A_k;
    app.A_v = A_v;
    app.rows = d_rows;
    app.D = desc->hidden;
    return decode_call(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta, out,
                       workspace, ws_bytes, &app, stream);
  }
  // separate append, then the decode call (the append's scratch after the decode workspace)
  const size_t dw = align_up(dck_decode_workspace_size(desc, batch, n_rows), 256);
  if (!workspace || ws_bytes < dw) return DCK_ERR_WORKSPACE;
  dck_status r = dck_latent_append(desc, x, batch, A_k, A_v, d_rows, kcache, vcache, n_rows,
                                   static_cast<char*>(workspace) + dw, ws_bytes - dw, stream);
  if (r != DCK_OK) return r;
  const int appended = t_last_launches;
  r = dck_decode_attention(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta,
                           out, workspace, dw, stream);
  t_last_launches += appended;
  return r;
}

size_t dck_latent_append_workspace_size(const dck_layer_desc* desc, int32_t n_tok) {
  if (check_desc(desc) != DCK_OK || n_tok < 0) return 0;
  const LayerTable lt = make_table(desc);
  if (tc_append_supports(desc->hidden, lt.Rk, lt.rv, desc->dtype)) return tc_append_workspace(n_tok, lt.Rk, lt.rv);
  return 0;
}

dck_status dck_latent_append(const dck_layer_desc* desc, const void* x, int32_t n_tok, const void* A_k,
                             const void* A_v, const int64_t* d_rows, void* kcache, void* vcache, int64_t n_rows,
                             void* workspace, size_t ws_bytes, void* stream) {
  t_last_launches = 0;
  dck_status st = check_desc(desc);
  if (st != DCK_OK) return st;
  if (n_tok < 0 || n_rows < 0) return DCK_ERR_INVALID;
  if (n_tok == 0) return DCK_OK;
  if (!x || !A_k || !A_v || !d_rows || !kcache || !vcache) return DCK_ERR_INVALID;
  if (!aligned(x, 16) || !aligned(A_k, 16) || !aligned(A_v, 16) || !aligned(kcache, 16) || !aligned(vcache, 16))
    return DCK_ERR_INVALID;
  int* err = nullptr;
  if (!device_state(&err, nullptr)) return DCK_ERR_CUDA;
  const LayerTable lt = make_table(desc);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int launches = 1;  // kernels this call put on the stream
  cudaError_t e;
  if (tc_append_supports(desc->hidden, lt.Rk, lt.rv, desc->dtype)) {
    const size_t need = tc_append_workspace(n_tok, lt.Rk, lt.rv);
    if (need && (!workspace || ws_bytes < need || !aligned(workspace, 256))) return DCK_ERR_WORKSPACE;
    e = launch_append_tc(x, n_tok, desc->hidden, A_k, A_v, lt.Rk, lt.rv, d_rows, kcache, vcache, n_rows, workspace,
                         ws_bytes, err, s, &launches);
  } else {
    e = launch_append_simt(x, n_tok, desc->hidden, A_k, A_v, lt.Rk, lt.rv, d_rows, kcache, vcache, n_rows,
                           desc->dtype, err, s);
  }
  if (e != cudaSuccess) return DCK_ERR_CUDA;
  t_last_launches = launches;
  return DCK_OK;
}

dck_status dck_last_device_error(void* stream) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return DCK_ERR_CUDA;
  int* p = nullptr;
  if (!device_state(&p, nullptr)) return DCK_ERR_CUDA;
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_dck_error_word, sizeof(int)) != cudaSuccess) return DCK_ERR_CUDA;
  const int zero = 0;
  if (cudaMemcpyToSymbol(g_dck_error_word, &zero, sizeof(int)) != cudaSuccess) return DCK_ERR_CUDA;
  if (v & kErrTimeout) return DCK_ERR_TIMEOUT;
  if (v) return DCK_ERR_INVALID;
  return DCK_OK;
}

dck_status dck_selftest_bounded_wait(int64_t limit_cycles, void* stream) {
  if (limit_cycles < 1000 || limit_cycles > 4000000000LL) return DCK_ERR_INVALID;
  int* err = nullptr;
  if (!device_state(&err, nullptr)) return DCK_ERR_CUDA;
  return launch_bounded_wait_selftest((long long)limit_cycles, err, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DCK_OK
             : DCK_ERR_CUDA;
}

dck_status dck_synth_gaussian(void* dst, int64_t n, uint64_t key, int64_t start, float scale, int32_t dtype,
                              void* stream) {
  if (n < 0 || start < 0 || (dtype != DCK_BF16 && dtype != DCK_F32)) return DCK_ERR_INVALID;
  if (n == 0) return DCK_OK;
  if (!dst || !aligned(dst, dtype == DCK_F32 ? 4 : 2)) return DCK_ERR_INVALID;
  return launch_synth_gaussian(dst, n, key, start, scale, dtype, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? DCK_OK
             : DCK_ERR_CUDA;
}

}  // extern "C"
