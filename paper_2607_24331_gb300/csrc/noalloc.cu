// Decode attention for callers that cannot allocate device memory.
//
// Some callers of this library are not allowed to call cudaMalloc at the point
// where they run decode attention: a serving runtime that reserved all device
// memory for its own pool at start-up, a plug-in that is handed only the
// tensors it reads and writes, or a latency-critical loop whose rules forbid
// any allocation after initialisation.  They cannot provide the scratch buffer
// that dck_decode_attention needs for its split partials.
//
// dck_decode_attention_noalloc gives them the same computation with the scratch
// taken from a fixed array that lives in the library's own device memory
// (kNoallocScratchBytes, 32 MiB; every GPU that loads the library holds it
// until the process exits).  It forwards to dck_decode_attention with that
// array as the workspace, so the kernels, their results and the error
// behaviour are those of the regular entry point.
#include <mutex>

#include "common.cuh"

namespace {

constexpr size_t kNoallocScratchBytes = size_t(32) << 20;

// The scratch array.  Host code must not pass its name to a kernel: on the
// host the symbol is only a stand-in, not a device address.  The device
// address is looked up once per device with cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDev = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDev] = {};

// Device address of the scratch array on the current device (set up on the
// first call per device), or nullptr if the lookup fails.
void* noalloc_scratch() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return nullptr;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_noalloc_ptr[dev] = p;
  }
  return g_noalloc_ptr[dev];
}

}  // namespace

extern "C" dck_status dck_decode_attention_noalloc(const dck_layer_desc* desc, const void* q, const void* kcache,
                                                   const void* vcache, int64_t n_rows, const void* B_k,
                                                   const void* B_v, const int64_t* d_seq_start,
                                                   const int32_t* d_seq_len, int32_t batch, float rope_theta,
                                                   void* out, void* stream) {
  // the regular entry point's argument checks, in its order, before the size test
  const dck_status st = dck::decode_precheck(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len,
                                             batch, rope_theta, out);
  if (st != DCK_OK || batch == 0) return st;
  const size_t need = dck_decode_workspace_size(desc, batch, n_rows);
  if (need == 0) return DCK_ERR_CUDA;  // valid arguments: only a failed device query gives 0
  if (need > kNoallocScratchBytes) return DCK_ERR_WORKSPACE;  // beyond the fixed 32 MiB scratch
  void* ws = noalloc_scratch();
  if (!ws) return DCK_ERR_CUDA;
  return dck_decode_attention(desc, q, kcache, vcache, n_rows, B_k, B_v, d_seq_start, d_seq_len, batch, rope_theta,
                              out, ws, kNoallocScratchBytes, stream);
}
