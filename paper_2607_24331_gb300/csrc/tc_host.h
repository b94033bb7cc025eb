// Host-side interface between the tensor-core decode kernels: the scores
// kernel (decode_tc.cu) writes per-tile probabilities P and reference maxima
// into the workspace; the absorption kernel (absorb_tc.cu) turns them into the
// split partials U.
#pragma once

#include <cuda_runtime.h>

#include "common.cuh"

namespace dck {

struct TcRegions {
  const uint8_t* pglob;  // [max_tiles][hq_pad * 256 B]: P of flattened tile x as the UMMA B-operand image
  const float* mglob;    // [max_tiles][Hq]: reference max (log2 units) P of tile x was computed with
  int64_t max_tiles;
  int hq_pad;
  bool early_values;     // value loads may start before the scores kernel completes (that kernel lets
                         // the absorption launch only once the call's first launch, which may append
                         // latents, is complete)
};

// A decode step's latent append fused into the decode call (dck_decode_step).
struct TcStepAppend {
  const void* x;        // [B, D] bf16
  const void* A_k;      // [D, R_k]
  const void* A_v;      // [D, r_v]
  const int64_t* rows;  // [B] cache row of each sequence's new token
  int D;
};

// Launches the absorption kernel for the tiles the scores kernel just processed.
cudaError_t launch_absorb_tc(const LayerTable& lt, const DecodeArgs& a, const TcRegions& r, cudaStream_t s);

}  // namespace dck
