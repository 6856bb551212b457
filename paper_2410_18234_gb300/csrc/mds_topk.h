// Internal interface of the top-k verification kernel (mds_topk.cu) to the C
// ABI (mds_api.cu, mds_noalloc.cu).  Not installed; not part of the public ABI.
//
// With top-k restriction (Section 5's top-k runs, Tables 2 and 3) every row
// the walk visits keeps only its k largest logits and is renormalised, so a
// depth's laws live on at most (1 + models) * k tokens.  One CTA verifies one
// sequence: it reads each visited row once, keeps its top k exactly (ties to
// the lower token id), and one warp runs the depth's decision on the union of
// the kept tokens.  No workspace beyond the status word.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "mds_internal.h"

namespace mds {
namespace topk {

struct Params {
  const char* target;                  // [B][K][L+1][V]
  const char* drafts[MDS_MAX_K];       // K x [B][L][V]
  int8_t model_of[MDS_MAX_K];          // dense model index of each branch
  const int32_t* tokens;               // [B][K][L]
  const float* temps;                  // [B][1+K]
  int32_t* out_tokens;                 // [B][L+1]
  int32_t* out_accept;                 // [B]
  float* out_diag;                     // [B][L+1][4] or null
  unsigned* status;                    // status word (MDS_ST_* bits)
  unsigned long long seed;
  int B, K, L, V;
  int dtype, esize;
  int top_k, wis_s, scheme, acc_prob;
  int vec;                             // 1: 16-byte aligned rows of a multiple of 16 bytes
};

// Schemes the kernel serves.
inline bool serves(int scheme) {
  return scheme == MDS_SINGLE || scheme == MDS_WIS || scheme == MDS_SPECTR || scheme == MDS_WISSORT;
}

// One CTA per sequence on `stream`.
cudaError_t launch(const Params& p, cudaStream_t stream);

// The entry points' top-k call on the current device: checks the scheme
// (MDS_EUNSUP unless served), fills Params from the validated arguments
// (model_of: dense model index per branch; vec: every row is 16-byte aligned
// with a length of a multiple of 16 bytes) and launches.  Returns an MDS_*
// code; CUDA errors are recorded.
int verify(const mds_config& c, int scheme, const int8_t* model_of, bool vec, const void* target_logits,
           const void* const* draft_logits, const int32_t* draft_tokens, const float* temperatures,
           int32_t* out_tokens, int32_t* out_accept_len, float* out_diag, int B, uint64_t seed, unsigned* status,
           cudaStream_t stream);

}  // namespace topk
}  // namespace mds
