// Internal interface between the C ABI (mds_api.cu) and the verification
// kernel (mds_kernel.cu).  Not installed; not part of the public ABI.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/mds.h"

namespace mds {

constexpr int kThreads = 256;          // threads per CTA
constexpr int kMaxRows = 1 + MDS_MAX_K; // target + one row per distinct draft model
constexpr int kMaxSpecial = MDS_MAX_S * (MDS_MAX_K - 1);
constexpr int kIsNodesMax = 1024;      // trapezoid nodes for plain IS
constexpr int kIsChunk = 16;           // nodes accumulated per pass
constexpr int kXch = 34;               // floats one CTA contributes to a cluster exchange
constexpr int kMaxCluster = 16;
constexpr int kListN = 32;             // WIS candidate list: the largest target logits of a sequence

struct Params {
  const char* target;                  // [B][K][L+1][V]
  const char* drafts[MDS_MAX_K];       // K x [B][L][V]
  const int32_t* tokens;               // [B][K][L]
  const float* temps;                  // [B][1+K]
  int32_t* out_tokens;                 // [B][L+1]
  int32_t* out_accept;                 // [B]
  float* out_diag;                     // [B][L+1][4] or null
  unsigned* status;                    // status word (workspace)
  unsigned* queue;                     // work counter (workspace): monotonic tickets
  unsigned ticket0;                    // counter value when this launch starts
  unsigned long long seed;
  int B, K, L, V;
  int scheme;
  int dtype;                           // MDS_F32 / MDS_BF16
  int esize;                           // bytes per logit
  int wis_s;
  int omega0;                          // |Omega_0| bound M of MDS_WIS0
  int acc_prob;                        // 1: residual mass R at accepted depths too
  float is_h;
  int cn;                              // CTAs per cluster
  int slice;                           // tokens per CTA (multiple of 8)
  int ring_bytes;                      // streaming rings of all warps (each warp: 5 stages)
  int rows_max;                        // rows per depth at most (1 + distinct models)
  int n_models;                        // distinct draft models (ids are 0..n_models-1 after remap)
  int tma_ok;                          // rows are 16-byte aligned with a 16-byte-multiple length
  int bulk_ok;                         // rows may be read with bulk copies (device memory, not mapped host memory)
  int cand_cap;                        // WIS candidate list capacity (kListN; 0: no candidate path)
  int cand_stage;                      // WIS staging capacity (every CTA's list: cn * kListN)
  unsigned long long* dbg_exps;        // IS: quadrature exponentials evaluated (test export), or null
  int8_t model_of[MDS_MAX_K];          // remapped model id per branch
};

// Dynamic shared memory bytes the kernel needs for `p`.
size_t smem_bytes(const Params& p);

// Configure the kernel attributes once per process (dynamic smem limit,
// non-portable cluster size).  Returns a CUDA error code.
cudaError_t configure_kernel(int dtype);

// Largest number of co-resident clusters for this configuration.
int max_active_clusters(const Params& p);

// Launch the persistent verification kernel with `clusters` clusters.
cudaError_t launch(const Params& p, int clusters, cudaStream_t stream);

// Launch geometry (cluster size, slice, ring and list capacities) that
// mds_verify would use for this configuration; MDS_OK or MDS_EVOCAB.
int launch_geometry(const mds_config& cfg, int device, int scheme, int n_models, Params& p);

// One-time kernel attribute set-up for a logit type on the current device;
// MDS_OK or MDS_ECUDA.
int prepare_kernels(int dtype);

// Record the CUDA error behind an MDS_ECUDA return (the detail mds_error_string
// reports for this host thread); returns MDS_ECUDA.
int record_cuda_error(cudaError_t e, const char* where);

// Description of the highest status bit set (static string).
const char* status_message(unsigned status);

namespace flow {
struct Params;
}
constexpr int kNotServed = 1;   // a configuration left to the per-sequence engine

// Slice-dataflow engine parameters of a call with configuration c on a grid
// of `grid` CTAs (geometry sized for c.max_B sequences): false if the engine
// does not serve the call.  Buffers are filled in by flow_buffers.
bool flow_params(const mds_config& c, int grid, int scheme, const int8_t* model_of, int n_models, bool bulk_ok,
                 bool aligned16, flow::Params& p);
void flow_buffers(flow::Params& p, const void* target_logits, const void* const* draft_logits,
                  const int32_t* draft_tokens, const float* temperatures, int32_t* out_tokens,
                  int32_t* out_accept_len, float* out_diag, int B, uint64_t seed);

}  // namespace mds
