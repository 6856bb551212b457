// mds_verify_noalloc: the verification entry point for callers that cannot
// allocate device memory.  See include/mds.h for the contract.
//
// The call takes the same engine as mds_verify for the same configuration:
// the slice-dataflow engine (single, WIS, WIS0) with its workspace carved out
// of the static array, or the per-sequence engine, whose scratch is the first
// two words of the array.
#include <mutex>

#include "mds_flow.h"
#include "mds_internal.h"
#include "mds_topk.h"

namespace {

// The kernels' scratch.  Bytes [0, 256): word 0 the status word, word 1 the
// per-sequence engine's work counter.  Bytes [256, end): the dataflow
// engine's workspace (control words, task ring, per-sequence state, slice
// records).  Every GPU that loads the library holds this array until the
// process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[MDS_NOALLOC_SCRATCH_BYTES];

constexpr size_t kHead = 256;
constexpr size_t kScratchNeeded = 2 * sizeof(unsigned);
constexpr int kMaxDevices = 64;

std::mutex g_mu;
unsigned char* g_scratch_ptr[kMaxDevices] = {};
int g_grid[kMaxDevices] = {};
unsigned g_epoch[kMaxDevices] = {};

bool aligned_to(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

// Device address of the scratch on the current device, and the dataflow
// engine's grid there.  In host code the array's name is only a host-side
// stand-in; the kernels must get the address cudaGetSymbolAddress returns
// with the device current.
int scratch_for(int device, unsigned char** out, int* grid) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_scratch_ptr[device]) {
    void* ptr = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || !ptr) return mds::record_cuda_error(e, "cudaGetSymbolAddress");
    g_scratch_ptr[device] = static_cast<unsigned char*>(ptr);
    g_grid[device] = mds::flow::grid_size(device);
  }
  *out = g_scratch_ptr[device];
  *grid = g_grid[device];
  return MDS_OK;
}

unsigned next_epoch(int device) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_epoch[device] = (g_epoch[device] + 1u == 0u) ? 1u : g_epoch[device] + 1u;
  return g_epoch[device];
}

}  // namespace

extern "C" int mds_verify_noalloc(const mds_config* cfg_in, int device, const void* target_logits,
                                  const void* const* draft_logits, const int32_t* draft_model_id,
                                  const int32_t* draft_tokens, const float* temperatures, int scheme,
                                  uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len, float* out_diag,
                                  int B, void* stream) {
  if (!cfg_in) return MDS_EINVAL;
  mds_config c = *cfg_in;
  if (c.wis_s == 0) c.wis_s = 5;
  if (c.is_h == 0.f) c.is_h = 0.25f;
  if (c.omega0 == 0) c.omega0 = 20;
  if (c.omega0 < 1 || c.omega0 > MDS_MAX_OMEGA0) return MDS_EINVAL;
  if (c.acc_prob != 0 && c.acc_prob != 1) return MDS_EINVAL;
  if (c.top_k < 0 || c.top_k > MDS_MAX_TOPK) return MDS_EINVAL;
  if (c.max_B < 1 || c.K < 1 || c.K > MDS_MAX_K || c.L < 1 || c.L > MDS_MAX_L || c.V < 1 || c.V > (1 << 24))
    return MDS_ESHAPE;
  if (c.dtype != MDS_F32 && c.dtype != MDS_BF16) return MDS_EINVAL;
  if (c.wis_s < 1 || c.wis_s > MDS_MAX_S || !(c.is_h > 0.f) || c.is_h > 4.f) return MDS_EINVAL;
  if (c.cluster != 0 && c.cluster != 1 && c.cluster != 2 && c.cluster != 4 && c.cluster != 8 && c.cluster != 16)
    return MDS_EINVAL;
  if (scheme < MDS_SINGLE || scheme > MDS_WISSORT) return MDS_EINVAL;
  if (scheme == MDS_WISSORT && c.top_k <= 0) return MDS_EUNSUP;   // the top-k kernel's scheme only
  if (B < 0 || B > c.max_B) return MDS_ESHAPE;
  if (device < 0 || device >= kMaxDevices) return MDS_EINVAL;
  if (B == 0) return MDS_OK;
  if (!target_logits || !draft_logits || !draft_model_id || !draft_tokens || !temperatures || !out_tokens ||
      !out_accept_len)
    return MDS_EINVAL;
  const int es = c.dtype == MDS_F32 ? 4 : 2;
  if (!aligned_to(target_logits, es) || !aligned_to(draft_tokens, 4) || !aligned_to(temperatures, 4) ||
      !aligned_to(out_tokens, 4) || !aligned_to(out_accept_len, 4) || (out_diag && !aligned_to(out_diag, 4)))
    return MDS_EINVAL;
  mds::Params p{};
  int remap[MDS_MAX_K];
  for (int m = 0; m < MDS_MAX_K; ++m) remap[m] = -1;
  int n_models = 0;
  bool tma_ok = ((size_t)c.V * es) % 16 == 0 && aligned_to(target_logits, 16);
  for (int k = 0; k < c.K; ++k) {
    if (!draft_logits[k] || !aligned_to(draft_logits[k], es)) return MDS_EINVAL;
    tma_ok = tma_ok && aligned_to(draft_logits[k], 16);
    const int m = draft_model_id[k];
    if (m < 0 || m >= MDS_MAX_K) return MDS_EINVAL;
    if (remap[m] < 0) remap[m] = n_models++;
    p.model_of[k] = (int8_t)remap[m];
    p.drafts[k] = static_cast<const char*>(draft_logits[k]);
  }
  if (scheme == MDS_IS && n_models > MDS_MAX_IS_MODELS) return MDS_EUNSUP;

  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != device) {
    const cudaError_t se = cudaSetDevice(device);
    if (se != cudaSuccess) return mds::record_cuda_error(se, "cudaSetDevice");
  }
  int rc = mds::prepare_kernels(c.dtype);
  unsigned char* scratch = nullptr;
  int grid = 0;
  if (rc == MDS_OK) rc = scratch_for(device, &scratch, &grid);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (rc == MDS_OK && c.top_k > 0) {
    // rows restricted to their top k: the top-k kernel, the status word its only scratch
    if (!mds::topk::serves(scheme)) {
      rc = MDS_EUNSUP;
    } else {
      const cudaError_t e = cudaMemsetAsync(scratch, 0, kHead, st);
      rc = (e != cudaSuccess) ? mds::record_cuda_error(e, "mds_verify_noalloc launch")
                              : mds::topk::verify(c, scheme, p.model_of, tma_ok, target_logits, draft_logits,
                                                  draft_tokens, temperatures, out_tokens, out_accept_len, out_diag, B,
                                                  philox_seed, reinterpret_cast<unsigned*>(scratch), st);
    }
    if (prev >= 0 && prev != device) cudaSetDevice(prev);
    return rc;
  }
  if (rc == MDS_OK) {
    // the dataflow engine where mds_verify takes it (same geometry: same results)
    mds::flow::Params fp{};
    if (mds::flow_params(c, grid, scheme, p.model_of, n_models, true, tma_ok, fp)) {
      const size_t need = mds::flow::workspace_bytes(fp, B, grid);
      if (kHead + need > MDS_NOALLOC_SCRATCH_BYTES) {
        rc = MDS_ESHAPE;
      } else {
        mds::flow::carve_workspace(fp, reinterpret_cast<char*>(scratch + kHead), B, grid);
        mds::flow_buffers(fp, target_logits, draft_logits, draft_tokens, temperatures, out_tokens, out_accept_len,
                          out_diag, B, philox_seed);
        fp.status = reinterpret_cast<unsigned*>(scratch);
        fp.epoch = next_epoch(device);
        cudaError_t e = cudaMemsetAsync(scratch, 0, kHead, st);
        if (e == cudaSuccess) e = cudaMemsetAsync(scratch + kHead, 0, mds::flow::clear_bytes(fp, B, grid), st);
        if (e == cudaSuccess) e = mds::flow::launch(fp, grid, st);
        if (e != cudaSuccess) rc = mds::record_cuda_error(e, "mds_verify_noalloc launch");
      }
      if (prev >= 0 && prev != device) cudaSetDevice(prev);
      return rc;
    }
  }
  p.dtype = c.dtype;
  if (rc == MDS_OK && scheme == MDS_WIS0 && c.omega0 > MDS_MAX_OMEGA0_CLUSTER) rc = MDS_EUNSUP;
  if (rc == MDS_OK) rc = mds::launch_geometry(c, device, scheme, n_models, p);
  if (rc == MDS_OK) {
    p.target = static_cast<const char*>(target_logits);
    p.tokens = draft_tokens;
    p.temps = temperatures;
    p.out_tokens = out_tokens;
    p.out_accept = out_accept_len;
    p.out_diag = out_diag;
    p.status = reinterpret_cast<unsigned*>(scratch);
    p.queue = reinterpret_cast<unsigned*>(scratch) + 1;
    p.ticket0 = 0u;   // the counter is cleared below for every call
    p.seed = philox_seed;
    p.B = B;
    p.K = c.K;
    p.L = c.L;
    p.V = c.V;
    p.wis_s = c.wis_s;
    p.omega0 = c.omega0;
    p.acc_prob = c.acc_prob;
    p.is_h = c.is_h;
    p.bulk_ok = 1;
    p.n_models = n_models;
    p.tma_ok = tma_ok ? 1 : 0;
    int clusters = mds::max_active_clusters(p);
    if (clusters < 1) clusters = 1;
    if (clusters > B) clusters = B;
    cudaError_t e = cudaMemsetAsync(scratch, 0, kScratchNeeded, st);
    if (e == cudaSuccess) e = mds::launch(p, clusters, st);
    if (e != cudaSuccess) rc = mds::record_cuda_error(e, "mds_verify_noalloc launch");
  }
  if (prev >= 0 && prev != device) cudaSetDevice(prev);
  return rc;
}

extern "C" int mds_noalloc_status(int device, void* stream, const char** msg) {
  int count = 0;
  if (cudaGetDeviceCount(&count) != cudaSuccess || device < 0 || device >= count || device >= kMaxDevices) {
    cudaGetLastError();
    return MDS_EINVAL;
  }
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != device) {
    const cudaError_t se = cudaSetDevice(device);
    if (se != cudaSuccess) return mds::record_cuda_error(se, "cudaSetDevice");
  }
  unsigned char* scratch = nullptr;
  int grid = 0;
  int rc = scratch_for(device, &scratch, &grid);
  unsigned st = 0;
  if (rc == MDS_OK) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(&st, scratch, sizeof(st), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) rc = mds::record_cuda_error(e, "mds_noalloc_status");
  }
  if (prev >= 0 && prev != device) cudaSetDevice(prev);
  if (rc != MDS_OK) return rc;
  if (msg) *msg = mds::status_message(st);
  return (int)st;
}
