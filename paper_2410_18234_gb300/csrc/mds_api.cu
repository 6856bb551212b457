// C ABI of the verification library (declared in include/mds.h): argument
// validation, launch geometry, workspace and the host-buffer entry point.
#include <cstdio>
#include <cstring>
#include <mutex>
#include <vector>

#include "mds_flow.h"
#include "mds_internal.h"
#include "mds_topk.h"

struct mds_ctx {
  mds_config cfg;
  int device;
  unsigned* work;          // [0] status word, [1] work counter (monotonic tickets)
  unsigned tickets;        // tickets consumed by earlier launches
  int last_cn;
  // occupancy cache: (cn, dynamic smem) -> max active clusters
  struct Occ {
    int cn;
    size_t smem;
    int dtype;
    int clusters;
  };
  std::vector<Occ> occ;
  // staging buffers of mds_verify_host
  void* h_buf;
  size_t h_bytes;
  // slice-dataflow engine: workspace (control words, task ring, per-sequence
  // state and slice records; grown on demand, zero between launches) and the
  // launch counter that tags the ring's entries
  void* f_buf;
  size_t f_bytes;
  unsigned epoch;
  int f_grid;
  float* dbg_rows;         // test export of row statistics (caller-owned), or null
  unsigned long long* dbg_exps;   // count of IS quadrature exponentials (caller-owned), or null
};

namespace {

constexpr int kRingBytes = 80 * 1024;   // streaming rings: 8 warps x 5 stages of 2 KB

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    cudaGetDevice(&prev);
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    cudaGetDevice(&cur);
    if (prev >= 0 && cur != prev) cudaSetDevice(prev);
  }
};

int esize_of(int dtype) { return dtype == MDS_F32 ? 4 : 2; }

size_t round_up(size_t x, size_t m) { return (x + m - 1) / m * m; }

thread_local char g_cuda_detail[256] = "";

// Remember the CUDA error behind an MDS_ECUDA return (per host thread).
int cuda_fail(cudaError_t e, const char* where) {
  std::snprintf(g_cuda_detail, sizeof(g_cuda_detail), "CUDA runtime error in %s: %s", where,
                cudaGetErrorString(e));
  cudaGetLastError();
  return MDS_ECUDA;
}

// Kernel attributes (dynamic shared memory limit, non-portable cluster size)
// belong to a device's context: set once per (device, logit type), on the
// current device.
constexpr int kMaxDevices = 64;
bool configured[kMaxDevices][2] = {};
std::mutex config_mu;

int ensure_configured(int dtype) {
  int dev = 0;
  const cudaError_t ge = cudaGetDevice(&dev);
  if (ge != cudaSuccess) return cuda_fail(ge, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return cuda_fail(cudaErrorInvalidDevice, "kernel configuration");
  std::lock_guard<std::mutex> lk(config_mu);
  if (!configured[dev][dtype]) {
    cudaError_t e = mds::configure_kernel(dtype);
    if (e == cudaSuccess) e = mds::flow::configure(dtype);
    if (e != cudaSuccess) return cuda_fail(e, "kernel configuration");
    configured[dev][dtype] = true;
  }
  return MDS_OK;
}

int optin_smem(int device) {
  int v = 0;
  cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, device);
  return v;
}

// Fill the launch geometry (cluster size, slice, ring and list sizes) for
// n_models distinct draft models.  Rows stream through per-warp rings, so
// shared memory grows with V only through the special-token bitmap and the
// segment sums; the cluster size sets the slice each CTA streams per depth.
// Returns MDS_OK or MDS_EVOCAB.
int geometry(const mds_ctx* ctx, int scheme, int n_models, mds::Params& p) {
  const mds_config& c = ctx->cfg;
  p.esize = esize_of(c.dtype);
  p.rows_max = 1 + n_models;
  p.scheme = scheme;
  p.ring_bytes = kRingBytes;
  // candidate lists: WIS with at most three draft models in the stats pass;
  // the truncated alphabet always (its Omega_0 comes from the list)
  const bool lists = (scheme == MDS_WIS && p.rows_max <= 4) || scheme == MDS_WIS0;
  auto fill = [&](int cn) {
    p.cn = cn;
    p.slice = (int)round_up((size_t)((c.V + cn - 1) / cn), 8);
    if (lists) {
      p.cand_cap = mds::kListN;
      p.cand_stage = cn * mds::kListN;
    } else {
      p.cand_cap = p.cand_stage = 0;
    }
    return mds::smem_bytes(p);
  };
  const size_t limit = (size_t)optin_smem(ctx->device) - 12 * 1024;  // static shared state
  int cn = c.cluster;
  if (cn <= 0) {
    // Every sequence is a serial chain of depths, so as many sequences as
    // possible should be in flight: the largest cluster with cn * max_B
    // within the co-resident CTAs (two per SM), then larger while two CTAs
    // per SM would not fit the shared memory.
    int sms = 0, per_sm = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, ctx->device);
    cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, ctx->device);
    const long slots = 2L * (sms > 0 ? sms : 1);
    cn = 1;
    while (cn < mds::kMaxCluster && 2L * cn * (c.max_B > 0 ? c.max_B : 1) <= slots) cn *= 2;
    while (cn < mds::kMaxCluster && 2 * (fill(cn) + 12 * 1024) > (size_t)per_sm) cn *= 2;
    while (cn > 1 && (c.V + cn - 1) / cn < 8) cn /= 2;
  }
  if (fill(cn) > limit) return MDS_EVOCAB;
  return MDS_OK;
}

int clusters_for(mds_ctx* ctx, const mds::Params& p) {
  const size_t smem = mds::smem_bytes(p);
  for (const auto& o : ctx->occ)
    if (o.cn == p.cn && o.smem == smem && o.dtype == p.dtype) return o.clusters;
  int n = mds::max_active_clusters(p);
  if (n < 1) n = 1;
  ctx->occ.push_back({p.cn, smem, p.dtype, n});
  return n;
}

bool aligned(const void* ptr, size_t a) { return ((uintptr_t)ptr % a) == 0; }

// Page-locked host memory mapped into the device's address space: the
// pointer the device reads it through; null for any other memory.
const void* mapped_host(const void* h) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, h) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return (a.type == cudaMemoryTypeHost) ? a.devicePointer : nullptr;
}

}  // namespace

extern "C" {

const char* mds_error_string(int code) {
  switch (code) {
    case MDS_OK: return "ok";
    case MDS_EINVAL: return "invalid argument (null pointer, bad enum or misaligned buffer)";
    case MDS_ESHAPE: return "B, K, L or V outside the supported range";
    case MDS_EVOCAB: return "vocabulary does not fit the shared-memory budget";
    case MDS_ECUDA: return g_cuda_detail[0] ? g_cuda_detail : "CUDA runtime error";
    case MDS_EUNSUP: return "unsupported combination of arguments";
    default: return "unknown error";
  }
}

int mds_create(mds_ctx** out, const mds_config* cfg, int device) {
  if (!out || !cfg) return MDS_EINVAL;
  *out = nullptr;
  mds_config c = *cfg;
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
  int ndev = 0;
  const cudaError_t de = cudaGetDeviceCount(&ndev);
  if (de != cudaSuccess) return cuda_fail(de, "cudaGetDeviceCount");
  if (device < 0 || device >= ndev) return cuda_fail(cudaErrorInvalidDevice, "mds_create");
  DeviceGuard g(device);
  if (ensure_configured(c.dtype) != MDS_OK) return MDS_ECUDA;
  mds_ctx* ctx = new mds_ctx();
  ctx->cfg = c;
  ctx->device = device;
  ctx->last_cn = 0;
  ctx->tickets = 0u;
  ctx->h_buf = nullptr;
  ctx->h_bytes = 0;
  ctx->f_buf = nullptr;
  ctx->f_bytes = 0;
  ctx->epoch = 0u;
  ctx->f_grid = mds::flow::grid_size(device);
  cudaError_t me = cudaMalloc(&ctx->work, 256);
  if (me == cudaSuccess) me = cudaMemset(ctx->work, 0, 256);
  if (me != cudaSuccess) {
    delete ctx;
    return cuda_fail(me, "workspace allocation");
  }
  *out = ctx;
  return MDS_OK;
}

// The slice-dataflow engine serves single, WIS and WIS0 where its slice
// geometry fits (every configuration of the benchmarks); the per-sequence
// engine serves the rest.  Grows the context's workspace (zeroed) as needed.
int flow_verify(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits, const int8_t* model_of,
                int n_models, const int32_t* draft_tokens, const float* temperatures, int scheme,
                uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len, float* out_diag, int B,
                void* stream, bool bulk_ok, bool aligned16) {
  const mds_config& c = ctx->cfg;
  mds::flow::Params p{};
  if (!mds::flow_params(c, ctx->f_grid, scheme, model_of, n_models, bulk_ok, aligned16, p)) return mds::kNotServed;
  const size_t total = mds::flow::workspace_bytes(p, c.max_B, ctx->f_grid);
  DeviceGuard g(ctx->device);
  if (total > ctx->f_bytes) {
    // the previous buffer may still be in use by an earlier launch
    if (ctx->f_buf) {
      cudaDeviceSynchronize();
      cudaFree(ctx->f_buf);
    }
    ctx->f_buf = nullptr;
    ctx->f_bytes = 0;
    cudaError_t e = cudaMalloc(&ctx->f_buf, total);
    if (e == cudaSuccess) e = cudaMemset(ctx->f_buf, 0, total);
    if (e != cudaSuccess) {
      if (ctx->f_buf) cudaFree(ctx->f_buf);
      ctx->f_buf = nullptr;
      return cuda_fail(e, "dataflow workspace allocation");
    }
    ctx->f_bytes = total;
  }
  mds::flow::carve_workspace(p, static_cast<char*>(ctx->f_buf), c.max_B, ctx->f_grid);
  mds::flow_buffers(p, target_logits, draft_logits, draft_tokens, temperatures, out_tokens, out_accept_len, out_diag,
                    B, philox_seed);
  p.status = ctx->work;
  p.dbg_rows = ctx->dbg_rows;
  ctx->epoch = (ctx->epoch + 1u == 0u) ? 1u : ctx->epoch + 1u;
  p.epoch = ctx->epoch;
  const cudaError_t le = mds::flow::launch(p, ctx->f_grid, static_cast<cudaStream_t>(stream));
  if (le != cudaSuccess) return cuda_fail(le, "dataflow kernel launch");
  ctx->last_cn = 0;
  return MDS_OK;
}

// mds_verify with the choice of reading rows by bulk copies (device memory)
// or by plain loads only (rows in mapped host memory).
static int verify_impl(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits,
                       const int32_t* draft_model_id, const int32_t* draft_tokens, const float* temperatures,
                       int scheme, uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len,
                       float* out_diag, int B, void* stream, bool bulk_ok) {
  if (!ctx) return MDS_EINVAL;
  const mds_config& c = ctx->cfg;
  if (scheme < MDS_SINGLE || scheme > MDS_WISSORT) return MDS_EINVAL;
  if (scheme == MDS_WISSORT && c.top_k <= 0) return MDS_EUNSUP;   // the top-k kernel's scheme only
  if (B < 0 || B > c.max_B) return MDS_ESHAPE;
  if (B == 0) return MDS_OK;
  if (!target_logits || !draft_logits || !draft_model_id || !draft_tokens || !temperatures || !out_tokens ||
      !out_accept_len)
    return MDS_EINVAL;
  const int es = esize_of(c.dtype);
  if (!aligned(target_logits, es) || !aligned(draft_tokens, 4) || !aligned(temperatures, 4) ||
      !aligned(out_tokens, 4) || !aligned(out_accept_len, 4) || (out_diag && !aligned(out_diag, 4)))
    return MDS_EINVAL;
  mds::Params p{};
  int remap[MDS_MAX_K];
  for (int m = 0; m < MDS_MAX_K; ++m) remap[m] = -1;
  int n_models = 0;
  bool tma_ok = ((size_t)c.V * es) % 16 == 0 && aligned(target_logits, 16);
  for (int k = 0; k < c.K; ++k) {
    if (!draft_logits[k] || !aligned(draft_logits[k], es)) return MDS_EINVAL;
    tma_ok = tma_ok && aligned(draft_logits[k], 16);
    const int m = draft_model_id[k];
    if (m < 0 || m >= MDS_MAX_K) return MDS_EINVAL;
    if (remap[m] < 0) remap[m] = n_models++;
    p.model_of[k] = (int8_t)remap[m];
    p.drafts[k] = static_cast<const char*>(draft_logits[k]);
  }
  if (scheme == MDS_IS && n_models > MDS_MAX_IS_MODELS) return MDS_EUNSUP;
  if (c.top_k > 0) {
    // rows restricted to their top k: the top-k kernel (no workspace)
    DeviceGuard g(ctx->device);
    ctx->last_cn = 0;
    return mds::topk::verify(c, scheme, p.model_of, tma_ok, target_logits, draft_logits, draft_tokens, temperatures,
                             out_tokens, out_accept_len, out_diag, B, philox_seed, ctx->work,
                             static_cast<cudaStream_t>(stream));
  }
  {
    const int frc = flow_verify(ctx, target_logits, draft_logits, p.model_of, n_models, draft_tokens, temperatures,
                                scheme, philox_seed, out_tokens, out_accept_len, out_diag, B, stream, bulk_ok, tma_ok);
    if (frc != mds::kNotServed) return frc;
  }
  // the per-sequence engine's list holds 32 entries: |Omega_0| <= 30 there
  if (scheme == MDS_WIS0 && c.omega0 > MDS_MAX_OMEGA0_CLUSTER) return MDS_EUNSUP;
  p.dtype = c.dtype;
  int rc = geometry(ctx, scheme, n_models, p);
  if (rc != MDS_OK) return rc;
  p.target = static_cast<const char*>(target_logits);
  p.tokens = draft_tokens;
  p.temps = temperatures;
  p.out_tokens = out_tokens;
  p.out_accept = out_accept_len;
  p.out_diag = out_diag;
  p.status = ctx->work;
  p.queue = ctx->work + 1;
  p.dbg_exps = ctx->dbg_exps;
  p.seed = philox_seed;
  p.B = B;
  p.K = c.K;
  p.L = c.L;
  p.V = c.V;
  p.wis_s = c.wis_s;
  p.omega0 = c.omega0;
  p.acc_prob = c.acc_prob;
  p.is_h = c.is_h;
  p.n_models = n_models;
  p.tma_ok = tma_ok ? 1 : 0;
  p.bulk_ok = bulk_ok ? 1 : 0;
  DeviceGuard g(ctx->device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int clusters = clusters_for(ctx, p);
  if (clusters > B) clusters = B;
  // Every cluster takes tickets until one maps past B: a launch consumes
  // exactly B + clusters tickets, so the next launch's base is known here and
  // the counter never needs a reset.
  p.ticket0 = ctx->tickets;
  const cudaError_t e = mds::launch(p, clusters, st);
  if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
  ctx->tickets += (unsigned)(B + clusters);
  ctx->last_cn = p.cn;
  return MDS_OK;
}

int mds_verify(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits,
               const int32_t* draft_model_id, const int32_t* draft_tokens, const float* temperatures,
               int scheme, uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len,
               float* out_diag, int B, void* stream) {
  return verify_impl(ctx, target_logits, draft_logits, draft_model_id, draft_tokens, temperatures, scheme,
                     philox_seed, out_tokens, out_accept_len, out_diag, B, stream, true);
}

int mds_verify_host(mds_ctx* ctx, const void* target_logits, const void* const* draft_logits,
                    const int32_t* draft_model_id, const int32_t* draft_tokens, const float* temperatures,
                    int scheme, uint64_t philox_seed, int32_t* out_tokens, int32_t* out_accept_len,
                    float* out_diag, int B, void* stream) {
  if (!ctx) return MDS_EINVAL;
  const mds_config& c = ctx->cfg;
  if (B < 0 || B > c.max_B) return MDS_ESHAPE;
  if (B == 0) return MDS_OK;
  if (!target_logits || !draft_logits || !draft_model_id || !draft_tokens || !temperatures || !out_tokens ||
      !out_accept_len)
    return MDS_EINVAL;
  for (int k = 0; k < c.K; ++k)
    if (!draft_logits[k]) return MDS_EINVAL;
  const size_t es = (size_t)esize_of(c.dtype);
  DeviceGuard g0(ctx->device);
  // Logits in mapped page-locked host memory are read in place: only the
  // rows the walk visits cross the host link (plain loads, no bulk copies).
  const void* z_tgt = mapped_host(target_logits);
  const void* z_drf[MDS_MAX_K];
  bool zero_copy = z_tgt != nullptr;
  for (int k = 0; k < c.K; ++k) {
    z_drf[k] = zero_copy ? mapped_host(draft_logits[k]) : nullptr;
    zero_copy = zero_copy && z_drf[k] != nullptr;
  }
  const size_t n_tgt = zero_copy ? 0 : round_up((size_t)B * c.K * (c.L + 1) * c.V * es, 256);
  const size_t n_drf = zero_copy ? 0 : round_up((size_t)B * c.L * c.V * es, 256);
  const size_t n_tok = round_up((size_t)B * c.K * c.L * 4, 256);
  const size_t n_tmp = round_up((size_t)B * (1 + c.K) * 4, 256);
  const size_t n_out = round_up((size_t)B * (c.L + 1) * 4, 256);
  const size_t n_acc = round_up((size_t)B * 4, 256);
  const size_t n_dg = out_diag ? round_up((size_t)B * (c.L + 1) * 16, 256) : 0;
  const size_t total = n_tgt + c.K * n_drf + n_tok + n_tmp + n_out + n_acc + n_dg;
  DeviceGuard g(ctx->device);
  if (total > ctx->h_bytes) {
    if (ctx->h_buf) cudaFree(ctx->h_buf);
    ctx->h_buf = nullptr;
    ctx->h_bytes = 0;
    if (cudaMalloc(&ctx->h_buf, total) != cudaSuccess) {
      cudaGetLastError();
      return MDS_ECUDA;
    }
    ctx->h_bytes = total;
  }
  char* base = static_cast<char*>(ctx->h_buf);
  char* d_tgt = base;
  char* d_drf = d_tgt + n_tgt;
  char* d_tok = d_drf + c.K * n_drf;
  char* d_tmp = d_tok + n_tok;
  char* d_out = d_tmp + n_tmp;
  char* d_acc = d_out + n_out;
  char* d_dg = d_acc + n_acc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const void* dptr[MDS_MAX_K];
  const void* tptr = z_tgt;
  bool ok = true;
  if (zero_copy) {
    for (int k = 0; k < c.K; ++k) dptr[k] = z_drf[k];
  } else {
    tptr = d_tgt;
    ok = cudaMemcpyAsync(d_tgt, target_logits, (size_t)B * c.K * (c.L + 1) * c.V * es, cudaMemcpyHostToDevice,
                         st) == cudaSuccess;
    for (int k = 0; k < c.K && ok; ++k) {
      dptr[k] = d_drf + k * n_drf;
      ok = cudaMemcpyAsync(d_drf + k * n_drf, draft_logits[k], (size_t)B * c.L * c.V * es, cudaMemcpyHostToDevice,
                           st) == cudaSuccess;
    }
  }
  ok = ok && cudaMemcpyAsync(d_tok, draft_tokens, (size_t)B * c.K * c.L * 4, cudaMemcpyHostToDevice, st) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(d_tmp, temperatures, (size_t)B * (1 + c.K) * 4, cudaMemcpyHostToDevice, st) == cudaSuccess;
  if (!ok) {
    cudaGetLastError();
    return MDS_ECUDA;
  }
  int rc = verify_impl(ctx, tptr, dptr, draft_model_id, reinterpret_cast<const int32_t*>(d_tok),
                       reinterpret_cast<const float*>(d_tmp), scheme, philox_seed, reinterpret_cast<int32_t*>(d_out),
                       reinterpret_cast<int32_t*>(d_acc), out_diag ? reinterpret_cast<float*>(d_dg) : nullptr, B,
                       stream, !zero_copy);
  if (rc != MDS_OK) {
    cudaStreamSynchronize(st);
    return rc;
  }
  ok = cudaMemcpyAsync(out_tokens, d_out, (size_t)B * (c.L + 1) * 4, cudaMemcpyDeviceToHost, st) == cudaSuccess;
  ok = ok && cudaMemcpyAsync(out_accept_len, d_acc, (size_t)B * 4, cudaMemcpyDeviceToHost, st) == cudaSuccess;
  if (out_diag)
    ok = ok && cudaMemcpyAsync(out_diag, d_dg, (size_t)B * (c.L + 1) * 16, cudaMemcpyDeviceToHost, st) == cudaSuccess;
  ok = (cudaStreamSynchronize(st) == cudaSuccess) && ok;
  if (!ok) {
    cudaGetLastError();
    return MDS_ECUDA;
  }
  return MDS_OK;
}

int mds_status(mds_ctx* ctx, const char** msg) {
  if (!ctx) return MDS_EINVAL;
  DeviceGuard g(ctx->device);
  unsigned st = 0;
  if (cudaDeviceSynchronize() != cudaSuccess || cudaMemcpy(&st, ctx->work, sizeof(st), cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemset(ctx->work, 0, sizeof(st)) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "CUDA runtime error while reading the status word";
    return MDS_ECUDA;
  }
  if (msg) *msg = mds::status_message(st);
  return (int)st;
}

int mds_cluster_size(const mds_ctx* ctx) { return ctx ? ctx->last_cn : 0; }

int mds_debug_row_stats(mds_ctx* ctx, float* row_stats) {
  if (!ctx) return MDS_EINVAL;
  ctx->dbg_rows = row_stats;
  return MDS_OK;
}

int mds_debug_exp_count(mds_ctx* ctx, unsigned long long* counter) {
  if (!ctx) return MDS_EINVAL;
  ctx->dbg_exps = counter;
  return MDS_OK;
}

int mds_debug_probs(const void* row, int dtype, int V, float M, float invZ, float c, float* out, void* stream) {
  if (!row || !out || V <= 0 || (dtype != MDS_F32 && dtype != MDS_BF16)) return MDS_EINVAL;
  const cudaError_t e = mds::flow::launch_probs(row, dtype, V, M, invZ, c, out, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "mds_debug_probs");
  return MDS_OK;
}

int mds_phase_timers(int device, unsigned long long* cycles, int n) {
  if (!cycles || n < 0) return MDS_EINVAL;
  DeviceGuard g(device);
  const int r = mds::flow::read_phase_timers(cycles, n);
  if (r == -2) return MDS_EUNSUP;
  if (r < 0) return cuda_fail(cudaGetLastError(), "mds_phase_timers");
  return r;
}

void mds_destroy(mds_ctx* ctx) {
  if (!ctx) return;
  DeviceGuard g(ctx->device);
  if (ctx->h_buf) cudaFree(ctx->h_buf);
  if (ctx->f_buf) cudaFree(ctx->f_buf);
  if (ctx->work) cudaFree(ctx->work);
  delete ctx;
}

}  // extern "C"

// Internal helpers for entry points that have no context (mds_noalloc.cu).
namespace mds {
int launch_geometry(const mds_config& cfg, int device, int scheme, int n_models, Params& p) {
  mds_ctx view;   // host-side view only: no device work, no allocation
  view.cfg = cfg;
  view.device = device;
  return geometry(&view, scheme, n_models, p);
}
int prepare_kernels(int dtype) { return ensure_configured(dtype); }
int record_cuda_error(cudaError_t e, const char* where) { return cuda_fail(e, where); }

const char* status_message(unsigned st) {
  if (st & MDS_ST_OMEGA0) return "Omega_0 cut not certified by the candidate list; certified subset used";
  if (st & MDS_ST_BADTOKEN) return "draft token outside [0, V); token 0 used";
  if (st & MDS_ST_LP_CAP) return "stage LP reached its augmentation cap";
  if (st & MDS_ST_TIMEOUT) return "a bounded wait gave up";
  if (st & MDS_ST_ZERO_RESID) return "zero residual mass after a rejection; target row sampled";
  if (st & MDS_ST_BADTEMP) return "temperature <= 0 or not finite (1.0 used)";
  if (st & MDS_ST_NONFINITE) return "non-finite logits or normaliser";
  return "ok";
}

bool flow_params(const mds_config& c, int grid, int scheme, const int8_t* model_of, int n_models, bool bulk_ok,
                 bool aligned16, flow::Params& p) {
  if (scheme != MDS_SINGLE && scheme != MDS_WIS && scheme != MDS_WIS0) return false;
  if (grid <= 0 || c.cluster != 0 || c.max_B > 65535) return false;   // ring entries hold 16-bit ids
  p = flow::Params{};
  p.scheme = scheme;
  p.dtype = c.dtype;
  p.esize = esize_of(c.dtype);
  p.K = c.K;
  p.L = c.L;
  p.V = c.V;
  p.B = c.max_B;
  p.wis_s = c.wis_s;
  p.omega0 = c.omega0;
  p.acc_prob = c.acc_prob;
  p.n_models = n_models;
  for (int k = 0; k < c.K; ++k) p.model_of[k] = model_of[k];
  if (!flow::plan_geometry(p, grid)) return false;
  p.aligned = aligned16 ? 1 : 0;
  p.bulk = (bulk_ok && aligned16) ? 1 : 0;
  return true;
}

void flow_buffers(flow::Params& p, const void* target_logits, const void* const* draft_logits,
                  const int32_t* draft_tokens, const float* temperatures, int32_t* out_tokens,
                  int32_t* out_accept_len, float* out_diag, int B, uint64_t seed) {
  p.target = static_cast<const char*>(target_logits);
  for (int k = 0; k < p.K; ++k) p.drafts[k] = static_cast<const char*>(draft_logits[k]);
  p.tokens = draft_tokens;
  p.temps = temperatures;
  p.out_tokens = out_tokens;
  p.out_accept = out_accept_len;
  p.out_diag = out_diag;
  p.B = B;
  p.seed = seed;
}
}  // namespace mds
