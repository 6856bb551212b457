// Slice-dataflow engine for batched multi-draft speculative verification on
// GB300 (sm_103a): schemes single, weighted importance sampling (WIS) and the
// truncated alphabet (WIS0).
//
// Every row the walk visits (the target row and one row per distinct draft
// model at a depth, the target row at the bonus depth) is cut into slices of
// T tokens.  One pass of one sequence is ns slice tasks over the same rows.
// The grid is persistent (every CTA of the launch resident): in each CTA one
// scheduler warp takes task numbers from a global counter, waits for the
// task's publication in a ring in global memory, reads the sequence's pass
// descriptor and bulk-copies the task's slice of every row of the pass into
// one of two shared-memory buffers (cp.async.bulk, mbarrier completion).  The
// eight compute warps reduce the slice to a record in global memory:
//   stats    row maxima and exp sums (2^fma(l, c, -round(m c)) against the
//            slice maximum m) and, for the weighted schemes, the slice's
//            largest target logits (the candidate list) with every row's logit
//            there; the sums leave the list out, so every later mass is a sum
//            of positive terms;
//   resid    the residual mass sum max(0, q - p_I) of Algorithm 1;
//   replace  the target mass outside Omega_0 (truncated alphabet);
//   full     a full-vocabulary stage of the weighted scheme: the slice's top-s
//            keys q - a b with a and b, and the Omega_2 masses of the rest;
//   bonus    the target row's maximum and sum at depth L.
// The CTA whose task completes a pass (a per-sequence counter) runs the
// decision for that sequence: it combines the records in slice order, runs the
// importance step (the WIS stages on the merged candidate list, Omega_1 by
// the keys q - a b, the stage LP, Remark 4's pairwise stages), Algorithm 1's
// accept test, and the inverse-CDF search of a residual draw (slice by the
// records, token by one re-read of that slice), then advances the walk and
// publishes the sequence's next pass.  Decisions depend only on the data and
// the Philox draws, never on which CTA takes a task, so results are
// bit-reproducible.  Every wait is bounded in time; a wait that gives up sets
// MDS_ST_TIMEOUT and an abort flag on which every CTA leaves, after waiting
// for its own copies in flight.
#include <cstdlib>
#include <cuda_bf16.h>

#include "mds_device.cuh"
#include "mds_flow.h"

namespace mds {
namespace flow {
namespace {

using namespace mds::dev;

constexpr int kCW = 8;                 // compute warps
constexpr int kCT = kCW * 32;          // compute threads
constexpr int kBlock = kCT + 32;       // + the scheduler warp
constexpr int kNBuf = 2;               // slice buffers per CTA
constexpr int kCtasPerSm = 2;          // resident CTAs per SM (the launch bound)
constexpr int kCandCap = 512;          // candidate tokens one slice may set aside
constexpr int kListMax = 64;           // candidate list length at most
constexpr int kHdr = 2 * kMaxRows + 2; // record: (max, sum) per row, tau, list length
constexpr int kTopF = 8;               // per-thread candidates of a full stage (>= MDS_MAX_S)
constexpr int kMaxEntries = 512;       // slices x slice list length, at most
constexpr int kDecStage = 8192;        // bytes of a pass's slice records ([ns][rec_floats]) at most
// A stats pass's combined record (written over the sequence's slice records
// by the CTA that completes the pass): per row M, 1/Z and the complement
// mass, the list's length, tau, completeness and q(tau), then the list:
// ids, target logits and per row exp terms (token order of the merge).
constexpr int kCmbM = 0, kCmbIz = kMaxRows, kCmbPc = 2 * kMaxRows, kCmbN = 2 * kMaxRows + kListRowsMax;
constexpr int kCmbHdr = kCmbN + 4;
constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s bound on every wait
constexpr unsigned FULLM = 0xffffffffu;
static_assert(kHdr % 4 == 0, "record header keeps 16-byte alignment");
static_assert(kTopF >= MDS_MAX_S, "full-stage candidates");

enum : int { kNone = 0, kStats = 1, kResid = 2, kBonus = 3, kFull = 4, kReplace = 5 };

// A decision request: sequence (16 bits), kind (3), depth (7), rows (5), list (1).
__host__ __device__ constexpr unsigned dec_payload(int b, int kind, int j, int R, int list) {
  return ((unsigned)b << 16) | ((unsigned)kind << 13) | ((unsigned)j << 6) | ((unsigned)R << 1) | (unsigned)(list != 0);
}
static_assert(MDS_MAX_L < 127 && kMaxRows < 32, "decision request fields");

// Phase-timer slots (SM cycles summed over CTAs, or counts).
enum : int {
  kPhKernel = 0,        // time in the kernel (per CTA, summed)
  kPhWaitFull,          // compute warps waiting for a loaded slice
  kPhTaskList,          // stats tasks with the candidate list
  kPhTaskStats,         // stats tasks without it (and the bonus row)
  kPhTaskResid,         // residual and replace tasks
  kPhTaskFull,          // full-vocabulary stage tasks
  kPhDecStats,          // stats decisions (all of it)
  kPhDecCombine,        //   of which: combining records and the list merge
  kPhDecStages,         //   of which: the WIS stages on the list
  kPhDecResid,          // residual and replace decisions (with the search)
  kPhDecFull,           // full-stage decisions
  kPhDecBonus,          // bonus decisions
  kPhPush,              // publishing the next pass
  kPhSchedPoll,         // scheduler waiting for a published task
  kPhSchedEmpty,        // scheduler waiting for a free buffer
  kPhDecPoll,           // decision warps waiting for a request
  kPhDecPlan,           // decisions: planning a pass (rows, tokens, cached logits)
  kPhDecLoad,           // decisions: staging the state, inputs and records
  kPhDecSelect,         // decisions: WIS stage selection and masses (list)
  kPhDecAccept,         // decisions: the accept step (with its push or walk)
  kPhDecWalk,           // decisions: the walk to the next depth
  kPhListA,             // list tasks: maxima and the candidate threshold
  kPhListB,             // list tasks: the sums and the candidates
  kPhListC,             // list tasks: ranking and the record
  kPhPublish,           // a task's record publication (fence, pass counter)
  kPhCombine,           // combining a completed stats pass (the last task's CTA)
  kPhLp,                // the stage LPs (one thread)
  kPhLpCalls,           // count: stage LPs
  kPhTasks,             // count: slice tasks
  kPhDecisions,         // count: decisions
  kPhaseN
};

// ------------------------------------------------------------------ state

struct FRow {
  const char* ptr;     // row start (token 0)
  float c;             // log2(e) / temperature
  float M, invZ;       // row maximum and inverse normaliser (after the stats decision)
  float gamma;         // WIS: coefficient of this draft row in the generic law
};
struct __align__(16) FPass {   // what the slice tasks of a pass read
  int kind, j, nrows, nstream;
  int list, rb, nspec, all0;
  float cut;
  int pad0, pad1, pad2;
  FRow row[kMaxRows];          // target, then one row per distinct draft model of the valid branches
  int spec_id[kMaxSpecial];    // WIS: tokens with an explicit law value (every Omega_1 so far)
  float spec_val[kMaxSpecial];
  int pad3[2];
};
static_assert(sizeof(FPass) % 16 == 0, "pass descriptor copies in 16-byte chunks");
struct __align__(16) FWalk {   // decision state of a sequence between passes
  unsigned valid;              // valid branches at the current depth
  int stage, A;                // WIS full stages: next stage, current stage input
  int Y;                       // intermediate token
  float qY, pIY;
  int acc;                     // accept test passed
  float ures;                  // uniform of the pending inverse-CDF draw
  float R;                     // residual mass (diagnostics)
  int Yp;                      // WIS0: output of the inner step on Omega_0 (-1: none)
  int Ydiag;
  int zres;                    // the pending draw is the zero-residual fallback (sample q)
  int pad[4];
};
static_assert(sizeof(FWalk) % 16 == 0, "walk state copies in 16-byte chunks");
struct __align__(16) FSeq {
  FPass P;
  FWalk W;
};

struct __align__(16) FDesc {
  FPass P;
  int b, slice, exit, pad;
};
static_assert(sizeof(FDesc) % 16 == 0, "descriptor moves in 16-byte chunks");

struct Cand {  // full-stage candidate: larger key first, then smaller token id
  float key;
  int id;
  float a, b;
};
#define CAND_NONE Cand{kNegInf, 0x7fffffff, 0.f, 0.f}
__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

struct DState {                // the decision's working state (shared memory)
  FPass P;
  FWalk W;
  int nv;
  int vbr[MDS_MAX_K], X[MDS_MAX_K], vrow[MDS_MAX_K];
  float xl[MDS_MAX_K][kMaxRows];   // every row's logit at each valid draft token (X[k])
  int xl_ok;
  // candidate list (token-id order)
  int n, cand_all;
  float cand_q, cand_tau;
  int cm_id[kListMax];
  float cm_l0[kListMax];
  float cm_e[kListRowsMax][kListMax];
  float cm_a[kListMax];
  int cm_sp[kListMax];
  float pc[kListRowsMax];
  int ksl[kMaxSlicesList];
  int fin_s[kListMax], fin_i[kListMax];
  // stage
  int om[MDS_MAX_S];
  float om_q[MDS_MAX_S], om_a[MDS_MAX_S], om_b[MDS_MAX_S], om_x[MDS_MAX_S];
  float A2, B2;
  int Y, fast_ok;
  Cand fin[kTopF];
  float lp_rs[kMaxPairs], lp_fl[kMaxPairs], lp_fh[kMaxPairs];   // LP pair state in shared memory
  // search
  int seg, cross, lastp, tok;
  float run;
  // truncated alphabet
  int k_lane[MDS_MAX_K], k_row[MDS_MAX_K];
  int o0_n, o0_all, o0_Yp;
  // inputs of the sequence staged by the decision: draft tokens at the
  // depth (tk0) and the next depth (tk1), temperatures (target, drafts)
  int tk0[MDS_MAX_K], tk1[MDS_MAX_K];
  float tmp[MDS_MAX_K + 1];
  int xl_wait;                 // the row logits at the draft tokens are still in flight
  float o0_cut, o0_pa, o0_R;
  float rtot;
  unsigned tbase;
};
static_assert(offsetof(DState, W) == offsetof(DState, P) + sizeof(FPass) && offsetof(FSeq, W) == sizeof(FPass),
              "a sequence's state copies into the decision state in one piece");

struct FShared {
  uint64_t full[kNBuf], empty[kNBuf];
  FDesc desc[kNBuf];
  FDesc pend;                  // the scheduler's next task, resolved ahead
  float red[kCW * 2 * kMaxRows];
  float wth[kCW];
  int ncand, last, issued, consumed;
  int cmb_nv;                  // combine of a pass: valid entries
  unsigned cmb_tau;            // ... order key of tau
  float addtau;
  float add[kMaxRows];
  uint32_t bitmap[64];         // one bit per 16-byte unit of a slice holding a special token
  Cand wcand[kCW * kTopF];
  Cand blk[kTopF];
  int flag_ok, flag_ab;
#ifdef MDS_PHASE_TIMERS
  unsigned long long tm[kPhaseN];
#endif
};

// ------------------------------------------------------------------ memory helpers

__device__ __forceinline__ unsigned long long ld_acquire(const unsigned long long* a) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.u64 %0, [%1];" : "=l"(v) : "l"(a) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(unsigned long long* a, unsigned long long v) {
  asm volatile("st.release.gpu.u64 [%0], %1;" ::"l"(a), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_relaxed(const unsigned* a) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
  return v;
}
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* a, unsigned v) {
  unsigned old;
  asm volatile("atom.add.acq_rel.gpu.u32 %0, [%1], %2;" : "=r"(old) : "l"(a), "r"(v) : "memory");
  return old;
}
__device__ __forceinline__ unsigned long long now_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void cbar() { asm volatile("bar.sync 1, %0;" ::"n"(kCT) : "memory"); }

// 16-byte chunk copies of state between global (L2, coherent) and shared memory.
__device__ __forceinline__ void copy_in(void* dst, const void* src, int bytes, int t, int nt) {
  const int4* s = reinterpret_cast<const int4*>(src);
  int4* d = reinterpret_cast<int4*>(dst);
  for (int i = t; i < bytes / 16; i += nt) d[i] = __ldcg(s + i);
}
__device__ __forceinline__ void copy_out(void* dst, const void* src, int bytes, int t, int nt) {
  const int4* s = reinterpret_cast<const int4*>(src);
  int4* d = reinterpret_cast<int4*>(dst);
  for (int i = t; i < bytes / 16; i += nt) __stcg(d + i, s[i]);
}

// Asynchronous copies global -> shared (the issuing thread's own copies
// complete at cpa_wait): 16 bytes through L2 only (data other SMs write
// during the launch), 4 bytes cached (inputs only).
__device__ __forceinline__ void cpa16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa_wait() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// ------------------------------------------------------------------ phase timers
// Built with -DMDS_PHASE_TIMERS, every CTA accumulates SM cycles per phase
// (thread 0 of the compute warps, lane 0 of the scheduler warp) and adds them
// to g_phase when it leaves; mds_phase_timers() reads and clears them.
// Without it the macros vanish.
#ifdef MDS_PHASE_TIMERS
__device__ unsigned long long g_phase[kPhaseN];
#define PT_T0(v) const long long v = clock64()
#define PT_ADD(i, v)                                             \
  do {                                                           \
    if ((threadIdx.x & 0xff) == 0) S.tm[i] += (unsigned long long)(clock64() - (v)); \
  } while (0)
#define PT_CNT(i)                                 \
  do {                                            \
    if ((threadIdx.x & 0xff) == 0) S.tm[i] += 1ull; \
  } while (0)
#define PT_ADDW(i, v)                                                               \
  do {                                                                              \
    if ((threadIdx.x & 31) == 0) atomicAdd(&S.tm[i], (unsigned long long)(clock64() - (v))); \
  } while (0)
#define PT_CNTW(i)                                         \
  do {                                                     \
    if ((threadIdx.x & 31) == 0) atomicAdd(&S.tm[i], 1ull); \
  } while (0)
#else
#define PT_T0(v)
#define PT_ADD(i, v)
#define PT_CNT(i)
#define PT_ADDW(i, v)
#define PT_CNTW(i)
#endif

// ------------------------------------------------------------------ the engine

template <int DT>
struct Eng {
  using E = Elt<DT>;
  static constexpr int VE = E::VE;

  const Params& p;
  FShared& S;
  char* bufs;     // kNBuf x kBufBytes
  int* cid;       // candidate ids
  float* cl;      // candidate target logits
  int* crank;     // candidate ranks
  int* cord;      // candidates ranked past the list, in rank order

  __device__ __forceinline__ unsigned long long tag_of(unsigned t) const {
    return ((unsigned long long)p.epoch << 32) | (unsigned long long)(t + 1u);
  }
  __device__ __forceinline__ bool aborted() const { return ld_relaxed(&p.ctl[kCtlAbort]) != 0u; }
  __device__ __forceinline__ void set_abort(unsigned bits) const {
    atomicOr(p.status, bits);
    atomicExch(&p.ctl[kCtlAbort], 1u);
  }
  __device__ __forceinline__ char* buf(int bi) const { return bufs + (size_t)bi * kBufBytes; }
  __device__ __forceinline__ const char* srow(const char* b, int r) const { return b + (size_t)r * p.T * p.esize; }
  __device__ __forceinline__ uint4 raw(const char* b, int r, int u) const {
    return *reinterpret_cast<const uint4*>(srow(b, r) + 16 * u);
  }
  // Explicit value of a special token of the current law, else fallback.
  __device__ __forceinline__ float spec_lookup(const FPass& P, int tok, float fallback) const {
    for (int i = 0; i < P.nspec; ++i)
      if (P.spec_id[i] == tok) return P.spec_val[i];
    return fallback;
  }

  // -------------------------------------------------------------- scheduler warp
  __device__ bool wait_mbar(uint64_t* bar, uint32_t parity) const {
    const unsigned long long t0 = now_ns();
    for (int it = 0;; ++it) {
      if (mbar_try_wait(bar, parity)) return true;
      if ((it & 63) == 63 && now_ns() - t0 > kWaitNs) return false;
    }
  }

  // Warp-parallel plan of a sequence's depth-0 pass (every branch valid):
  // lane k < K takes branch k, and a draft model's row is that of its first
  // branch (the same rows, in the same order, as Dec::plan_warp).
  __device__ void plan_depth0_warp(int b, FPass& P) const {
    const int lane = threadIdx.x & 31;
    const int K = p.K;
    const int m = (lane < K) ? (int)p.model_of[lane] : 64 + lane;
    const unsigned same = __match_any_sync(FULLM, m);
    const bool first = lane < K && (__ffs(same) - 1) == lane;
    const unsigned fm = __ballot_sync(FULLM, first);
    const int nr = 1 + __popc(fm);
    if (first) {
      const int r = 1 + __popc(fm & ((1u << lane) - 1u));
      P.row[r].ptr = p.drafts[lane] + ((size_t)b * p.L * (size_t)p.V) * p.esize;
      float td = p.temps[(size_t)b * (1 + K) + 1 + lane];
      if (!(td > 0.f) || !(td < kPosInf)) {
        atomicOr(p.status, MDS_ST_BADTEMP);
        td = 1.f;
      }
      P.row[r].c = __fdiv_rn(kLog2e, td);
      P.row[r].M = 0.f;
      P.row[r].invZ = 0.f;
      P.row[r].gamma = 0.f;
    }
    if (lane == 0) {
      P.row[0].ptr = p.target + ((size_t)b * K * (p.L + 1) * (size_t)p.V) * p.esize;
      float tq = p.temps[(size_t)b * (1 + K)];
      if (!(tq > 0.f) || !(tq < kPosInf)) {
        atomicOr(p.status, MDS_ST_BADTEMP);
        tq = 1.f;
      }
      P.row[0].c = __fdiv_rn(kLog2e, tq);
      P.row[0].M = 0.f;
      P.row[0].invZ = 0.f;
      P.row[0].gamma = 0.f;
      P.nrows = nr;
      P.j = 0;
      P.nspec = 0;
      P.rb = 0;
      P.cut = 0.f;
      P.all0 = 0;
      P.kind = kStats;
      if (p.scheme == MDS_WIS0) {
        P.nstream = 1;
        P.list = 1;
      } else if (p.scheme == MDS_WIS) {
        P.nstream = nr;
        P.list = (K > 1 && nr <= kListRowsMax && p.ln > 0) ? 1 : 0;
      } else {
        P.nstream = min(2, nr);
        P.list = 0;
      }
    }
  }

  // Claim the next task number and resolve it into Pd: the sequence, the
  // slice and the sequence's pass descriptor (depth-0 tasks are implicit:
  // task t < B * ns is slice t % ns of sequence t / ns).  Returns 0 when no
  // work is left (every sequence finished, or an abort).  Warp-wide.
  __device__ int resolve(FDesc& Pd) {
    const int lane = threadIdx.x & 31;
    const unsigned N0 = (unsigned)p.B * (unsigned)p.ns;
    int have = 0, b = 0, s = 0;
    if (lane == 0 && !aborted()) {
      const unsigned t = atomicAdd(&p.ctl[kCtlHead], 1u);
      if (t < N0) {
        b = (int)(t / (unsigned)p.ns);
        s = (int)(t % (unsigned)p.ns);
        st_release(&p.ring_rtag[t % (unsigned)p.ring_cap], tag_of(t));
        have = 1;
      } else {
        const unsigned slot = t % (unsigned)p.ring_cap;
        const unsigned long long want = tag_of(t);
        const unsigned long long t0 = now_ns();
        PT_T0(t_poll);
        for (int it = 0;; ++it) {
          if (ld_acquire(&p.ring_tag[slot]) == want) {
            const unsigned pay = __ldcg(&p.ring_pay[slot]);
            b = (int)(pay >> 16);
            s = (int)(pay & 0xffffu);
            st_release(&p.ring_rtag[slot], want);
            have = 2;
            break;
          }
          if (ld_relaxed(&p.ctl[kCtlDone]) >= (unsigned)p.B || aborted()) break;
          if ((it & 15) == 15 && now_ns() - t0 > kWaitNs) {
            set_abort(MDS_ST_TIMEOUT);
            break;
          }
          __nanosleep(it < 16 ? 32 : 256);
        }
        PT_ADD(kPhSchedPoll, t_poll);
      }
    }
    have = __shfl_sync(FULLM, have, 0);
    b = __shfl_sync(FULLM, b, 0);
    s = __shfl_sync(FULLM, s, 0);
    if (have == 1)
      plan_depth0_warp(b, Pd.P);
    else if (have == 2)
      copy_in(&Pd.P, &reinterpret_cast<const FSeq*>(p.seq)[b].P, (int)sizeof(FPass), lane, 32);
    if (lane == 0) {
      Pd.b = b;
      Pd.slice = s;
      Pd.exit = have ? 0 : 1;
    }
    __syncwarp();
    return have != 0;
  }

  // The scheduler warp: the next task is resolved ahead (while the compute
  // warps work on the other buffer), so that a freed buffer only waits for
  // the descriptor move and the bulk copies.
  __device__ void scheduler() {
    const int lane = threadIdx.x & 31;
    int have = resolve(S.pend);
    for (int k = 0;; ++k) {
      const int bi = k % kNBuf;
      FDesc& D = S.desc[bi];
      // the compute warps released this buffer (lane 0 waits; bounded)
      int ok = 1;
      PT_T0(t_empty);
      if (lane == 0 && k >= kNBuf) ok = wait_mbar(&S.empty[bi], ((k / kNBuf) - 1) & 1) ? 1 : 0;
      PT_ADD(kPhSchedEmpty, t_empty);
      ok = __shfl_sync(FULLM, ok, 0);
      if (!ok) {
        // the compute warps still hold the buffer: leave it untouched
        if (lane == 0) set_abort(MDS_ST_TIMEOUT);
        return;
      }
      {
        const int4* src = reinterpret_cast<const int4*>(&S.pend);
        int4* dst = reinterpret_cast<int4*>(&D);
        for (int i = lane; i < (int)(sizeof(FDesc) / 16); i += 32) dst[i] = src[i];
      }
      __syncwarp();
      if (lane == 0) {
        if (have && p.bulk) {
          const int s = D.slice;
          const int tok0 = s * p.T;
          const int n = min(p.T, p.V - tok0);
          const uint32_t bytes = (uint32_t)n * (uint32_t)p.esize;
          fence_proxy_async();
          mbar_expect_tx(&S.full[bi], bytes * (uint32_t)D.P.nstream);
          for (int r = 0; r < D.P.nstream; ++r)
            bulk_copy(buf(bi) + (size_t)r * p.T * p.esize, D.P.row[r].ptr + (size_t)tok0 * p.esize, bytes, &S.full[bi]);
        } else {
          mbar_arrive(&S.full[bi]);
        }
        S.issued = k + 1;
      }
      __syncwarp();
      if (!have) return;
      have = resolve(S.pend);
    }
  }

  // -------------------------------------------------------------- slice loading (plain loads)
  // Rows [0, R) of the slice [tok0, tok0 + n) into shared memory; units past
  // n read -inf.  Used where bulk copies are not (mapped host memory, rows
  // not 16-byte aligned) and by the search's re-read of one slice.
  __device__ void load_plain(const FPass& P, int R, char* b, int tok0, int n) const {
    const int U = (n + VE - 1) / VE;
    for (int r = 0; r < R; ++r) {
      const char* src = P.row[r].ptr + (size_t)tok0 * p.esize;
      char* dst = b + (size_t)r * p.T * p.esize;
      for (int u = threadIdx.x; u < U; u += kCT) {
        uint4 x;
        if (p.aligned) {
          x = __ldg(reinterpret_cast<const uint4*>(src + 16 * (size_t)u));
        } else {
          uint32_t w[4];
          if constexpr (DT == MDS_BF16) {
            const unsigned short* s16 = reinterpret_cast<const unsigned short*>(src);
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int t0 = u * VE + 2 * h;
              const uint32_t lo = (t0 < n) ? (uint32_t)__ldg(s16 + t0) : 0xff80u;
              const uint32_t hi = (t0 + 1 < n) ? (uint32_t)__ldg(s16 + t0 + 1) : 0xff80u;
              w[h] = lo | (hi << 16);
            }
          } else {
            const float* s32 = reinterpret_cast<const float*>(src);
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const int t0 = u * VE + h;
              w[h] = (t0 < n) ? __float_as_uint(__ldg(s32 + t0)) : 0xff800000u;
            }
          }
          x = make_uint4(w[0], w[1], w[2], w[3]);
        }
        *reinterpret_cast<uint4*>(dst + 16 * (size_t)u) = x;
      }
    }
    cbar();
  }

  // One bit per 16-byte unit of the slice that holds a special token.
  __device__ void build_bitmap(const FPass& P, int tok0, int n) const {
    const int words = ((n + VE - 1) / VE + 31) / 32;
    for (int i = threadIdx.x; i < words; i += kCT) S.bitmap[i] = 0u;
    cbar();
    for (int i = threadIdx.x; i < P.nspec; i += kCT) {
      const int loc = P.spec_id[i] - tok0;
      if (loc >= 0 && loc < n) atomicOr(&S.bitmap[(loc / VE) >> 5], 1u << ((loc / VE) & 31));
    }
    cbar();
  }

  // -------------------------------------------------------------- block reductions (fixed order)
  // Sum over the compute threads: warp trees, then warps in order.  Every
  // compute thread gets the result.
  __device__ float block_sum(float v, float* scratch) const {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    cbar();
    if (lane == 0) scratch[warp] = v;
    cbar();
    float t = 0.f;
#pragma unroll
    for (int w = 0; w < kCW; ++w) t = __fadd_rn(t, scratch[w]);
    return t;
  }
  __device__ float block_max(float v, float* scratch) const {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_max(v);
    cbar();
    if (lane == 0) scratch[warp] = v;
    cbar();
    float t = kNegInf;
#pragma unroll
    for (int w = 0; w < kCW; ++w) t = fmaxf(t, scratch[w]);
    return t;
  }

  // -------------------------------------------------------------- stats task
  // R rows (compile time, at most kListRowsMax) with or without the candidate
  // list, in two passes over the slice in shared memory.  Pass A: every
  // row's maximum (the slice's exponent reference) and the candidate
  // threshold theta: the smallest of the warps' largest target logits, so
  // that at least one token per warp is >= theta (theta = -inf for a slice
  // of at most kCandCap tokens: every token is a candidate).  Pass B: every
  // row's sum of 2^(l c - m c) over the tokens that are not candidates (the
  // candidates, target logit > theta, are set aside with every row's logit).
  // Then the candidates are ranked (larger target logit first, ties to the
  // smaller id): the first LN form the slice's list, the others rejoin the
  // sums in rank order.  tau = the largest target logit outside the list.
  // Should more than kCandCap tokens pass theta, theta is raised to the
  // kCandCap-th largest target logit (bisection) and pass B repeated.
  // Record: (max, sum) per row, tau, list length, then the list: ids, then
  // each row's logits.
  template <int R, bool LIST>
  __device__ void stats_small(const FPass& P, const char* b, int tok0, int n, float* rec) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int U = (n + VE - 1) / VE;
    const int LN = p.lns;   // this slice's list length
    float c[R];
#pragma unroll
    for (int r = 0; r < R; ++r) c[r] = P.row[r].c;
    // pass A: maxima
    PT_T0(t_a);
    float tmax = kNegInf;
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float mx = kNegInf;
      for (int u = tid; u < U; u += kCT) mx = fmaxf(mx, E::unit_max(raw(b, r, u)));
      if (r == 0) tmax = mx;
      mx = warp_max(mx);
      if (lane == 0) S.red[warp * kMaxRows + r] = mx;
    }
    if constexpr (LIST) {
      // this warp's k-th largest thread maximum (distinct tokens), k = LN / kCW
      // rounded up: every warp then holds k tokens >= its value
      const int k = (LN + kCW - 1) / kCW;
      unsigned key = (tmax > kNegInf) ? ord_key(__fadd_rn(tmax, 0.f)) : 0u;
      unsigned km = 0u;
      for (int t = 0; t < k; ++t) {
        km = __reduce_max_sync(FULLM, key);
        if (!km) break;
        const unsigned who = __ballot_sync(FULLM, key == km);
        if (lane == __ffs(who) - 1) key = 0u;
      }
      if (lane == 0) S.wth[warp] = km ? ord_val(km) : kNegInf;
    }
    cbar();
    float m[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float t = kNegInf;
#pragma unroll
      for (int w = 0; w < kCW; ++w) t = fmaxf(t, S.red[w * kMaxRows + r]);
      m[r] = t;
    }
    // theta: the smallest of the warps' k-th largest thread maxima (warps
    // with fewer than k tokens left out), so at least LN tokens are >= theta
    // when every warp takes part; -inf (every token a candidate) for a slice
    // of at most kCandCap tokens
    float theta = kNegInf;
    if constexpr (LIST) {
      if (n > kCandCap) {
        theta = kPosInf;
#pragma unroll
        for (int w = 0; w < kCW; ++w) {
          const float wm = S.wth[w];
          if (wm > kNegInf) theta = fminf(theta, wm);
        }
        if (theta == kPosInf) theta = kNegInf;
      }
    }
    if (LIST) PT_ADD(kPhListA, t_a);
    PT_T0(t_b);
    float sm[R], tau;
    int nc = 0;
    for (int attempt = 0; attempt < 2; ++attempt) {
#pragma unroll
      for (int r = 0; r < R; ++r) sm[r] = 0.f;
      tau = kNegInf;
      for (int u = tid; u < U; u += kCT) {
        const uint4 x0 = raw(b, 0, u);
        float v0[VE];
        E::unpack(x0, v0);
        uint32_t cm = 0u;
        if constexpr (LIST) {
          const float um = E::unit_max(x0);
          if (um > theta) {
#pragma unroll
            for (int e = 0; e < VE; ++e) {
              if (v0[e] > theta)
                cm |= 1u << e;
              else
                tau = fmaxf(tau, v0[e]);
            }
            const int cnt = __popc(cm);
            const int pos = atomicAdd(&S.ncand, cnt);
            int q = pos;
#pragma unroll
            for (int e = 0; e < VE; ++e)
              if (cm >> e & 1u) {
                if (q < kCandCap) {
                  cid[q] = tok0 + u * VE + e;
                  cl[q] = v0[e];
                }
                ++q;
              }
          } else {
            tau = fmaxf(tau, um);
          }
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
          float v[VE];
          if (r == 0) {
#pragma unroll
            for (int e = 0; e < VE; ++e) v[e] = v0[e];
          } else {
            E::unpack(raw(b, r, u), v);
          }
          if (m[r] > kNegInf) {
            const float mc = __fmul_rn(m[r], c[r]);
            if (!cm) {
#pragma unroll
              for (int e = 0; e < VE; ++e) sm[r] = __fadd_rn(sm[r], ex2(__fmaf_rn(v[e], c[r], -mc)));
            } else {
#pragma unroll
              for (int e = 0; e < VE; ++e) {
                const float t = ex2(__fmaf_rn(v[e], c[r], -mc));
                sm[r] = __fadd_rn(sm[r], (cm >> e & 1u) ? 0.f : t);
              }
            }
          }
        }
      }
      cbar();
      nc = S.ncand;
      if (!LIST || nc <= kCandCap) break;
      // more than kCandCap tokens above theta: raise it to the kCandCap-th
      // largest target logit (bisection on order-preserving keys over every
      // bit: keys of negative logits use the low bits too) and repeat
      unsigned t = 0u;
      for (int bit = 31; bit >= 0; --bit) {
        const unsigned cand = t | (1u << bit);
        int cnt = 0;
        for (int u = tid; u < U; u += kCT) {
          float v[VE];
          E::unpack(raw(b, 0, u), v);
#pragma unroll
          for (int e = 0; e < VE; ++e) cnt += (v[e] == v[e] && ord_key(__fadd_rn(v[e], 0.f)) >= cand) ? 1 : 0;
        }
        cnt = __reduce_add_sync(FULLM, cnt);
        cbar();
        if (lane == 0) S.red[warp] = __int_as_float(cnt);
        cbar();
        int tot = 0;
#pragma unroll
        for (int w = 0; w < kCW; ++w) tot += __float_as_int(S.red[w]);
        if (tot >= kCandCap) t = cand;
      }
      theta = fmaxf(theta, ord_val(t));
      cbar();
      if (tid == 0) S.ncand = 0;
      cbar();
    }
    nc = min(nc, kCandCap);   // the bisection leaves fewer than kCandCap; never read past the arrays
    if (LIST) PT_ADD(kPhListB, t_b);
    PT_T0(t_c);
    // block sums of the rows (fixed order)
    float tot[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const float v = warp_sum(sm[r]);
      if (lane == 0) S.red[warp * kMaxRows + r] = v;
    }
    if constexpr (LIST) {
      tau = warp_max(tau);
      if (lane == 0) S.wth[warp] = tau;
    }
    cbar();
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float t = 0.f;
#pragma unroll
      for (int w = 0; w < kCW; ++w) t = __fadd_rn(t, S.red[w * kMaxRows + r]);
      tot[r] = t;
    }
    if constexpr (LIST) {
      tau = kNegInf;
#pragma unroll
      for (int w = 0; w < kCW; ++w) tau = fmaxf(tau, S.wth[w]);
      // ranks; the first LN go to the record, the rest back to the sums
      for (int i = tid; i < nc; i += kCT) {
        const float li = cl[i];
        const int ii = cid[i];
        int rk = 0;
        for (int q = 0; q < nc; ++q) rk += better(cl[q], cid[q], li, ii) ? 1 : 0;
        crank[i] = rk;
        if (rk >= LN) cord[rk - LN] = i;
      }
      cbar();
      int* rid = reinterpret_cast<int*>(rec + kHdr);
      for (int i = tid; i < nc; i += kCT) {
        const int rk = crank[i];
        if (rk < LN) {
          const int id = cid[i];
          __stcg(rid + rk, id);
          __stcg(rec + kHdr + LN + rk, cl[i]);
#pragma unroll
          for (int r = 1; r < R; ++r) {
            float v[VE];
            const int loc = id - tok0;
            E::unpack(raw(b, r, loc / VE), v);
            float l = v[0];
#pragma unroll
            for (int e = 1; e < VE; ++e)
              if (e == loc % VE) l = v[e];
            __stcg(rec + kHdr + LN * (1 + r) + rk, l);
          }
        }
      }
      const int nd = nc - LN;
      if (nd > 0) {
        if (warp == 0) {
          float add[R];
#pragma unroll
          for (int r = 0; r < R; ++r) add[r] = 0.f;
          float at = kNegInf;
          for (int t = lane; t < nd; t += 32) {
            const int i = cord[t];
            const int loc = cid[i] - tok0;
            at = fmaxf(at, cl[i]);
#pragma unroll
            for (int r = 0; r < R; ++r) {
              float v[VE];
              E::unpack(raw(b, r, loc / VE), v);
              float l = v[0];
#pragma unroll
              for (int e = 1; e < VE; ++e)
                if (e == loc % VE) l = v[e];
              if (m[r] > kNegInf) add[r] = __fadd_rn(add[r], exp_term(l, m[r], c[r]));
            }
          }
#pragma unroll
          for (int r = 0; r < R; ++r) add[r] = warp_sum(add[r]);
          at = warp_max(at);
          if (lane == 0) {
#pragma unroll
            for (int r = 0; r < R; ++r) S.add[r] = add[r];
            S.addtau = at;
          }
        }
        cbar();
#pragma unroll
        for (int r = 0; r < R; ++r) tot[r] = __fadd_rn(tot[r], S.add[r]);
        tau = fmaxf(tau, S.addtau);
      }
    }
    if (tid == 0) {
#pragma unroll
      for (int r = 0; r < R; ++r) {
        __stcg(rec + 2 * r, m[r]);
        __stcg(rec + 2 * r + 1, tot[r]);
      }
      __stcg(rec + 2 * kMaxRows, tau);
      __stcg(reinterpret_cast<int*>(rec) + 2 * kMaxRows + 1, LIST ? min(nc, LN) : 0);
      S.ncand = 0;   // for the next slice (every reader is past the barriers above)
    }
    if (LIST) PT_ADD(kPhListC, t_c);
  }

  // Stats of any number of rows, one row at a time, no candidate list.
  __device__ void stats_rows(const FPass& P, const char* b, int n, float* rec) {
    const int tid = threadIdx.x;
    const int U = (n + VE - 1) / VE;
    for (int r = 0; r < P.nstream; ++r) {
      float mx = kNegInf;
      for (int u = tid; u < U; u += kCT) mx = fmaxf(mx, E::unit_max(raw(b, r, u)));
      mx = block_max(mx, S.red);
      const float c = P.row[r].c;
      float sm = 0.f;
      if (mx > kNegInf) {
        const float mc = __fmul_rn(mx, c);
        for (int u = tid; u < U; u += kCT) {
          float v[VE];
          E::unpack(raw(b, r, u), v);
#pragma unroll
          for (int e = 0; e < VE; ++e) sm = __fadd_rn(sm, ex2(__fmaf_rn(v[e], c, -mc)));
        }
      }
      sm = block_sum(sm, S.red + kCW);
      if (tid == 0) {
        __stcg(rec + 2 * r, mx);
        __stcg(rec + 2 * r + 1, sm);
      }
    }
  }

  // -------------------------------------------------------------- weights of the inverse-CDF draws
  // Residual max(0, q - p_I) (kResid; p_I = sum_r gamma_r p_r with the
  // special tokens' explicit values), or the target mass outside Omega_0
  // (kReplace: tokens with a logit above `cut` weigh 0 unless all0 says
  // Omega_0 is empty of them), or the target mass (kBonus).
  __device__ __forceinline__ void weights(const FPass& P, const char* b, int u, int tok0, float* w) const {
    float v0[VE];
    E::unpack(raw(b, 0, u), v0);
    const float M0 = P.row[0].M, c0 = P.row[0].c, iz0 = P.row[0].invZ;
    if (P.kind == kResid) {
      float a[VE];
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = 0.f;
      for (int r = 1; r < P.nstream; ++r) {
        const float g = P.row[r].gamma;
        if (g == 0.f) continue;
        float v[VE];
        E::unpack(raw(b, r, u), v);
        const float M = P.row[r].M, c = P.row[r].c, iz = P.row[r].invZ;
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = __fmaf_rn(g, prob_of(v[e], M, c, iz), a[e]);
      }
      if (P.nspec > 0 && ((S.bitmap[u >> 5] >> (u & 31)) & 1u)) {
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = spec_lookup(P, tok0 + u * VE + e, a[e]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = fmaxf(0.f, __fsub_rn(prob_of(v0[e], M0, c0, iz0), a[e]));
    } else if (P.kind == kReplace) {
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = (P.all0 || v0[e] > P.cut) ? 0.f : prob_of(v0[e], M0, c0, iz0);
    } else {
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = prob_of(v0[e], M0, c0, iz0);
    }
  }

  // The slice's mass (record[0]) and its 32 run masses (record[4 + q]): run q
  // is units [q * upl, (q + 1) * upl), upl = ceil(units / 32), the runs the
  // decision's search walks.  A unit's mass adds its tokens in order, a run's
  // its chunks of 32 units (each a butterfly over the units), the slice's
  // its runs in order.
  __device__ void resid_task(const FPass& P, const char* b, int tok0, int n, float* rec) {
    if (P.kind == kResid && P.nspec > 0) build_bitmap(P, tok0, n);
    const int U = (n + VE - 1) / VE;
    const int upl = (U + 31) / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int q = warp; q < 32; q += kCW) {
      const int u0 = min(U, q * upl), u1 = min(U, u0 + upl);
      float run = 0.f;
      for (int c = u0; c < u1; c += 32) {
        const int u = c + lane;
        float us = 0.f;
        if (u < u1) {
          float w[VE];
          weights(P, b, u, tok0, w);
#pragma unroll
          for (int e = 0; e < VE; ++e) us = __fadd_rn(us, w[e]);
        }
        run = __fadd_rn(run, warp_sum(us));
      }
      if (lane == 0) {
        S.red[q] = run;
        __stcg(rec + 4 + q, run);
      }
    }
    cbar();
    if (threadIdx.x == 0) {
      float tot = 0.f;
      for (int q = 0; q < 32; ++q) tot = __fadd_rn(tot, S.red[q]);
      __stcg(rec, tot);
    }
  }

  // -------------------------------------------------------------- a stats pass's combine
  // Run by the CTA that completes a stats pass, with the pass's slice records
  // (rec, [ns][rec_floats]) in global memory: every row's M and 1/Z and, with
  // candidate lists, the sequence's list (the first LF of the slices' lists
  // by (logit, then slice, then position: the slices hold increasing token
  // ids and sort their own lists that way)), its complement masses and tau;
  // written over the records as the combined record.  Scratch: the task's
  // slice buffer b.  Sums over slices and entries run in fixed orders.
  __device__ __noinline__ void combine_pass(const FPass& P, char* b, float* rec) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int ns = p.ns, rf = p.rec_floats, LN = p.lns, LF = p.ln;
    const int R = P.nstream;
    const bool list = P.list != 0;
    float* sr = reinterpret_cast<float*>(b);                       // records [ns][rf]
    unsigned* sk = reinterpret_cast<unsigned*>(b + kDecStage);     // entry keys [ns * LN]
    int* fin = reinterpret_cast<int*>(sk + kMaxEntries);           // taken entries by merge rank [LF]
    int* ksl = fin + kListMax;                                     // entries taken per slice [ns]
    float* part = reinterpret_cast<float*>(ksl + kMaxSlices);      // per-warp partials [kCW][3 * kListRowsMax]
    for (int i = tid; i < ns * rf / 4; i += kCT)
      reinterpret_cast<float4*>(sr)[i] = __ldcg(reinterpret_cast<const float4*>(rec) + i);
    if (tid < ns) ksl[tid] = 0;
    if (tid == 0) {
      S.cmb_nv = 0;
      S.cmb_tau = 0u;
    }
    cbar();
    // rows: warp w takes rows w, w + kCW, ...
    float* hdr = part + kCW * 3 * kListRowsMax;   // combined header being built [kCmbHdr]
    for (int r = warp; r < R; r += kCW) {
      float M = kNegInf;
      for (int sl = lane; sl < ns; sl += 32) M = fmaxf(M, sr[sl * rf + 2 * r]);
      M = warp_max(M);
      if (!(M > kNegInf) || M != M) {
        if (lane == 0) atomicOr(p.status, MDS_ST_NONFINITE);
        M = 0.f;
      }
      const float c = P.row[r].c;
      float z = 0.f;
      for (int sl = lane; sl < ns; sl += 32) {
        const float ms = sr[sl * rf + 2 * r];
        if (ms > kNegInf) z = __fadd_rn(z, __fmul_rn(sr[sl * rf + 2 * r + 1], ref_shift(ms, M, c)));
      }
      z = warp_sum(z);
      if (lane == 0) {
        hdr[kCmbM + r] = M;
        hdr[kCmbPc + (r < kListRowsMax ? r : 0)] = z;   // the slices' sums (list passes add the entries left out)
        if (!list) {
          if (!(z > 0.f) || !(z < kPosInf) || z != z) {
            atomicOr(p.status, MDS_ST_NONFINITE);
            z = 1.f;
          }
          hdr[kCmbIz + r] = __frcp_rn(z);
        }
      }
    }
    if (!list) {
      cbar();
      for (int i = tid; i < 2 * kMaxRows; i += kCT) __stcg(rec + i, hdr[i]);
      return;
    }
    // entries: keys (0: no entry), the valid count
    const int NE = ns * LN;
    for (int i0 = warp * 32; i0 < NE; i0 += kCT) {   // warp-uniform trips (the ballot below)
      const int i = i0 + lane;
      unsigned k = 0u;
      if (i < NE) {
        const int sl = i / LN, q = i - sl * LN;
        if (q < __float_as_int(sr[sl * rf + 2 * kMaxRows + 1]))
          k = ord_key(__fadd_rn(sr[sl * rf + kHdr + LN + q], 0.f));
        sk[i] = k;
      }
      const unsigned vb = __ballot_sync(FULLM, k != 0u);
      if (lane == 0 && vb) atomicAdd(&S.cmb_nv, __popc(vb));
    }
    cbar();
    const int nf = min(LF, S.cmb_nv);
    // rank of each valid entry in the merge order; the first nf are taken
    for (int i = tid; i < NE; i += kCT) {
      const unsigned k = sk[i];
      if (k == 0u) continue;
      int rank = 0;
      for (int u = 0; u < NE; ++u) {
        const unsigned ku = sk[u];
        rank += (ku > k || (ku == k && u < i)) ? 1 : 0;
      }
      if (rank < nf) {
        fin[rank] = i;
        atomicAdd(&ksl[i / LN], 1);
      }
    }
    cbar();
    // tau and the complement masses: entries not taken (and the slices' own tau)
    float add[kListRowsMax];
#pragma unroll
    for (int r = 0; r < kListRowsMax; ++r) add[r] = 0.f;
    float tau = kNegInf;
    for (int sl = tid; sl < ns; sl += kCT) tau = fmaxf(tau, sr[sl * rf + 2 * kMaxRows]);
    for (int i = tid; i < NE; i += kCT) {
      const int sl = i / LN, q = i - sl * LN;
      if (q >= ksl[sl] && q < __float_as_int(sr[sl * rf + 2 * kMaxRows + 1])) {
        const float* e = sr + sl * rf + kHdr + q;
        tau = fmaxf(tau, e[LN]);
#pragma unroll
        for (int r = 0; r < kListRowsMax; ++r)
          if (r < R) add[r] = __fadd_rn(add[r], exp_term(e[(1 + r) * LN], hdr[kCmbM + r], P.row[r].c));
      }
    }
    tau = warp_max(tau);
#pragma unroll
    for (int r = 0; r < kListRowsMax; ++r) add[r] = warp_sum(add[r]);
    if (lane == 0) {
      if (tau > kNegInf) atomicMax(&S.cmb_tau, ord_key(tau));
#pragma unroll
      for (int r = 0; r < kListRowsMax; ++r) part[warp * 3 * kListRowsMax + r] = add[r];
    }
    // the list into the combined record: merge order for the weighted
    // scheme, token-id order for the truncated alphabet
    const bool by_id = p.scheme == MDS_WIS0;
    float* out_id = rec + kCmbHdr;
    float* out_l0 = out_id + LF;
    float* out_e = out_l0 + LF;
    float z[kListRowsMax];
#pragma unroll
    for (int r = 0; r < kListRowsMax; ++r) z[r] = 0.f;
    for (int t = tid; t < nf; t += kCT) {
      const int i = fin[t];
      const int sl = i / LN, q = i - sl * LN;
      const float* e = sr + sl * rf + kHdr + q;
      const int id = __float_as_int(e[0]);
      int pos = t;
      if (by_id) {
        pos = 0;
        for (int u = 0; u < nf; ++u) {
          const int iu = fin[u];
          const int su = iu / LN, qu = iu - su * LN;
          pos += (__float_as_int(sr[su * rf + kHdr + qu]) < id) ? 1 : 0;
        }
      }
      __stcg(out_id + pos, __int_as_float(id));
      __stcg(out_l0 + pos, e[LN]);
#pragma unroll
      for (int r = 0; r < kListRowsMax; ++r)
        if (r < R) {
          const float ev = exp_term(e[(1 + r) * LN], hdr[kCmbM + r], P.row[r].c);
          __stcg(out_e + r * LF + pos, ev);
          z[r] = __fadd_rn(z[r], ev);
        }
    }
#pragma unroll
    for (int r = 0; r < kListRowsMax; ++r) {
      z[r] = warp_sum(z[r]);
      if (lane == 0) part[warp * 3 * kListRowsMax + kListRowsMax + r] = z[r];
    }
    cbar();
    if (tid == 0) {
      for (int r = 0; r < R; ++r) {
        float a = 0.f, zz = 0.f;
        for (int w = 0; w < kCW; ++w) {
          a = __fadd_rn(a, part[w * 3 * kListRowsMax + r]);
          zz = __fadd_rn(zz, part[w * 3 * kListRowsMax + kListRowsMax + r]);
        }
        const float pc = __fadd_rn(hdr[kCmbPc + r], a);
        float Z = __fadd_rn(pc, zz);
        if (!(Z > 0.f) || !(Z < kPosInf) || Z != Z) {
          atomicOr(p.status, MDS_ST_NONFINITE);
          Z = 1.f;
        }
        hdr[kCmbPc + r] = pc;
        hdr[kCmbIz + r] = __frcp_rn(Z);
      }
      const float t = S.cmb_tau ? ord_val(S.cmb_tau) : kNegInf;
      hdr[kCmbN] = __int_as_float(nf);
      hdr[kCmbN + 1] = t;
      hdr[kCmbN + 2] = __int_as_float(nf == p.V ? 1 : 0);
      hdr[kCmbN + 3] = (t > kNegInf) ? exp_term(t, hdr[kCmbM], P.row[0].c) : 0.f;
    }
    cbar();
    for (int i = tid; i < kCmbHdr; i += kCT) __stcg(rec + i, hdr[i]);
  }

  // -------------------------------------------------------------- full-vocabulary stage task
  __device__ __forceinline__ static void cand_insert(Cand (&top)[kTopF], const Cand& c, float& ra, float& rb) {
    if (better(c.key, c.id, top[kTopF - 1].key, top[kTopF - 1].id)) {
      ra = __fadd_rn(ra, top[kTopF - 1].a);
      rb = __fadd_rn(rb, top[kTopF - 1].b);
      top[kTopF - 1] = c;
#pragma unroll
      for (int t = kTopF - 1; t > 0; --t) {
        if (better(top[t].key, top[t].id, top[t - 1].key, top[t - 1].id)) {
          const Cand x = top[t];
          top[t] = top[t - 1];
          top[t - 1] = x;
        }
      }
    } else {
      ra = __fadd_rn(ra, c.a);
      rb = __fadd_rn(rb, c.b);
    }
  }

  // Warp-wide merge of per-lane sorted lists (best first): lane 0 writes the
  // warp's best `rounds` entries to out[0..rounds) and CAND_NONE after them;
  // every entry not popped adds its a and b (fixed order) to rest_a / rest_b.
  __device__ static void warp_merge(Cand (&top)[kTopF], Cand* out, int rounds, float& rest_a, float& rest_b) {
    const int lane = threadIdx.x & 31;
#pragma unroll 1
    for (int t = 0; t < kTopF; ++t) {
      if (t >= rounds) {
        if (lane == 0) out[t] = CAND_NONE;
        continue;
      }
      float bk = top[0].key;
      int bid = top[0].id;
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        const float ok = __shfl_xor_sync(FULLM, bk, o);
        const int oid = __shfl_xor_sync(FULLM, bid, o);
        if (better(ok, oid, bk, bid)) {
          bk = ok;
          bid = oid;
        }
      }
      const bool mine = (top[0].id == bid && top[0].key == bk && bid != 0x7fffffff);
      const unsigned who = __ballot_sync(FULLM, mine);
      const int src = who ? __ffs(who) - 1 : 0;
      const float wa = __shfl_sync(FULLM, top[0].a, src);
      const float wb = __shfl_sync(FULLM, top[0].b, src);
      if (mine) {
#pragma unroll
        for (int i = 0; i < kTopF - 1; ++i) top[i] = top[i + 1];
        top[kTopF - 1] = CAND_NONE;
      }
      if (lane == 0) out[t] = who ? Cand{bk, bid, wa, wb} : CAND_NONE;
    }
    float ra = 0.f, rb = 0.f;
#pragma unroll
    for (int i = 0; i < kTopF; ++i) {
      ra = __fadd_rn(ra, top[i].a);
      rb = __fadd_rn(rb, top[i].b);
    }
    rest_a = warp_sum(ra);
    rest_b = warp_sum(rb);
  }

  // Record: [0] a-mass and [1] b-mass of the slice outside its top s, [4..)
  // the top s (key, id, a, b) as four arrays of kTopF.
  __device__ void full_task(const FPass& P, const char* b, int tok0, int n, float* rec) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int s = min(p.wis_s, p.V);
    const int rb = P.rb;
    if (P.nspec > 0) build_bitmap(P, tok0, n);
    Cand top[kTopF];
#pragma unroll
    for (int t = 0; t < kTopF; ++t) top[t] = CAND_NONE;
    float suma = 0.f, sumb = 0.f;
    const int U = (n + VE - 1) / VE;
    const float M0 = P.row[0].M, c0 = P.row[0].c, iz0 = P.row[0].invZ;
    for (int u = tid; u < U; u += kCT) {
      float v0[VE], a[VE], bb[VE];
      E::unpack(raw(b, 0, u), v0);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        a[e] = 0.f;
        bb[e] = 0.f;
      }
      for (int r = 1; r < P.nstream; ++r) {
        const float g = P.row[r].gamma;
        if (g == 0.f && r != rb) continue;
        float v[VE];
        E::unpack(raw(b, r, u), v);
        const float M = P.row[r].M, c = P.row[r].c, iz = P.row[r].invZ;
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float pr = prob_of(v[e], M, c, iz);
          if (g != 0.f) a[e] = __fmaf_rn(g, pr, a[e]);
          if (r == rb) bb[e] = pr;
        }
      }
      if (P.nspec > 0 && ((S.bitmap[u >> 5] >> (u & 31)) & 1u)) {
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = spec_lookup(P, tok0 + u * VE + e, a[e]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        if (u * VE + e >= n) break;
        const float q = prob_of(v0[e], M0, c0, iz0);
        cand_insert(top, Cand{__fmaf_rn(-a[e], bb[e], q), tok0 + u * VE + e, a[e], bb[e]}, suma, sumb);
      }
    }
    {
      float ra, rbs;
      warp_merge(top, S.wcand + warp * kTopF, s, ra, rbs);
      suma = warp_sum(suma);
      sumb = warp_sum(sumb);
      if (lane == 0) {
        S.red[warp * 2] = __fadd_rn(suma, ra);
        S.red[warp * 2 + 1] = __fadd_rn(sumb, rbs);
      }
    }
    cbar();
    if (warp == 0) {
#pragma unroll
      for (int t = 0; t < kTopF; ++t) top[t] = (lane < kCW) ? S.wcand[lane * kTopF + t] : CAND_NONE;
      float ra, rbs;
      warp_merge(top, S.blk, s, ra, rbs);
      __syncwarp();
      if (lane == 0) {
        float sa = ra, sb = rbs;
        for (int w = 0; w < kCW; ++w) {
          sa = __fadd_rn(sa, S.red[w * 2]);
          sb = __fadd_rn(sb, S.red[w * 2 + 1]);
        }
        __stcg(rec + 0, sa);
        __stcg(rec + 1, sb);
      }
      if (lane < kTopF) {
        __stcg(rec + 4 + lane, S.blk[lane].key);
        __stcg(reinterpret_cast<int*>(rec) + 4 + kTopF + lane, S.blk[lane].id);
        __stcg(rec + 4 + 2 * kTopF + lane, S.blk[lane].a);
        __stcg(rec + 4 + 3 * kTopF + lane, S.blk[lane].b);
      }
    }
  }

  // -------------------------------------------------------------- compute warps
  // The pass of a sequence is complete: publish a decision request (thread
  // 0, after acquiring every slice's record through the pass counter; the
  // release of the request's tag passes them on to the decision warp).
  __device__ void post_decision(unsigned pay) const {
    const unsigned t = atomicAdd(&p.ctl[kCtlDecTail], 1u);
    const unsigned slot = t % (unsigned)p.dec_cap;
    if (t >= (unsigned)p.dec_cap) {
      const unsigned long long prev = tag_of(t - (unsigned)p.dec_cap);
      const unsigned long long t0 = now_ns();
      for (int it = 0; ld_acquire(&p.dec_rtag[slot]) != prev; ++it) {
        if (aborted()) break;
        if ((it & 15) == 15 && now_ns() - t0 > kWaitNs) {
          set_abort(MDS_ST_TIMEOUT);
          break;
        }
        __nanosleep(64);
      }
    }
    __stcg(p.dec_pay + slot, pay);
    st_release(&p.dec_tag[slot], tag_of(t));
  }

  __device__ void process(int bi) {
    FDesc& Dd = S.desc[bi];
    char* b = buf(bi);
    const int s = Dd.slice, seqb = Dd.b;
    const int tok0 = s * p.T, n = min(p.T, p.V - tok0);
    const FPass& P = Dd.P;
    if (!p.bulk) load_plain(P, P.nstream, b, tok0, n);
    float* rec = p.rec + ((size_t)seqb * p.ns + s) * p.rec_floats;
    PT_T0(t_task);
    PT_CNT(kPhTasks);
    switch (P.kind) {
      case kStats:
      case kBonus:
        if (P.list) {
          switch (P.nstream) {
            case 1: stats_small<1, true>(P, b, tok0, n, rec); break;
            case 2: stats_small<2, true>(P, b, tok0, n, rec); break;
            case 3: stats_small<3, true>(P, b, tok0, n, rec); break;
            default: stats_small<4, true>(P, b, tok0, n, rec); break;
          }
        } else {
          switch (P.nstream) {
            case 1: stats_small<1, false>(P, b, tok0, n, rec); break;
            case 2: stats_small<2, false>(P, b, tok0, n, rec); break;
            default: stats_rows(P, b, n, rec); break;
          }
        }
        break;
      case kResid:
      case kReplace: resid_task(P, b, tok0, n, rec); break;
      case kFull: full_task(P, b, tok0, n, rec); break;
      default: break;
    }
    PT_ADD(P.kind == kStats ? (P.list ? kPhTaskList : kPhTaskStats)
                            : (P.kind == kBonus ? kPhTaskStats : (P.kind == kFull ? kPhTaskFull : kPhTaskResid)),
           t_task);
    if (P.kind == kStats && P.j == 0 && s == 0) {
      // the sequence's outputs start as -1 (the decisions overwrite them)
      for (int j = threadIdx.x; j <= p.L; j += kCT) __stcg(p.out_tokens + (size_t)seqb * (p.L + 1) + j, -1);
      if (threadIdx.x == 0) __stcg(p.out_accept + seqb, -1);
    }
    // publish the record: the barrier orders every thread's record writes
    // before thread 0's release (acq_rel: the last arriver also acquires the
    // other slices' records)
    PT_T0(t_pub);
    cbar();
    if (threadIdx.x == 0) S.last = (atom_add_acq_rel(&p.cnt[seqb], 1u) == (unsigned)(p.ns - 1)) ? 1 : 0;
    cbar();
    PT_ADD(kPhPublish, t_pub);
    if (S.last) {
      // thread 0 acquired the other slices' records; the barrier passes that on
      PT_T0(t_cmb);
      if (P.kind == kStats) combine_pass(P, b, rec - (size_t)s * p.rec_floats);
      cbar();
      if (threadIdx.x == 0) {
        __threadfence();   // the combined record before the request
        post_decision(dec_payload(seqb, P.kind, P.j, P.nstream, P.list));
      }
      PT_ADD(kPhCombine, t_cmb);
    }
  }

  __device__ void compute() {
    for (int k = 0;; ++k) {
      const int bi = k % kNBuf;
      const uint32_t par = (k / kNBuf) & 1;
      // thread 0 waits (bounded); the others then see the completed phase
      PT_T0(t_wait);
      if (threadIdx.x == 0) {
        const bool ok = wait_mbar(&S.full[bi], par);
        if (!ok) set_abort(MDS_ST_TIMEOUT);
        S.flag_ok = ok ? 1 : 0;
        S.flag_ab = aborted() ? 1 : 0;
      }
      cbar();
      PT_ADD(kPhWaitFull, t_wait);
      if (!S.flag_ok) break;
      while (!mbar_try_wait(&S.full[bi], par)) {
      }
      if (S.desc[bi].exit) break;
      if (!S.flag_ab) process(bi);
      // generic accesses of this buffer before the next bulk copy into it
      fence_proxy_async();
      cbar();
      if (threadIdx.x == 0) {
        S.consumed = k + 1;
        mbar_arrive(&S.empty[bi]);
      }
    }
  }

};

// ================================================================== decisions
// One decision warp (on a decision SM) runs one sequence's decision at a
// time: the records of the pass just completed, the importance step, the
// accept test and the inverse-CDF search, then the sequence's next pass.
// Single-warp code throughout (lane 0 for the serial steps); its state and
// scratch are this warp's own shared memory.

constexpr int kDecScratch = kDecStage + 2 * kMaxSlices * 4 + 64 * 4;   // + slice masses, maxima, bitmap

// Each kind of decision out of line (its own register allocation); each
// rebuilds the warp's view of its shared state.
template <int DT> __device__ __noinline__ void dec_stats_nl(int b, int j, int R, bool list);
template <int DT> __device__ __noinline__ void dec_resid_nl(int b);
template <int DT> __device__ __noinline__ void dec_replace_nl(int b);
template <int DT> __device__ __noinline__ void dec_full_nl(int b);
template <int DT> __device__ __noinline__ void dec_bonus_nl(int b);
template <int DT> __device__ __noinline__ void dec_wis0_nl(int b);
template <int DT> __device__ __noinline__ void dec_accept_nl(int b);
__device__ __forceinline__ int lp_solve5(int s, float A2, float B2, int A, int Btok, float u);
__device__ __noinline__ int lp_solve8(int s, float A2, float B2, int A, int Btok, float u);

template <int DT>
struct Dec {
  using E = Elt<DT>;
  static constexpr int VE = E::VE;

  const Params& p;
  FShared& S;      // the CTA's shared state (phase timers)
  DState& D;       // this warp's decision state
  char* scr;       // this warp's scratch: staged records
  float* Rs;       // slice masses of a search [kMaxSlices]
  float* Hm;       // slice maxima of the bonus draw [kMaxSlices]
  uint32_t* bm;    // special-token bits of a re-read slice [64]
  int lane;

  __device__ __forceinline__ unsigned long long tag_of(unsigned t) const {
    return ((unsigned long long)p.epoch << 32) | (unsigned long long)(t + 1u);
  }
  __device__ __forceinline__ bool aborted() const { return ld_relaxed(&p.ctl[kCtlAbort]) != 0u; }
  __device__ __forceinline__ void set_abort(unsigned bits) const {
    atomicOr(p.status, bits);
    atomicExch(&p.ctl[kCtlAbort], 1u);
  }

  // -------------------------------------------------------------- point values
  __device__ __forceinline__ float logit_at(const FPass& P, int r, int x) const {
    if (D.xl_ok)
      for (int k = 0; k < D.nv; ++k)
        if (D.X[k] == x) return D.xl[k][r];
    return E::global(P.row[r].ptr, x);
  }
  __device__ __forceinline__ float prob_row(const FPass& P, int r, int x) const {
    return prob_of(logit_at(P, r, x), P.row[r].M, P.row[r].c, P.row[r].invZ);
  }
  __device__ __forceinline__ float spec_lookup(const FPass& P, int tok, float fallback) const {
    for (int i = 0; i < P.nspec; ++i)
      if (P.spec_id[i] == tok) return P.spec_val[i];
    return fallback;
  }
  // Point value of the current law p_I (WIS): explicit value of a special
  // token, else sum_r gamma_r p_r(x) in row order.
  __device__ float law_at(const FPass& P, int x) const {
    float a = 0.f;
    for (int r = 1; r < P.nrows; ++r)
      if (P.row[r].gamma != 0.f) a = __fmaf_rn(P.row[r].gamma, prob_row(P, r, x), a);
    return spec_lookup(P, x, a);
  }

  // -------------------------------------------------------------- planning
  // Rows of depth j for the valid branches (the lowest valid branch's target
  // row, then one row per distinct draft model in branch order), one lane per
  // branch; the valid branches, their tokens (tk: the staged tokens of depth
  // j) and rows; with want_xl, every row's logit at each draft token, by
  // asynchronous copies that xl_sync completes.
  __device__ void plan_warp(int b, int j, unsigned valid, bool bonus, bool set_pass, bool want_xl, const int* tk) {
    FPass& P = D.P;
    const int K = p.K;
    const bool v = !bonus && lane < K && ((valid >> lane) & 1u);
    const int m = v ? (int)p.model_of[lane] : 64 + lane;
    const unsigned same = __match_any_sync(FULLM, m);
    const bool first = v && (__ffs(same) - 1) == lane;
    const unsigned fm = __ballot_sync(FULLM, first);
    const unsigned vm = __ballot_sync(FULLM, v);
    const int nr = 1 + __popc(fm);
    const int myrow = first ? 1 + __popc(fm & ((1u << lane) - 1u)) : 0;
    const int row = __shfl_sync(FULLM, myrow, __ffs(same) - 1);
    if (v) {
      const int i = __popc(vm & ((1u << lane) - 1u));
      int x = tk[lane];
      if (x < 0 || x >= p.V) {
        atomicOr(p.status, MDS_ST_BADTOKEN);
        x = 0;
      }
      D.vbr[i] = lane;
      D.X[i] = x;
      D.vrow[i] = row;
    }
    if (set_pass && first) {
      P.row[myrow].ptr = p.drafts[lane] + (((size_t)b * p.L + j) * (size_t)p.V) * p.esize;
      float td = D.tmp[1 + lane];
      if (!(td > 0.f) || !(td < kPosInf)) {
        atomicOr(p.status, MDS_ST_BADTEMP);
        td = 1.f;
      }
      P.row[myrow].c = __fdiv_rn(kLog2e, td);
      P.row[myrow].M = 0.f;
      P.row[myrow].invZ = 0.f;
      P.row[myrow].gamma = 0.f;
    }
    if (lane == 0) {
      D.nv = __popc(vm);
      if (set_pass) {
        const int kstar = __ffs(valid) - 1;
        P.row[0].ptr = p.target + ((((size_t)b * K + kstar) * (p.L + 1) + j) * (size_t)p.V) * p.esize;
        float tq = D.tmp[0];
        if (!(tq > 0.f) || !(tq < kPosInf)) {
          atomicOr(p.status, MDS_ST_BADTEMP);
          tq = 1.f;
        }
        P.row[0].c = __fdiv_rn(kLog2e, tq);
        P.row[0].M = 0.f;
        P.row[0].invZ = 0.f;
        P.row[0].gamma = 0.f;
        P.nrows = nr;
        P.j = j;
        P.nspec = 0;
        P.rb = 0;
        P.cut = 0.f;
        P.all0 = 0;
        if (bonus) {
          P.kind = kBonus;
          P.nstream = 1;
          P.list = 0;
        } else {
          P.kind = kStats;
          if (p.scheme == MDS_WIS0) {
            P.nstream = 1;
            P.list = 1;
          } else if (p.scheme == MDS_WIS) {
            P.nstream = nr;
            P.list = (__popc(vm) > 1 && nr <= kListRowsMax && p.ln > 0) ? 1 : 0;
          } else {
            P.nstream = min(2, nr);
            P.list = 0;
          }
        }
      }
    }
    if (lane == 0) {
      D.xl_ok = 0;
      D.xl_wait = 0;
    }
    __syncwarp();
    if (want_xl && !bonus) {
      const int nv = D.nv, nrow = P.nrows;
      for (int i = lane; i < nv * nrow; i += 32) {
        const int k = i / nrow, r = i - k * nrow;
        const char* at = P.row[r].ptr + (size_t)D.X[k] * p.esize;
        if (p.bulk)
          cpa4(&D.xl[k][r], reinterpret_cast<const char*>(reinterpret_cast<uintptr_t>(at) & ~uintptr_t(3)));
        else
          D.xl[k][r] = E::global(P.row[r].ptr, D.X[k]);
      }
      if (lane == 0) D.xl_wait = 1;
      __syncwarp();
    }
  }

  // Complete plan_warp's copies of the row logits at the draft tokens (the
  // 4-byte word holding a 16-bit logit is copied, its half taken here).
  // Warp-wide; afterwards logit_at answers those points from the cache.
  __device__ void xl_sync() {
    if (!D.xl_wait) return;
    cpa_wait();
    __syncwarp();
    if (p.bulk) {
      const int nv = D.nv, nrow = D.P.nrows;
      for (int i = lane; i < nv * nrow; i += 32) {
        const int k = i / nrow, r = i - k * nrow;
        if constexpr (DT == MDS_BF16) {
          const uint32_t w = __float_as_uint(D.xl[k][r]);
          const uintptr_t at = reinterpret_cast<uintptr_t>(D.P.row[r].ptr) + (uintptr_t)D.X[k] * 2u;
          D.xl[k][r] = __uint_as_float((at & 2u) ? (w & 0xffff0000u) : (w << 16));
        }
      }
    }
    __syncwarp();
    if (lane == 0) {
      D.xl_wait = 0;
      D.xl_ok = 1;
    }
    __syncwarp();
  }

  // -------------------------------------------------------------- publishing
  __device__ void push(int b, int kind) {
    PT_T0(t_push);
    if (lane == 0) D.P.kind = kind;
    __syncwarp();
    FSeq* g = &reinterpret_cast<FSeq*>(p.seq)[b];
    copy_out(&g->P, &D.P, (int)sizeof(FPass), lane, 32);
    copy_out(&g->W, &D.W, (int)sizeof(FWalk), lane, 32);
    if (lane == 0) __stcg(p.cnt + b, 0u);
    __threadfence();   // every lane's state writes before any publication
    __syncwarp();
    unsigned base = 0u;
    if (lane == 0) base = (unsigned)p.B * (unsigned)p.ns + atomicAdd(&p.ctl[kCtlTail], (unsigned)p.ns);
    base = __shfl_sync(FULLM, base, 0);
    for (int i = lane; i < p.ns; i += 32) {
      const unsigned t = base + (unsigned)i;
      const unsigned slot = t % (unsigned)p.ring_cap;
      if (t >= (unsigned)p.ring_cap) {
        // the slot's previous task must have been taken
        const unsigned long long prev = tag_of(t - (unsigned)p.ring_cap);
        const unsigned long long t0 = now_ns();
        for (int it = 0; ld_acquire(&p.ring_rtag[slot]) != prev; ++it) {
          if (aborted()) break;
          if ((it & 15) == 15 && now_ns() - t0 > kWaitNs) {
            set_abort(MDS_ST_TIMEOUT);
            break;
          }
          __nanosleep(64);
        }
      }
      __stcg(p.ring_pay + slot, ((unsigned)b << 16) | (unsigned)i);
      st_release(&p.ring_tag[slot], tag_of(t));
    }
    __syncwarp();
    PT_ADDW(kPhPush, t_push);
  }

  __device__ void finish(int b, int acc_len) {
    if (lane == 0) {
      __stcg(p.out_accept + b, acc_len);
      __stcg(p.cnt + b, 0u);
      __threadfence();
      atomicAdd(&p.ctl[kCtlDone], 1u);
    }
    __syncwarp();
  }

  // Z decided at the current depth: outputs, then the next depth's pass,
  // the bonus pass, or the end of the sequence.
  __device__ void walk(int b, int Z, float R, float qY, float pIY, int Ydiag) {
    const int j = D.P.j;
    PT_T0(t_walk);
    __syncwarp();
    int next = kNone;
    if (lane == 0) {
      __stcg(p.out_tokens + (size_t)b * (p.L + 1) + j, Z);
      if (p.out_diag) {
        float* dg = p.out_diag + ((size_t)b * (p.L + 1) + j) * 4;
        __stcg(dg + 0, qY);
        __stcg(dg + 1, pIY);
        __stcg(dg + 2, R);
        __stcg(dg + 3, (float)Ydiag);
      }
      unsigned nv = 0u;
      for (int i = 0; i < D.nv; ++i)
        if (D.X[i] == Z) nv |= 1u << D.vbr[i];
      D.W.valid = nv;
      next = nv ? ((j + 1 == p.L) ? kBonus : kStats) : kNone;
      if (nv) {
        D.W.stage = 0;
        D.W.zres = 0;
      }
    }
    next = __shfl_sync(FULLM, next, 0);
    __syncwarp();
    // the next depth's pass, planned from the staged tokens of depth j + 1
    if (next != kNone) plan_warp(b, j + 1, D.W.valid, next == kBonus, true, false, D.tk1);
    if (next == kNone)
      finish(b, j);
    else
      push(b, next);
    PT_ADDW(kPhDecWalk, t_walk);
  }

  // -------------------------------------------------------------- stats decision
  // The records of a stats pass into the scratch: per row the slice maxima
  // and sums, and with lists each slice's tau, list length and entries.
  __device__ void finish_row(int r, float Z) {
    if (!(Z > 0.f) || !(Z < kPosInf) || Z != Z) {
      atomicOr(p.status, MDS_ST_NONFINITE);
      Z = 1.f;
    }
    D.P.row[r].invZ = __frcp_rn(Z);
  }

  // Test export: the statistics of the depth's rows (M, 1/Z, c, source:
  // the target row's branch, or 100 + the branch whose draft row it is).
  __device__ void debug_rows(int b, int j, int R) const {
    for (int r = lane; r < R && r < MDS_DEBUG_ROWS; r += 32) {
      int src = __ffs(D.W.valid) - 1;
      if (r > 0) {
        src = -1;
        for (int i = 0; i < D.nv; ++i)
          if (D.vrow[i] == r) {
            src = 100 + D.vbr[i];
            break;
          }
      }
      float* o = p.dbg_rows + (((size_t)b * (p.L + 1) + j) * MDS_DEBUG_ROWS + r) * 4;
      o[0] = D.P.row[r].M;
      o[1] = D.P.row[r].invZ;
      o[2] = D.P.row[r].c;
      o[3] = (float)src;
    }
    __syncwarp();
  }

  // The combined record of a stats pass (staged in scr; written by the CTA
  // that completed the pass): every row's M and 1/Z and, with candidate
  // lists, the sequence's list, its complement masses and tau.
  __device__ void adopt_combined(int R, bool list) {
    const float* c = reinterpret_cast<const float*>(scr);
    for (int r = lane; r < R; r += 32) {
      D.P.row[r].M = c[kCmbM + r];
      D.P.row[r].invZ = c[kCmbIz + r];
      if (list) D.pc[r] = c[kCmbPc + r];
    }
    if (list) {
      const int LF = p.ln;
      const int n = __float_as_int(c[kCmbN]);
      for (int t = lane; t < n; t += 32) {
        D.cm_id[t] = __float_as_int(c[kCmbHdr + t]);
        D.cm_l0[t] = c[kCmbHdr + LF + t];
        for (int r = 0; r < R; ++r) D.cm_e[r][t] = c[kCmbHdr + (2 + r) * LF + t];
        D.cm_sp[t] = 0;
        D.cm_a[t] = 0.f;
      }
      if (lane == 0) {
        D.n = n;
        D.cand_tau = c[kCmbN + 1];
        D.cand_all = __float_as_int(c[kCmbN + 2]);
        D.cand_q = c[kCmbN + 3];
      }
    }
    __syncwarp();
  }

  // -------------------------------------------------------------- WIS stage on the candidate list
  // One list entry per lane.  Returns false (changing nothing) if
  // the list cannot certify Omega_1: fewer than s entries, or the s-th key
  // not above every key outside the list (each such key is <= its q <= q(tau)).
  __device__ bool wis_stage_list(int A, int Btok, int rb, float u) {
    const int s = min(p.wis_s, p.V);
    const int n = D.n;
    PT_T0(t_sel);
    {
      const float iz0 = D.P.row[0].invZ, izb = D.P.row[rb].invZ;
      const bool have = lane < n;
      float q = 0.f, a = 0.f, bq = 0.f, key = kNegInf;
      if (have) {
        q = __fmul_rn(D.cm_e[0][lane], iz0);
        if (D.cm_sp[lane]) {
          a = D.cm_a[lane];
        } else {
          for (int r = 1; r < D.P.nrows; ++r)
            if (D.P.row[r].gamma != 0.f) a = __fmaf_rn(D.P.row[r].gamma, __fmul_rn(D.cm_e[r][lane], D.P.row[r].invZ), a);
        }
        bq = __fmul_rn(D.cm_e[rb][lane], izb);
        key = __fadd_rn(__fmaf_rn(-a, bq, q), 0.f);   // -0 -> +0: keys compare as floats
      }
      // Omega_1: s rounds of a warp max over order-preserving keys, ties to
      // the smaller token id (the list is in logit order, not id order)
      const int myid = have ? D.cm_id[lane] : 0x7fffffff;
      unsigned kk = have ? ord_key(key) : 0u;
      uint32_t selm = 0u;
      float kth = kNegInf;
      for (int t = 0; t < s; ++t) {
        const unsigned km = __reduce_max_sync(FULLM, kk);
        if (!km) break;
        const int idm = __reduce_min_sync(FULLM, (kk == km) ? myid : 0x7fffffff);
        const uint32_t who = __ballot_sync(FULLM, kk == km && myid == idm);
        const int wl = __ffs(who) - 1;
        selm |= 1u << wl;
        if (lane == wl) kk = 0u;
        kth = ord_val(km);
      }
      const bool sel = (selm >> lane) & 1u;
      const float qout = __fmul_rn(__fmul_rn(D.cand_q, iz0), 1.0001f);
      const bool ok = __popc(selm) == s && (D.cand_all || kth > qout);
      const float ra = warp_sum((have && !sel) ? a : 0.f);
      const float rbm = warp_sum((have && !sel) ? bq : 0.f);
      if (!ok) {
        if (lane == 0) D.fast_ok = 0;
      } else {
        // position in Omega_1 by token id
        int rk = 0;
        for (uint32_t mm = selm; mm; mm &= mm - 1u) rk += (__shfl_sync(FULLM, myid, __ffs(mm) - 1) < myid) ? 1 : 0;
        if (lane >= s && lane < MDS_MAX_S) {
          D.om[lane] = -1;
          D.om_q[lane] = 0.f;
          D.om_a[lane] = 0.f;
          D.om_b[lane] = 0.f;
        }
        if (sel) {
          D.om[rk] = D.cm_id[lane];
          D.om_q[rk] = q;
          D.om_a[rk] = a;
          D.om_b[rk] = bq;
        }
        __syncwarp();
        PT_ADDW(kPhDecSelect, t_sel);
        if (lane == 0) {
          // Omega_2 masses: complement (generic law) + list entries outside Omega_1
          float sa = 0.f;
          for (int r = 1; r < D.P.nrows; ++r)
            if (D.P.row[r].gamma != 0.f) sa = __fmaf_rn(D.P.row[r].gamma, __fmul_rn(D.pc[r], D.P.row[r].invZ), sa);
          const float sb = __fadd_rn(__fmul_rn(D.pc[rb], izb), rbm);
          sa = __fadd_rn(sa, ra);
          D.Y = solve(s, sa, sb, A, Btok, u);
          D.A2 = sa;
          D.B2 = sb;
          D.fast_ok = 1;
        }
        __syncwarp();
        const float A2 = D.A2, B2 = D.B2;
        if (sel) {
          D.cm_a[lane] = D.om_x[rk];
          D.cm_sp[lane] = 1;
        } else if (have && D.cm_sp[lane]) {
          D.cm_a[lane] = __fmul_rn(0.5f, __fadd_rn(__fmul_rn(a, B2), __fmul_rn(bq, A2)));
        }
        __syncwarp();
        if (lane == 0) gamma_update(rb, A2, B2);
      }
    }
    __syncwarp();
    return D.fast_ok != 0;
  }

  // The stage LP on one thread.  Out of line, so that it has the kernel's
  // whole register budget: s <= 5 keeps its pair state in registers, larger
  // s in shared memory.
  __device__ int solve(int s, float A2, float B2, int A, int Btok, float u) {
    PT_T0(t_lp);
    const int y = (s <= 5) ? lp_solve5(s, A2, B2, A, Btok, u) : lp_solve8(s, A2, B2, A, Btok, u);
    PT_ADDW(kPhLp, t_lp);
    PT_CNTW(kPhLpCalls);
    return y;
  }

  // Generic law after a stage: gamma <- (B2/2) gamma + (A2/2) e_rb.  One thread.
  __device__ void gamma_update(int rb, float A2, float B2) {
    const float hB = __fmul_rn(0.5f, B2), hA = __fmul_rn(0.5f, A2);
    for (int r = 1; r < D.P.nrows; ++r) D.P.row[r].gamma = __fmul_rn(hB, D.P.row[r].gamma);
    D.P.row[rb].gamma = __fadd_rn(D.P.row[rb].gamma, hA);
  }

  // The list's special tokens into the table form used by the residual and
  // the point lookups.  One thread.
  __device__ void list_to_table() {
    int k = 0;
    for (int i = 0; i < D.n && k < kMaxSpecial; ++i)
      if (D.cm_sp[i]) {
        D.P.spec_id[k] = D.cm_id[i];
        D.P.spec_val[k] = D.cm_a[i];
        ++k;
      }
    D.P.nspec = k;
  }

  // -------------------------------------------------------------- decisions per pass kind
  __device__ void accept_step(int b) {
    PT_T0(t_acc);
    int walk_now = 0;
    if (lane == 0) {
      const int j = D.P.j;
      const float u = draw_uniform(p.seed, b, j, kDrawAccept);
      const float ratio = D.W.pIY > 0.f ? __fdiv_rn(D.W.qY, D.W.pIY) : kPosInf;
      const bool acc = u < fminf(1.f, ratio);
      D.W.acc = acc ? 1 : 0;
      D.W.Ydiag = D.W.Y;
      walk_now = (acc && !p.acc_prob) ? 1 : 0;
      if (!walk_now) {
        D.W.ures = acc ? 0.f : draw_uniform(p.seed, b, j, kDrawResidual);
        if (p.scheme == MDS_SINGLE || D.nv == 1 || p.scheme != MDS_WIS) {
          // residual against one draft law: rows 0 and the first valid branch's
          for (int r = 0; r < D.P.nrows; ++r) D.P.row[r].gamma = 0.f;
          D.P.row[D.vrow[0]].gamma = 1.f;
          D.P.nspec = 0;
          D.P.nstream = max(2, D.vrow[0] + 1);
        } else {
          D.P.nstream = D.P.nrows;
        }
      }
    }
    walk_now = __shfl_sync(FULLM, walk_now, 0);
    __syncwarp();
    if (walk_now)
      walk(b, D.W.Y, 0.f, D.W.qY, D.W.pIY, D.W.Y);
    else
      push(b, kResid);
    PT_ADDW(kPhDecAccept, t_acc);
  }

  __device__ void decide_stats(int b, int j, int R, bool list) {
    if (j == 0 && lane == 0) {
      D.W = FWalk{};
      D.W.valid = (p.K >= 32) ? FULLM : ((1u << p.K) - 1u);
      D.W.Yp = -1;
    }
    __syncwarp();
    PT_T0(t_plan);
    plan_warp(b, j, D.W.valid, false, true, true, D.tk0);
    PT_ADDW(kPhDecPlan, t_plan);
    PT_T0(t_comb);
    adopt_combined(R, list);
    if (p.dbg_rows) debug_rows(b, j, R);
    xl_sync();
    PT_ADDW(kPhDecCombine, t_comb);
    if (p.scheme == MDS_WIS0) {
      dec_wis0_nl<DT>(b);
      return;
    }
    if (p.scheme == MDS_SINGLE || D.nv == 1) {
      if (lane == 0) {
        const int Y = D.X[0];
        D.W.Y = Y;
        D.W.qY = prob_row(D.P, 0, Y);
        D.W.pIY = prob_row(D.P, D.vrow[0], Y);
      }
      __syncwarp();
      dec_accept_nl<DT>(b);
      return;
    }
    // WIS: the pairwise stages (Remark 4) on the candidate list while it
    // certifies Omega_1; from the first stage it cannot, full-vocabulary passes
    PT_T0(t_stg);
    if (lane == 0) {
      for (int r = 0; r < D.P.nrows; ++r) D.P.row[r].gamma = 0.f;
      D.P.row[D.vrow[0]].gamma = 1.f;
      D.P.nspec = 0;
    }
    __syncwarp();
    int A = D.X[0];
    int m = 1;
    if (list) {
      // every stage's selection uniform at once (lane m - 1 draws stage m's)
      const float ul = (lane + 1 < D.nv) ? draw_uniform(p.seed, b, j, kDrawSelect + lane) : 0.f;
      for (; m < D.nv; ++m) {
        const float u = __shfl_sync(FULLM, ul, m - 1);
        if (!wis_stage_list(A, D.X[m], D.vrow[m], u)) break;
        A = D.Y;
      }
      if (lane == 0) list_to_table();
    }
    if (lane == 0) {
      D.W.stage = m;
      D.W.A = A;
      if (m < D.nv) {
        D.P.rb = D.vrow[m];
        D.P.nstream = D.P.nrows;
      } else {
        D.W.Y = A;
        D.W.qY = prob_row(D.P, 0, A);
        D.W.pIY = law_at(D.P, A);
      }
    }
    __syncwarp();
    PT_ADDW(kPhDecStages, t_stg);
    if (m < D.nv) {
      push(b, kFull);
      return;
    }
    dec_accept_nl<DT>(b);
  }

  // One full-vocabulary stage's decision: Omega_1 = the top s of the slices'
  // top s (s rounds of a warp argmax), the Omega_2 masses (the slices' rests
  // plus their entries not taken), the LP, the selection and the law update.
  __device__ void decide_full(int b) {
    const int j = D.P.j, ns = p.ns;
    plan_warp(b, j, D.W.valid, false, false, false, D.tk0);
    const int m = D.W.stage;
    const int A = D.W.A, Btok = D.X[m], rb = D.vrow[m];
    const float u = draw_uniform(p.seed, b, j, kDrawSelect + m - 1);
    const int s = min(p.wis_s, p.V);
    const float* recb = p.rec + (size_t)b * ns * p.rec_floats;
    for (int r = 0; r < s; ++r) {
      float bk = kNegInf;
      int bid = 0x7fffffff, bi = -1;
      for (int i = lane; i < ns * kTopF; i += 32) {
        const int sl = i / kTopF, t = i - sl * kTopF;
        if (t >= s) continue;
        const float* rc = recb + (size_t)sl * p.rec_floats;
        const int id = __ldcg(reinterpret_cast<const int*>(rc) + 4 + kTopF + t);
        bool taken = false;
        for (int q = 0; q < r; ++q) taken |= (D.fin[q].id == id);
        if (taken) continue;
        const float key = __ldcg(rc + 4 + t);
        if (id != 0x7fffffff && better(key, id, bk, bid)) {
          bk = key;
          bid = id;
          bi = i;
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        const float ok = __shfl_xor_sync(FULLM, bk, o);
        const int oid = __shfl_xor_sync(FULLM, bid, o);
        const int oi = __shfl_xor_sync(FULLM, bi, o);
        if (better(ok, oid, bk, bid)) {
          bk = ok;
          bid = oid;
          bi = oi;
        }
      }
      if (lane == 0) {
        Cand c = CAND_NONE;
        if (bi >= 0) {
          const float* rc = recb + (size_t)(bi / kTopF) * p.rec_floats;
          const int t = bi % kTopF;
          c = Cand{bk, bid, __ldcg(rc + 4 + 2 * kTopF + t), __ldcg(rc + 4 + 3 * kTopF + t)};
        }
        D.fin[r] = c;
      }
      __syncwarp();
    }
    // Omega_2 masses: the slices' rests plus their top-s entries not taken
    float sa = 0.f, sb = 0.f;
    for (int i = lane; i < ns * kTopF; i += 32) {
      const int sl = i / kTopF, t = i - sl * kTopF;
      const float* rc = recb + (size_t)sl * p.rec_floats;
      if (t == 0) {
        sa = __fadd_rn(sa, __ldcg(rc + 0));
        sb = __fadd_rn(sb, __ldcg(rc + 1));
      }
      if (t >= s) continue;
      const int id = __ldcg(reinterpret_cast<const int*>(rc) + 4 + kTopF + t);
      if (id == 0x7fffffff) continue;
      bool taken = false;
      for (int q = 0; q < s; ++q) taken |= (D.fin[q].id == id);
      if (taken) continue;
      sa = __fadd_rn(sa, __ldcg(rc + 4 + 2 * kTopF + t));
      sb = __fadd_rn(sb, __ldcg(rc + 4 + 3 * kTopF + t));
    }
    const float ra = warp_sum(sa), rbs = warp_sum(sb);
    if (lane < s) {
      int id = D.fin[lane].id;
      if (id < 0 || id >= p.V) id = 0;   // only with non-finite keys (status already set)
      D.fin[lane].id = id;
      D.om_q[lane] = prob_row(D.P, 0, id);
    }
    __syncwarp();
    if (lane == 0) {
      // Omega_1 by token id; q follows its token
      int om[MDS_MAX_S];
      float ak[MDS_MAX_S], bk[MDS_MAX_S], qk[MDS_MAX_S];
      for (int t = 0; t < MDS_MAX_S; ++t) {
        om[t] = (t < s) ? D.fin[t].id : 0x7fffffff;
        ak[t] = (t < s) ? D.fin[t].a : 0.f;
        bk[t] = (t < s) ? D.fin[t].b : 0.f;
        qk[t] = (t < s) ? D.om_q[t] : 0.f;
      }
      for (int x = 1; x < MDS_MAX_S; ++x)   // insertion sort by id (at most 8 entries)
        for (int y = x; y > 0 && om[y] < om[y - 1]; --y) {
          const int ti = om[y];
          om[y] = om[y - 1];
          om[y - 1] = ti;
          float tf = ak[y];
          ak[y] = ak[y - 1];
          ak[y - 1] = tf;
          tf = bk[y];
          bk[y] = bk[y - 1];
          bk[y - 1] = tf;
          tf = qk[y];
          qk[y] = qk[y - 1];
          qk[y - 1] = tf;
        }
      for (int t = 0; t < MDS_MAX_S; ++t) {
        D.om[t] = om[t];
        D.om_a[t] = ak[t];
        D.om_b[t] = bk[t];
        D.om_q[t] = qk[t];
      }
      D.Y = solve(s, ra, rbs, A, Btok, u);
      D.A2 = ra;
      D.B2 = rbs;
    }
    __syncwarp();
    // law update: special tokens outside Omega_1, gamma, Omega_1 values
    const float A2 = D.A2, B2 = D.B2;
    for (int i = lane; i < D.P.nspec; i += 32) {
      const int tokn = D.P.spec_id[i];
      bool in1 = false;
      for (int t = 0; t < s; ++t) in1 |= (D.om[t] == tokn);
      if (!in1)
        D.P.spec_val[i] =
            __fmul_rn(0.5f, __fadd_rn(__fmul_rn(D.P.spec_val[i], B2), __fmul_rn(prob_row(D.P, rb, tokn), A2)));
    }
    __syncwarp();
    if (lane == 0) {
      gamma_update(rb, A2, B2);
      for (int t = 0; t < s; ++t) {
        int i = 0;
        while (i < D.P.nspec && D.P.spec_id[i] != D.om[t]) ++i;
        if (i == D.P.nspec && D.P.nspec < kMaxSpecial) {
          D.P.spec_id[i] = D.om[t];
          ++D.P.nspec;
        }
        if (i < kMaxSpecial) D.P.spec_val[i] = D.om_x[t];
      }
      D.W.A = D.Y;
      D.W.stage = m + 1;
      if (m + 1 < D.nv) D.P.rb = D.vrow[m + 1];
    }
    __syncwarp();
    if (m + 1 < D.nv) {
      push(b, kFull);
      return;
    }
    if (lane == 0) {
      const int Y = D.W.A;
      D.W.Y = Y;
      D.W.qY = prob_row(D.P, 0, Y);
      D.W.pIY = law_at(D.P, Y);
    }
    __syncwarp();
    dec_accept_nl<DT>(b);
  }

  // -------------------------------------------------------------- inverse-CDF search
  // Weights of unit u (tokens tok0 + u*VE + e) of a re-read slice, read from
  // global memory: the residual max(0, q - p_I) (kResid), the target mass
  // outside Omega_0 (kReplace) or the target mass (kBonus); tokens past the
  // slice weigh 0.
  __device__ void weights_g(const FPass& P, int u, int tok0, int n, float* w) const {
    auto load = [&](int r, float* v) {
      const char* row = P.row[r].ptr;
      const int t0 = tok0 + u * VE;
      if (p.aligned && u * VE + VE <= n) {
        E::unit_global(row + (size_t)t0 * p.esize, v);
      } else {
#pragma unroll
        for (int e = 0; e < VE; ++e) v[e] = (u * VE + e < n) ? E::global(row, t0 + e) : kNegInf;
      }
    };
    float v0[VE];
    load(0, v0);
    const float M0 = P.row[0].M, c0 = P.row[0].c, iz0 = P.row[0].invZ;
    if (P.kind == kResid) {
      float a[VE];
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = 0.f;
      for (int r = 1; r < P.nstream; ++r) {
        const float g = P.row[r].gamma;
        if (g == 0.f) continue;
        float v[VE];
        load(r, v);
        const float M = P.row[r].M, c = P.row[r].c, iz = P.row[r].invZ;
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = __fmaf_rn(g, prob_of(v[e], M, c, iz), a[e]);
      }
      if (P.nspec > 0 && ((bm[u >> 5] >> (u & 31)) & 1u)) {
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = spec_lookup(P, tok0 + u * VE + e, a[e]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = fmaxf(0.f, __fsub_rn(prob_of(v0[e], M0, c0, iz0), a[e]));
    } else if (P.kind == kReplace) {
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = (P.all0 || v0[e] > P.cut) ? 0.f : prob_of(v0[e], M0, c0, iz0);
    } else {
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = prob_of(v0[e], M0, c0, iz0);
    }
  }

  // Inclusive warp scan (fixed order) of v over the lanes.
  __device__ __forceinline__ static float scan_incl(float v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(FULLM, v, o);
      if (lane >= o) v = __fadd_rn(v, t);
    }
    return v;
  }

  // The smallest token whose running mass exceeds T, else the last token
  // with positive weight.  Four levels in token order, each a warp scan:
  // the slices (masses Rs[0..ns)), the slice's 32 runs of upl units (masses
  // from its staged record when `runs`, else summed from a re-read), the
  // owning run's units (re-read, one per lane), the owning unit's tokens (in
  // that lane's registers).
  __device__ int search(FPass& P, float T, bool runs) {
    // level 0: slices
    int s = -1, slast = -1;
    float base = 0.f, blast = 0.f;
    {
      float run = 0.f;
      for (int c = 0; c < p.ns && s < 0; c += 32) {
        const int q = c + lane;
        const float v = q < p.ns ? Rs[q] : 0.f;
        const float incl = scan_incl(v, lane);
        const float ex = __fadd_rn(run, __fsub_rn(incl, v));
        const unsigned h = __ballot_sync(FULLM, __fadd_rn(run, incl) > T && v > 0.f);
        const unsigned pz = __ballot_sync(FULLM, v > 0.f);
        if (h) {
          const int l = __ffs(h) - 1;
          s = c + l;
          base = __shfl_sync(FULLM, ex, l);
        } else if (pz) {
          const int l = 31 - __clz(pz);
          slast = c + l;
          blast = __shfl_sync(FULLM, ex, l);
        }
        run = __shfl_sync(FULLM, __fadd_rn(run, incl), 31);
      }
      if (s < 0) {
        s = max(slast, 0);
        base = blast;
      }
    }
    const int tok0 = s * p.T, n = min(p.T, p.V - tok0);
    const int U = (n + VE - 1) / VE;
    if (P.kind == kResid && P.nspec > 0) {
      for (int i = lane; i < 64; i += 32) bm[i] = 0u;
      __syncwarp();
      for (int i = lane; i < P.nspec; i += 32) {
        const int loc = P.spec_id[i] - tok0;
        if (loc >= 0 && loc < n) atomicOr(&bm[(loc / VE) >> 5], 1u << ((loc / VE) & 31));
      }
      __syncwarp();
    }
    // level 1: runs of upl units, one per lane
    const int upl = (U + 31) / 32;
    const int u0 = min(U, lane * upl), u1 = min(U, u0 + upl);
    float part = 0.f;
    if (runs) {
      part = reinterpret_cast<const float*>(scr)[s * p.rec_floats + 4 + lane];
    } else {
      for (int u = u0; u < u1; ++u) {
        float w[VE];
        weights_g(P, u, tok0, n, w);
#pragma unroll
        for (int e = 0; e < VE; ++e) part = __fadd_rn(part, w[e]);
      }
    }
    const float incl = scan_incl(part, lane);
    const float excl = __fadd_rn(base, __fsub_rn(incl, part));
    const unsigned hit1 = __ballot_sync(FULLM, __fadd_rn(base, incl) > T && part > 0.f);
    const unsigned pos1 = __ballot_sync(FULLM, part > 0.f);
    if (!pos1) return tok0;   // no mass in the slice (only by rounding)
    const int own = hit1 ? __ffs(hit1) - 1 : 31 - __clz(pos1);
    // level 2: the owning run's units, one per lane (chunks of 32); level 3
    // in the owning lane
    float run = __shfl_sync(FULLM, excl, own);
    const int v0 = __shfl_sync(FULLM, u0, own), v1 = __shfl_sync(FULLM, u1, own);
    int ulast = -1;
    float ubase_last = 0.f;
    for (int c0 = v0; c0 < v1; c0 += 32) {
      const int u = c0 + lane;
      float w[VE], us = 0.f;
#pragma unroll
      for (int e = 0; e < VE; ++e) w[e] = 0.f;
      if (u < v1) {
        weights_g(P, u, tok0, n, w);
#pragma unroll
        for (int e = 0; e < VE; ++e) us = __fadd_rn(us, w[e]);
      }
      const float ui = scan_incl(us, lane);
      const float uex = __fadd_rn(run, __fsub_rn(ui, us));
      const unsigned h2 = __ballot_sync(FULLM, __fadd_rn(run, ui) > T && us > 0.f);
      const unsigned p2 = __ballot_sync(FULLM, us > 0.f);
      if (h2) {
        const int l2 = __ffs(h2) - 1;
        int tok = 0;
        if (lane == l2) {
          float acc = uex;
          int hit = -1, last = -1;
#pragma unroll
          for (int e = 0; e < VE; ++e) {
            if (w[e] > 0.f) last = e;
            acc = __fadd_rn(acc, w[e]);
            if (hit < 0 && acc > T && w[e] > 0.f) hit = e;
          }
          if (hit < 0) hit = last < 0 ? 0 : last;
          tok = min(tok0 + u * VE + hit, p.V - 1);
        }
        return __shfl_sync(FULLM, tok, l2);
      }
      if (p2) {
        const int l2 = 31 - __clz(p2);
        ulast = c0 + l2;
        ubase_last = __shfl_sync(FULLM, uex, l2);
      }
      run = __shfl_sync(FULLM, __fadd_rn(run, ui), 31);
    }
    // T beyond the run's mass (only by rounding): the last unit with mass
    int tok = tok0;
    if (lane == 0 && ulast >= 0) {
      float w[VE];
      weights_g(P, ulast, tok0, n, w);
      float acc = ubase_last;
      int hit = -1, last = -1;
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        if (w[e] > 0.f) last = e;
        acc = __fadd_rn(acc, w[e]);
        if (hit < 0 && acc > T && w[e] > 0.f) hit = e;
      }
      if (hit < 0) hit = last < 0 ? 0 : last;
      tok = min(tok0 + ulast * VE + hit, p.V - 1);
    }
    return __shfl_sync(FULLM, tok, 0);
  }

  // Slice masses of the pass just completed (Rs) and their total in slice order.
  __device__ float slice_masses(int b) {
    const float* rec = reinterpret_cast<const float*>(scr);
    for (int q = lane; q < p.ns; q += 32) Rs[q] = rec[q * p.rec_floats];
    __syncwarp();
    float R = 0.f;
    if (lane == 0)
      for (int q = 0; q < p.ns; ++q) R = __fadd_rn(R, Rs[q]);
    return __shfl_sync(FULLM, R, 0);
  }

  __device__ void decide_resid(int b) {
    plan_warp(b, D.P.j, D.W.valid, false, false, false, D.tk0);
    const float R = slice_masses(b);
    int Z = D.W.Y;
    if (!D.W.acc) {
      if (R > 0.f) {
        Z = search(D.P, __fmul_rn(D.W.ures, R), true);
      } else {
        // zero residual mass (only by rounding): sample the target row
        if (lane == 0) {
          atomicOr(p.status, MDS_ST_ZERO_RESID);
          D.W.zres = 1;
          D.W.R = R;
          D.P.cut = kPosInf;
          D.P.all0 = 0;
          D.P.nstream = 1;
        }
        __syncwarp();
        push(b, kReplace);
        return;
      }
    }
    walk(b, Z, R, D.W.qY, D.W.pIY, D.W.Ydiag);
  }

  __device__ void decide_replace(int b) {
    plan_warp(b, D.P.j, D.W.valid, false, false, false, D.tk0);
    const float R = slice_masses(b);
    int Z;
    if (R > 0.f) {
      Z = search(D.P, __fmul_rn(D.W.ures, R), true);
    } else if (!D.W.zres && D.W.Yp >= 0) {
      Z = D.W.Yp;   // no target mass outside Omega_0
    } else if (!D.W.zres) {
      if (lane == 0) {
        atomicOr(p.status, MDS_ST_ZERO_RESID);
        D.W.zres = 1;
        D.P.cut = kPosInf;
        D.P.all0 = 0;
      }
      __syncwarp();
      push(b, kReplace);
      return;
    } else {
      if (lane == 0) atomicOr(p.status, MDS_ST_NONFINITE);
      Z = 0;
    }
    const float Rd = (p.scheme == MDS_WIS0) ? D.W.R : (D.W.zres ? D.W.R : R);
    walk(b, Z, Rd, D.W.qY, D.W.pIY, D.W.Ydiag);
  }

  __device__ void decide_bonus(int b) {
    const float* rec = reinterpret_cast<const float*>(scr);
    for (int q = lane; q < p.ns; q += 32) {
      Hm[q] = rec[q * p.rec_floats];
      Rs[q] = rec[q * p.rec_floats + 1];
    }
    __syncwarp();
    if (lane == 0) {
      float M = kNegInf;
      for (int q = 0; q < p.ns; ++q) M = fmaxf(M, Hm[q]);
      if (!(M > kNegInf) || M != M) {
        atomicOr(p.status, MDS_ST_NONFINITE);
        M = 0.f;
      }
      const float c = D.P.row[0].c;
      float Z = 0.f;
      for (int q = 0; q < p.ns; ++q)
        if (Hm[q] > kNegInf) Z = __fadd_rn(Z, __fmul_rn(Rs[q], ref_shift(Hm[q], M, c)));
      D.P.row[0].M = M;
      finish_row(0, Z);
    }
    __syncwarp();
    if (p.dbg_rows && lane == 0) {
      float* o = p.dbg_rows + (((size_t)b * (p.L + 1) + p.L) * MDS_DEBUG_ROWS) * 4;
      o[0] = D.P.row[0].M;
      o[1] = D.P.row[0].invZ;
      o[2] = D.P.row[0].c;
      o[3] = (float)(__ffs(D.W.valid) - 1);
    }
    const float M = D.P.row[0].M, c = D.P.row[0].c, iz = D.P.row[0].invZ;
    for (int q = lane; q < p.ns; q += 32)
      Rs[q] = (Hm[q] > kNegInf) ? __fmul_rn(__fmul_rn(Rs[q], ref_shift(Hm[q], M, c)), iz) : 0.f;
    __syncwarp();
    float Q = 0.f;
    if (lane == 0)
      for (int q = 0; q < p.ns; ++q) Q = __fadd_rn(Q, Rs[q]);
    Q = __shfl_sync(FULLM, Q, 0);
    const int Z = search(D.P, __fmul_rn(draw_uniform(p.seed, b, p.L, kDrawBonus), Q), false);
    if (lane == 0) {
      __stcg(p.out_tokens + (size_t)b * (p.L + 1) + p.L, Z);
      if (p.out_diag) {
        float* dg = p.out_diag + ((size_t)b * (p.L + 1) + p.L) * 4;
        __stcg(dg + 0, 0.f);
        __stcg(dg + 1, 0.f);
        __stcg(dg + 2, Q);
        __stcg(dg + 3, -1.f);
      }
    }
    finish(b, p.L);
  }
  // -------------------------------------------------------------- truncated alphabet
  // Warp-wide inverse CDF over one weight per lane (lane order = token-id
  // order of the list): the smallest lane whose running sum exceeds
  // u * total, the last lane with positive weight if rounding leaves none,
  // -1 if the total is not positive.
  // Inverse CDF over the list entries in token order, two per lane (entry
  // lane and 32 + lane; weights w0, w1): the first entry whose running sum
  // exceeds u01 * total, else the last with positive weight; -1 when the
  // total is 0.  Sums: a warp scan of each half, the halves in order.
  __device__ __forceinline__ int lane_cdf2(float w0, float w1, float u01, float* total) const {
    float c0 = w0, c1 = w1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t0 = __shfl_up_sync(FULLM, c0, o);
      const float t1 = __shfl_up_sync(FULLM, c1, o);
      if (lane >= o) {
        c0 = __fadd_rn(c0, t0);
        c1 = __fadd_rn(c1, t1);
      }
    }
    const float h0 = __shfl_sync(FULLM, c0, 31);
    c1 = __fadd_rn(h0, c1);
    const float tot = __shfl_sync(FULLM, c1, 31);
    *total = tot;
    if (!(tot > 0.f)) return -1;
    const float T = __fmul_rn(u01, tot);
    const unsigned who0 = __ballot_sync(FULLM, c0 > T);
    if (who0) return __ffs(who0) - 1;
    const unsigned who1 = __ballot_sync(FULLM, c1 > T);
    if (who1) return 32 + __ffs(who1) - 1;
    const unsigned p1 = __ballot_sync(FULLM, w1 > 0.f);
    if (p1) return 32 + 31 - __clz(p1);
    return 31 - __clz(__ballot_sync(FULLM, w0 > 0.f));
  }

  // One depth of the truncated-alphabet scheme (Section 4, read with the
  // non-iid appendix's remark on keeping only the inputs in Omega_0).
  // Omega_0 = the target tokens above the (M+1)-th largest target logit, read
  // off the candidate list (exact when the list's (M+1)-th entry is >= tau,
  // the list holds the whole vocabulary, or every token outside it is -inf;
  // otherwise the tokens above tau, with MDS_ST_OMEGA0).  The warp runs the
  // WIS stages on Omega_0 against q~ = q / p_a with the kept inputs' draft
  // laws restricted to Omega_0 and renormalised (point loads of the draft
  // logits there), then Algorithm 1 against q~.  Y' is kept with probability
  // p_a, else a replace pass draws from the tokens outside Omega_0 by q.
  // The list (token-id order, up to 64 entries) sits two entries per lane:
  // entry lane (half 0) and 32 + lane (half 1).
  __device__ void wis0_decide(int b) {
    const int j = D.P.j;
    {
      const int n = D.n;
      bool have[2], in0[2];
      int id[2], rk[2] = {0, 0};
      float l[2], q[2], qt[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int e = lane + 32 * h;
        have[h] = e < n;
        id[h] = have[h] ? D.cm_id[e] : 0;
        l[h] = have[h] ? D.cm_l0[e] : kNegInf;
      }
      // rank in the list by (larger logit, then lower id)
      for (int t = 0; t < n; ++t) {
        const float lt = D.cm_l0[t];
        const int it = D.cm_id[t];
#pragma unroll
        for (int h = 0; h < 2; ++h) rk[h] += better(lt, it, l[h], id[h]) ? 1 : 0;
      }
      const int M = p.omega0;
      const bool all0 = M >= p.V;
      float cut = kNegInf;
      bool cert;
      if (all0) {
        cert = D.cand_all != 0;
      } else {
        const unsigned w0 = __ballot_sync(FULLM, have[0] && rk[0] == M);
        const unsigned w1 = __ballot_sync(FULLM, have[1] && rk[1] == M);
        const bool found = (w0 | w1) != 0u;
        if (w0)
          cut = __shfl_sync(FULLM, l[0], __ffs(w0) - 1);
        else if (w1)
          cut = __shfl_sync(FULLM, l[1], __ffs(w1) - 1);
        const float tau = D.cand_tau;
        cert = D.cand_all || (found ? cut >= tau : !(tau > kNegInf));
        if (!cert) cut = fmaxf(cut, tau);
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        in0[h] = have[h] && (all0 || l[h] > cut);
        q[h] = in0[h] ? prob_of(l[h], D.P.row[0].M, D.P.row[0].c, D.P.row[0].invZ) : 0.f;
      }
      const int n0 = __popc(__ballot_sync(FULLM, in0[0])) + __popc(__ballot_sync(FULLM, in0[1]));
      const float pa = warp_sum(__fadd_rn(q[0], q[1]));
#pragma unroll
      for (int h = 0; h < 2; ++h) qt[h] = (in0[h] && pa > 0.f) ? __fdiv_rn(q[h], pa) : 0.f;
      // draft laws restricted to Omega_0 (exponents against their own maximum
      // there; the rows' full normalisers cancel), per row and entry, in the
      // warp's scratch (the staged records are spent)
      float* ew = reinterpret_cast<float*>(scr);   // [nrows][64]
      for (int r = 1; r < D.P.nrows; ++r) {
        float lr[2], e[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) lr[h] = in0[h] ? E::global(D.P.row[r].ptr, id[h]) : kNegInf;
        const float ref = warp_max(fmaxf(lr[0], lr[1]));
        const float cr = D.P.row[r].c;
#pragma unroll
        for (int h = 0; h < 2; ++h) e[h] = (in0[h] && ref > kNegInf) ? exp_term(lr[h], ref, cr) : 0.f;
        const float Pm = warp_sum(__fadd_rn(e[0], e[1]));
        if (lane == 0 && Pm != Pm) atomicOr(p.status, MDS_ST_NONFINITE);
#pragma unroll
        for (int h = 0; h < 2; ++h) ew[r * 64 + lane + 32 * h] = (Pm > 0.f) ? __fdiv_rn(e[h], Pm) : 0.f;
      }
      __syncwarp();
      // kept inputs: valid branches (branch order) whose token lies in Omega_0
      int nk = 0;
      for (int i = 0; i < D.nv; ++i) {
        const unsigned w0 = __ballot_sync(FULLM, in0[0] && id[0] == D.X[i]);
        const unsigned w1 = __ballot_sync(FULLM, in0[1] && id[1] == D.X[i]);
        if (!(w0 | w1)) continue;
        const int ei = w0 ? __ffs(w0) - 1 : 32 + __ffs(w1) - 1;
        if (!(ew[D.vrow[i] * 64 + ei] > 0.f)) continue;   // impossible draw: dropped
        if (lane == 0) {
          D.k_lane[nk] = ei;
          D.k_row[nk] = D.vrow[i];
        }
        ++nk;
      }
      __syncwarp();
      int yl = -1, Yl = -1;
      float qY = 0.f, pIY = 0.f, R = 0.f;
      if (n0 > 0 && nk == 0) {
        float t;
        yl = lane_cdf2(qt[0], qt[1], draw_uniform(p.seed, b, j, kDrawResidual), &t);
      } else if (n0 > 0) {
        float a[2];
        {
          const float* w = ew + D.k_row[0] * 64;
          a[0] = w[lane];
          a[1] = w[lane + 32];
        }
        int A = D.k_lane[0];
        const int s = min(p.wis_s, n0);
        const unsigned lt = (1u << lane) - 1u;
        for (int m = 1; m < nk; ++m) {
          const int Bl = D.k_lane[m];
          const float* wb = ew + D.k_row[m] * 64;
          const float bb[2] = {wb[lane], wb[lane + 32]};
          const float u = draw_uniform(p.seed, b, j, kDrawSelect + m - 1);
          unsigned kk[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) kk[h] = in0[h] ? ord_key(__fadd_rn(__fmaf_rn(-a[h], bb[h], qt[h]), 0.f)) : 0u;
          // Omega_1: s rounds of the largest key, ties to the smaller id
          // (the lower entry)
          uint32_t sel0 = 0u, sel1 = 0u;
          for (int t = 0; t < s; ++t) {
            const unsigned km = __reduce_max_sync(FULLM, max(kk[0], kk[1]));
            if (!km) break;
            const uint32_t w0 = __ballot_sync(FULLM, kk[0] == km);
            if (w0) {
              const int wl = __ffs(w0) - 1;
              sel0 |= 1u << wl;
              if (lane == wl) kk[0] = 0u;
            } else {
              const int wl = __ffs(__ballot_sync(FULLM, kk[1] == km)) - 1;
              sel1 |= 1u << wl;
              if (lane == wl) kk[1] = 0u;
            }
          }
          const bool sl[2] = {((sel0 >> lane) & 1u) != 0u, ((sel1 >> lane) & 1u) != 0u};
          const int sn = __popc(sel0) + __popc(sel1);
          const float A2 = warp_sum(__fadd_rn((in0[0] && !sl[0]) ? a[0] : 0.f, (in0[1] && !sl[1]) ? a[1] : 0.f));
          const float B2 = warp_sum(__fadd_rn((in0[0] && !sl[0]) ? bb[0] : 0.f, (in0[1] && !sl[1]) ? bb[1] : 0.f));
          const int rk1[2] = {__popc(sel0 & lt), __popc(sel0) + __popc(sel1 & lt)};
          if (lane >= sn && lane < MDS_MAX_S) {
            D.om[lane] = -1;
            D.om_q[lane] = 0.f;
            D.om_a[lane] = 0.f;
            D.om_b[lane] = 0.f;
          }
#pragma unroll
          for (int h = 0; h < 2; ++h)
            if (sl[h]) {
              D.om[rk1[h]] = id[h];
              D.om_q[rk1[h]] = qt[h];
              D.om_a[rk1[h]] = a[h];
              D.om_b[rk1[h]] = bb[h];
            }
          __syncwarp();
          if (lane == 0) D.Y = solve(sn, A2, B2, D.cm_id[A], D.cm_id[Bl], u);
          __syncwarp();
          const int Yt = D.Y;
          const unsigned y0 = __ballot_sync(FULLM, in0[0] && id[0] == Yt);
          const unsigned y1 = __ballot_sync(FULLM, in0[1] && id[1] == Yt);
          A = y0 ? __ffs(y0) - 1 : (y1 ? 32 + __ffs(y1) - 1 : 0);
#pragma unroll
          for (int h = 0; h < 2; ++h)
            a[h] = sl[h] ? D.om_x[rk1[h]]
                         : (in0[h] ? __fmul_rn(0.5f, __fadd_rn(__fmul_rn(a[h], B2), __fmul_rn(bb[h], A2))) : 0.f);
          __syncwarp();
        }
        Yl = A;
        const int Ah = A >> 5, Alane = A & 31;
        qY = __shfl_sync(FULLM, Ah ? qt[1] : qt[0], Alane);
        pIY = __shfl_sync(FULLM, Ah ? a[1] : a[0], Alane);
        const float ratio = pIY > 0.f ? __fdiv_rn(qY, pIY) : kPosInf;
        if (draw_uniform(p.seed, b, j, kDrawAccept) < fminf(1.f, ratio)) {
          yl = A;
        } else {
          const float ures = draw_uniform(p.seed, b, j, kDrawResidual);
          yl = lane_cdf2(in0[0] ? fmaxf(0.f, __fsub_rn(qt[0], a[0])) : 0.f,
                         in0[1] ? fmaxf(0.f, __fsub_rn(qt[1], a[1])) : 0.f, ures, &R);
          if (yl < 0) {   // only by rounding: sample q~
            if (lane == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
            float t;
            yl = lane_cdf2(qt[0], qt[1], ures, &t);
          }
        }
      }
      if (lane == 0) {
        if (!cert) atomicOr(p.status, MDS_ST_OMEGA0);
        D.o0_n = n0;
        D.o0_all = (all0 && D.cand_all) ? 1 : 0;
        D.o0_cut = cut;
        D.o0_pa = pa;
        D.W.R = R;
        D.W.Yp = (yl >= 0) ? D.cm_id[yl] : -1;
        D.W.Ydiag = (Yl >= 0) ? D.cm_id[Yl] : -1;
        D.W.qY = qY;
        D.W.pIY = pIY;
        D.W.zres = 0;
        const bool keep = D.o0_n > 0 && (D.o0_all || draw_uniform(p.seed, b, j, kDrawKeep) < D.o0_pa);
        D.tok = keep ? 1 : 0;
        if (!keep) {
          D.W.ures = draw_uniform(p.seed, b, j, kDrawOutside);
          D.P.cut = cut;
          D.P.all0 = D.o0_all;
          D.P.nstream = 1;
        }
      }
    }
    __syncwarp();
    if (D.tok)
      walk(b, D.W.Yp, D.W.R, D.W.qY, D.W.pIY, D.W.Ydiag);
    else
      push(b, kReplace);
  }

  // -------------------------------------------------------------- one decision
  // Request fields: the sequence, the kind, depth, row count and list flag of
  // the pass that just completed.
  __device__ void decide(int b, int kind, int j, int R, bool list) {
    // One round of asynchronous copies: the sequence's state (a depth-0
    // stats pass has none yet), its draft tokens at depths j and j + 1, its
    // temperatures and the slice records of the pass.
    const int K = p.K, L = p.L;
    PT_T0(t_load);
    if (!(kind == kStats && j == 0)) {
      const int4* src = reinterpret_cast<const int4*>(reinterpret_cast<const FSeq*>(p.seq) + b);
      int4* dst = reinterpret_cast<int4*>(&D.P);
      for (int i = lane; i < (int)(sizeof(FSeq) / 16); i += 32) cpa16(dst + i, src + i);
    }
    if (lane < K) {
      const int32_t* tk = p.tokens + ((size_t)b * K + lane) * L;
      cpa4(&D.tk0[lane], tk + j);
      if (j + 1 < L) cpa4(&D.tk1[lane], tk + j + 1);
    }
    if (lane <= K) cpa4(&D.tmp[lane], p.temps + (size_t)b * (1 + K) + lane);
    {
      const float* recb = p.rec + (size_t)b * p.ns * p.rec_floats;
      const int n16 = p.ns * p.rec_floats / 4;
      for (int i = lane; i < n16; i += 32) cpa16(scr + 16 * i, recb + 4 * i);
    }
    cpa_wait();
    __syncwarp();
    if (lane == 0) {
      D.xl_ok = 0;
      D.xl_wait = 0;
    }
    __syncwarp();
    PT_ADDW(kPhDecLoad, t_load);
    PT_T0(t_dec);
    PT_CNTW(kPhDecisions);
    switch (kind) {
      case kStats: dec_stats_nl<DT>(b, j, R, list); break;
      case kResid: dec_resid_nl<DT>(b); break;
      case kReplace: dec_replace_nl<DT>(b); break;
      case kFull: dec_full_nl<DT>(b); break;
      case kBonus: dec_bonus_nl<DT>(b); break;
      default: break;
    }
    __syncwarp();
    PT_ADDW(kind == kStats ? kPhDecStats
                           : (kind == kFull ? kPhDecFull : (kind == kBonus ? kPhDecBonus : kPhDecResid)),
            t_dec);
  }

  // The decision warp's loop: take request numbers from the decision ring,
  // wait for each request's publication, decide.  Leaves when every sequence
  // is finished (or on an abort).
  __device__ __forceinline__ void loop() {
    for (;;) {
      int have = 0;
      unsigned pay = 0u;
      if (lane == 0 && !aborted()) {
        const unsigned t = atomicAdd(&p.ctl[kCtlDecHead], 1u);
        const unsigned slot = t % (unsigned)p.dec_cap;
        const unsigned long long want = tag_of(t);
        const unsigned long long t0 = now_ns();
        PT_T0(t_poll);
        for (int it = 0;; ++it) {
          if (ld_acquire(&p.dec_tag[slot]) == want) {
            pay = __ldcg(&p.dec_pay[slot]);
            st_release(&p.dec_rtag[slot], want);
            have = 1;
            break;
          }
          if (ld_relaxed(&p.ctl[kCtlDone]) >= (unsigned)p.B || aborted()) break;
          if ((it & 15) == 15 && now_ns() - t0 > kWaitNs) {
            set_abort(MDS_ST_TIMEOUT);
            break;
          }
          __nanosleep(it < 16 ? 32 : 256);
        }
        PT_ADDW(kPhDecPoll, t_poll);
      }
      have = __shfl_sync(FULLM, have, 0);
      pay = __shfl_sync(FULLM, pay, 0);
      if (!have) return;
      const int b = (int)(pay >> 16);
      const int kind = (int)((pay >> 13) & 7u);
      const int j = (int)((pay >> 6) & 127u);
      const int R = (int)((pay >> 1) & 31u);
      const bool list = (pay & 1u) != 0u;
      decide(b, kind, j, R, list);
    }
  }
};


// Shared memory of a CTA, at file scope so that the decision code (out of
// line) addresses it as shared memory: the dynamic buffers, the CTA state and,
// in decision CTAs, a copy of the launch parameters.
extern __shared__ __align__(128) char g_dsm[];
__shared__ FShared g_S;
__shared__ Params g_dp;

constexpr int kDStateBytes = (int)((sizeof(DState) + 127) / 128 * 128);
constexpr int kDecPerWarp = kDStateBytes + (kDecScratch + 127) / 128 * 128;
constexpr int kDynBytes = kNBuf * kBufBytes + 4 * kCandCap * 4;
constexpr int kDecWarps = (kDynBytes / kDecPerWarp < kBlock / 32) ? kDynBytes / kDecPerWarp : kBlock / 32;
static_assert(kDecWarps >= 2, "decision warps per decision CTA");

// The calling warp's decision view: its state and scratch in the CTA's
// dynamic shared memory, the parameters from the CTA's shared copy.
template <int DT>
__device__ __forceinline__ Dec<DT> dec_view() {
  char* base = g_dsm + (size_t)(threadIdx.x >> 5) * kDecPerWarp;
  char* scr = base + kDStateBytes;
  float* rs = reinterpret_cast<float*>(scr + kDecStage);
  return Dec<DT>{g_dp, g_S, *reinterpret_cast<DState*>(base), scr, rs, rs + kMaxSlices,
                 reinterpret_cast<uint32_t*>(rs + 2 * kMaxSlices), (int)(threadIdx.x & 31)};
}
template <int DT> __device__ __noinline__ void dec_stats_nl(int b, int j, int R, bool list) {
  dec_view<DT>().decide_stats(b, j, R, list);
}
template <int DT> __device__ __noinline__ void dec_resid_nl(int b) { dec_view<DT>().decide_resid(b); }
template <int DT> __device__ __noinline__ void dec_replace_nl(int b) { dec_view<DT>().decide_replace(b); }
template <int DT> __device__ __noinline__ void dec_full_nl(int b) { dec_view<DT>().decide_full(b); }
template <int DT> __device__ __noinline__ void dec_bonus_nl(int b) { dec_view<DT>().decide_bonus(b); }
template <int DT> __device__ __noinline__ void dec_wis0_nl(int b) { dec_view<DT>().wis0_decide(b); }
template <int DT> __device__ __noinline__ void dec_accept_nl(int b) { dec_view<DT>().accept_step(b); }

// The stage LP of the calling warp's decision (one lane), on its Omega_1
// tables: pair state in registers for s <= 5, in shared memory above.
__device__ __forceinline__ int lp_solve5(int s, float A2, float B2, int A, int Btok, float u) {
  DState& D = *reinterpret_cast<DState*>(g_dsm + (size_t)(threadIdx.x >> 5) * kDecPerWarp);
  bool capped = false;
  float RS[10], FL[10], FH[10];
  const int y = stage_solve<5>(s, A2, B2, A, Btok, u, D.om, D.om_q, D.om_a, D.om_b, D.om_x, &capped, RS, FL, FH);
  if (capped) atomicOr(g_dp.status, MDS_ST_LP_CAP);
  return y;
}
__device__ __noinline__ int lp_solve8(int s, float A2, float B2, int A, int Btok, float u) {
  DState& D = *reinterpret_cast<DState*>(g_dsm + (size_t)(threadIdx.x >> 5) * kDecPerWarp);
  bool capped = false;
  const int y = stage_solve<MDS_MAX_S>(s, A2, B2, A, Btok, u, D.om, D.om_q, D.om_a, D.om_b, D.om_x, &capped,
                                       D.lp_rs, D.lp_fl, D.lp_fh);
  if (capped) atomicOr(g_dp.status, MDS_ST_LP_CAP);
  return y;
}

// A decision warp's loop, out of line with the whole register budget.
template <int DT>
__device__ __noinline__ void decision_warp() { dec_view<DT>().loop(); }

template <int DT>
__global__ void __launch_bounds__(kBlock, kCtasPerSm) flow_kernel(const __grid_constant__ Params p) {
  char* dsm = g_dsm;
  FShared& S = g_S;
  Eng<DT> e{p, S};
  e.bufs = dsm;
  char* c = dsm + (size_t)kNBuf * kBufBytes;
  e.cid = reinterpret_cast<int*>(c);
  e.cl = reinterpret_cast<float*>(c + kCandCap * 4);
  e.crank = reinterpret_cast<int*>(c + 2 * kCandCap * 4);
  e.cord = reinterpret_cast<int*>(c + 3 * kCandCap * 4);
  if (threadIdx.x == 0) {
    for (int i = 0; i < kNBuf; ++i) {
      mbar_init(&S.full[i], 1);
      mbar_init(&S.empty[i], 1);
    }
    S.issued = 0;
    S.consumed = 0;
    S.ncand = 0;
#ifdef MDS_PHASE_TIMERS
    for (int i = 0; i < kPhaseN; ++i) S.tm[i] = 0ull;
#endif
    mbar_init_fence();
  }
  // Roles: the CTAs on the first dec_sms SMs run decisions (kDecWarps
  // decision warps each, the rest of their warps idle), every other CTA
  // streams slices (one scheduler warp, eight compute warps).  Decisions are
  // serial code: on their own SMs they do not wait behind the streaming warps.
  __shared__ int role;
  if (threadIdx.x == 0) {
    unsigned smid;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
    role = (smid < (unsigned)p.dec_sms) ? 1 : 0;
  }
  __syncthreads();
  PT_T0(t_kernel);
  if (role) {
    // the parameters into shared memory, where the decision code reads them
    static_assert(sizeof(Params) % 4 == 0, "parameter copy in words");
    for (int i = threadIdx.x; i < (int)(sizeof(Params) / 4); i += kBlock)
      reinterpret_cast<int*>(&g_dp)[i] = reinterpret_cast<const int*>(&p)[i];
    __syncthreads();
    const int w = threadIdx.x >> 5;
    if (w < kDecWarps) decision_warp<DT>();
  } else if (threadIdx.x >= kCT) {
    e.scheduler();
  } else {
    e.compute();
  }
  __syncthreads();
  // copies issued but never consumed (only after an abort): wait for them
  if (threadIdx.x == kCT) {
    for (int k = S.consumed; k < S.issued; ++k) (void)e.wait_mbar(&S.full[k % kNBuf], (k / kNBuf) & 1);
  }
  __syncthreads();
#ifdef MDS_PHASE_TIMERS
  if (threadIdx.x == 0) S.tm[kPhKernel] += (unsigned long long)(clock64() - t_kernel);
  __syncthreads();
  if (threadIdx.x < kPhaseN) atomicAdd(&g_phase[threadIdx.x], S.tm[threadIdx.x]);
#endif
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned out = atomicAdd(&p.ctl[kCtlExit], 1u);
    if (out == gridDim.x - 1) {
      // every CTA has left: reset for the next launch
      if (ld_relaxed(&p.ctl[kCtlAbort]))
        for (int b = 0; b < p.B; ++b) p.cnt[b] = 0u;
      p.ctl[kCtlHead] = 0u;
      p.ctl[kCtlTail] = 0u;
      p.ctl[kCtlDecHead] = 0u;
      p.ctl[kCtlDecTail] = 0u;
      p.ctl[kCtlDone] = 0u;
      p.ctl[kCtlAbort] = 0u;
      __threadfence();
      p.ctl[kCtlExit] = 0u;
    }
  }
}

size_t dyn_smem() { return (size_t)kDynBytes; }

}  // namespace

size_t seq_bytes() { return sizeof(FSeq); }

namespace {
size_t up256(size_t x) { return (x + 255) / 256 * 256; }
struct Layout {
  size_t ctl, tag, pay, dtag, dpay, cnt, seq, rec;
  size_t cap, dcap;
};
Layout layout(const Params& p, int nseq, int grid) {
  Layout L;
  L.cap = (size_t)nseq * p.ns + (size_t)grid + 64;
  L.dcap = (size_t)nseq + (size_t)grid * kDecWarps + 64;   // one request per sequence, plus the claims
  L.ctl = 256;
  L.tag = up256(L.cap * 8);
  L.pay = up256(L.cap * 4);
  L.dtag = up256(L.dcap * 8);
  L.dpay = up256(L.dcap * 4);
  L.cnt = up256((size_t)nseq * 4);
  L.seq = up256((size_t)nseq * sizeof(FSeq));
  L.rec = up256((size_t)nseq * p.ns * p.rec_floats * 4);
  return L;
}
}  // namespace

size_t workspace_bytes(const Params& p, int nseq, int grid) {
  const Layout L = layout(p, nseq, grid);
  return L.ctl + 2 * L.tag + L.pay + 2 * L.dtag + L.dpay + L.cnt + L.seq + L.rec;
}

size_t clear_bytes(const Params& p, int nseq, int grid) {
  const Layout L = layout(p, nseq, grid);
  return L.ctl + 2 * L.tag + L.pay + 2 * L.dtag + L.dpay + L.cnt;
}

void carve_workspace(Params& p, char* w, int nseq, int grid) {
  const Layout L = layout(p, nseq, grid);
  p.ctl = reinterpret_cast<unsigned*>(w);
  w += L.ctl;
  p.ring_tag = reinterpret_cast<unsigned long long*>(w);
  w += L.tag;
  p.ring_rtag = reinterpret_cast<unsigned long long*>(w);
  w += L.tag;
  p.ring_pay = reinterpret_cast<unsigned*>(w);
  w += L.pay;
  p.dec_tag = reinterpret_cast<unsigned long long*>(w);
  w += L.dtag;
  p.dec_rtag = reinterpret_cast<unsigned long long*>(w);
  w += L.dtag;
  p.dec_pay = reinterpret_cast<unsigned*>(w);
  w += L.dpay;
  p.cnt = reinterpret_cast<unsigned*>(w);
  w += L.cnt;
  p.seq = w;
  w += L.seq;
  p.rec = reinterpret_cast<float*>(w);
  p.ring_cap = (int)L.cap;
  p.dec_cap = (int)L.dcap;
}

// SMs whose CTAs run the decisions: about a tenth of the grid's SMs, at
// least one and never all of them.  The environment variable MDS_DEC_SMS
// overrides the count (read once per process), for tuning.
int decision_sms(int grid) {
  static const int env = [] {
    const char* e = getenv("MDS_DEC_SMS");
    return e ? atoi(e) : 0;
  }();
  const int sms = grid / kCtasPerSm;
  int d = env > 0 ? env : (sms + 5) / 10;
  if (d < 1) d = 1;
  if (d > sms - 1) d = sms - 1;
  return d;
}

bool plan_geometry(Params& p, int grid) {
  const int es = p.esize;
  int nstream;
  int list = 0;
  if (p.scheme == MDS_WIS0) {
    nstream = 1;
    list = 1;
  } else if (p.scheme == MDS_WIS) {
    nstream = 1 + p.n_models;
    list = (p.K > 1 && nstream <= kListRowsMax) ? 1 : 0;
  } else if (p.scheme == MDS_SINGLE) {
    nstream = 2;
  } else {
    return false;
  }
  if (nstream > kMaxRows) return false;
  int Tmax = kBufBytes / (nstream * es);   // the slice buffer's bound
  Tmax = (Tmax / kSliceQuantum) * kSliceQuantum;
  if (Tmax < kSliceQuantum) return false;
  const int cap = list ? kMaxSlicesList : kMaxSlices;
  int ns = (p.V + Tmax - 1) / Tmax;
  if (ns > cap) return false;
  // enough tasks for the grid: at least two per CTA at depth 0 where the
  // vocabulary allows
  const long want = (2L * grid + p.B - 1) / p.B;
  if (ns < want) {
    const int nsw = (int)(want < cap ? want : cap);
    int T = (p.V + nsw - 1) / nsw;
    T = ((T + kSliceQuantum - 1) / kSliceQuantum) * kSliceQuantum;
    if (T < kSliceQuantum) T = kSliceQuantum;
    if (T > Tmax) T = Tmax;
    ns = (p.V + T - 1) / T;
  }
  p.ln = list ? ((p.scheme == MDS_WIS0 && p.omega0 >= 32) ? 64 : 32) : 0;
  if (p.ln > kListMax) return false;
  const int lrows = list ? nstream : 0;
  // a decision stages a pass's records ([ns][rec_floats]) in its warp's
  // staging area: fewer, longer slices where they would not fit
  const int ns_min = (p.V + Tmax - 1) / Tmax;
  for (;; --ns) {
    if (ns < ns_min) return false;
    int T = (p.V + ns - 1) / ns;
    T = ((T + kSliceQuantum - 1) / kSliceQuantum) * kSliceQuantum;
    if (T > Tmax) return false;
    ns = (p.V + T - 1) / T;
    p.T = T;
    p.ns = ns;
    // a slice's list: enough that the slices' lists together hold the
    // sequence's list whenever its tokens are spread over the slices (a
    // slice holding more of them only shortens the certified list)
    if (list) {
      const int base = (p.scheme == MDS_WIS0) ? 16 : 8;
      int lns = (2 * p.ln + ns - 1) / ns;
      lns = (lns + 7) / 8 * 8;
      p.lns = lns < base ? base : (lns > p.ln ? p.ln : lns);
    } else {
      p.lns = 0;
    }
    int rf = kHdr + p.lns * (1 + lrows);
    if (rf < 4 + 4 * kTopF) rf = 4 + 4 * kTopF;
    // the combined record of a pass is written over the pass's records
    const int cmb = (kCmbHdr + p.ln * (2 + lrows) + ns - 1) / ns;
    if (rf < cmb) rf = cmb;
    p.rec_floats = (rf + 3) & ~3;
    p.hdr_floats = kHdr;
    if ((size_t)ns * p.rec_floats * 4 <= (size_t)kDecStage && ns * p.lns <= kMaxEntries) break;
  }
  p.dec_sms = decision_sms(grid);
  return p.dec_sms > 0;
}

// Every token's probability under given row statistics, by prob_of.
template <int DT>
__global__ void probs_kernel(const char* row, int V, float M, float invZ, float c, float* out) {
  for (int x = blockIdx.x * blockDim.x + threadIdx.x; x < V; x += gridDim.x * blockDim.x)
    out[x] = prob_of(Elt<DT>::global(row, x), M, c, invZ);
}

cudaError_t launch_probs(const void* row, int dtype, int V, float M, float invZ, float c, float* out,
                         cudaStream_t stream) {
  const int blocks = (V + 255) / 256 < 1024 ? (V + 255) / 256 : 1024;
  if (dtype == MDS_BF16)
    probs_kernel<MDS_BF16><<<blocks, 256, 0, stream>>>(static_cast<const char*>(row), V, M, invZ, c, out);
  else
    probs_kernel<MDS_F32><<<blocks, 256, 0, stream>>>(static_cast<const char*>(row), V, M, invZ, c, out);
  return cudaGetLastError();
}

int grid_size(int device) {
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) return 0;
  int per = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, flow_kernel<MDS_BF16>, kBlock, dyn_smem()) != cudaSuccess)
    return 0;
  int per32 = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per32, flow_kernel<MDS_F32>, kBlock, dyn_smem()) != cudaSuccess)
    return 0;
  if (per32 < per) per = per32;
  return per * sms;
}

cudaError_t configure(int) {
  // both logit types: the grid size is taken over both
  cudaError_t e = cudaFuncSetAttribute((const void*)flow_kernel<MDS_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)dyn_smem());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute((const void*)flow_kernel<MDS_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)dyn_smem());
  return e;
}

int read_phase_timers(unsigned long long* out, int n) {
#ifdef MDS_PHASE_TIMERS
  unsigned long long h[kPhaseN];
  if (cudaDeviceSynchronize() != cudaSuccess) return -1;
  if (cudaMemcpyFromSymbol(h, g_phase, sizeof(h)) != cudaSuccess) return -1;
  const unsigned long long z[kPhaseN] = {};
  if (cudaMemcpyToSymbol(g_phase, z, sizeof(z)) != cudaSuccess) return -1;
  const int m = n < kPhaseN ? n : kPhaseN;
  for (int i = 0; i < m; ++i) out[i] = h[i];
  return kPhaseN;
#else
  (void)out;
  (void)n;
  return -2;
#endif
}

cudaError_t launch(const Params& p, int grid, cudaStream_t stream) {
  const size_t smem = dyn_smem();
  if (p.dtype == MDS_F32) {
    flow_kernel<MDS_F32><<<grid, kBlock, smem, stream>>>(p);
  } else {
    flow_kernel<MDS_BF16><<<grid, kBlock, smem, stream>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace flow
}  // namespace mds
