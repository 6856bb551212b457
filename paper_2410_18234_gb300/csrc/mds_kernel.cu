// Batched multi-draft speculative verification on GB300 (sm_103a).
//
// One thread-block cluster verifies one sequence at a time and loops over
// sequences taken from a work counter (a persistent kernel sized to the
// co-resident clusters).  CTA r of the cluster owns tokens
// [r*slice, (r+1)*slice) of every row.  Per depth j of the walk it
//   1. streams its slice of the target row and of one row per distinct draft
//      model through a small shared-memory ring (cp.async.bulk with mbarrier
//      completion), computing the temperature-softmax statistics online and,
//      for the weighted schemes, collecting the candidate tokens; one exchange
//      over distributed shared memory combines the cluster (the truncated
//      alphabet streams the target row only: its draft laws on Omega_0 need
//      no draft normaliser),
//   2. runs the importance step of the selected scheme (Definition 1 /
//      Theorem 1) -- for the weighted scheme on the candidate list alone
//      whenever that list provably holds every stage's Omega_1, for the
//      truncated alphabet on Omega_0 read off the same list (Section 4),
//   3. applies Algorithm 1 (accept with probability min(1, q(Y)/p_I(Y)), else
//      an inverse-CDF draw from max(0, q - p_I) in token order, streaming the
//      rows again, typically from L2), and
//   4. advances the walk: continue while the output is one of the valid draft
//      tokens (Problem 1's event Z in S); after L accepted positions draw the
//      bonus token from the target row at depth L.
// Rows are not kept resident, so shared memory does not bound how many
// sequences are in flight.  Every decision is taken redundantly and
// identically by every CTA of the cluster from cluster-combined values, so
// control flow stays uniform and the cluster barriers always match.  No CTA
// waits on another CTA's flag; the only waits are on this CTA's own bulk
// copies and they are bounded.
#include <cuda_bf16.h>
#include <cooperative_groups.h>

#include "mds_internal.h"

namespace mds {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kNegInf = -__builtin_huge_valf();
constexpr float kPosInf = __builtin_huge_valf();
constexpr int kWarps = kThreads / 32;
constexpr int kTop = 8;                 // per-thread candidate list length (>= MDS_MAX_S)
constexpr int kMaxPairs = MDS_MAX_S * (MDS_MAX_S - 1) / 2;
constexpr int kLpMaxAugment = 4096;
constexpr float kLpEpsRel = 1e-6f;
constexpr long long kWaitLimit = 1ll << 24;
constexpr int kFastRows = 4;            // WIS candidate path: target + up to 3 draft models
constexpr int kWStages = 5;             // stages of each warp's streaming ring
constexpr int kWarpApp = 64;            // candidate tokens one warp can hold during the stats pass
constexpr int kSampleStride = 4;        // the candidate filter's starting threshold samples 1 unit in 4

// Order-preserving map of floats (not NaN) to unsigned; every key is > 0.
__device__ __forceinline__ unsigned ord_key(float f) {
  const unsigned u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord_val(unsigned k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

// ------------------------------------------------------------------ PTX helpers

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t dsmem_addr(const void* local, uint32_t rank) {
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(smem_u32(local)), "r"(rank));
  return ra;
}
__device__ __forceinline__ float ld_dsmem(const float* local, uint32_t rank) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(dsmem_addr(local, rank)) : "memory");
  return v;
}
__device__ __forceinline__ void st_dsmem(int* local, uint32_t rank, int v) {
  asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(dsmem_addr(local, rank)), "r"(v) : "memory");
}
__device__ __forceinline__ void mbar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)));
}
__device__ __forceinline__ void mbar_init_fence() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return done != 0;
}
__device__ __forceinline__ void bulk_copy(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// ---------------------------------------------------------------- Philox4x32-10
// Salmon, Moraes, Dror, Shaw, SC'11: ten rounds of two 32x32->64 products,
// round keys bumped by the Weyl constants.  Returns output word 0.
__device__ __forceinline__ uint32_t philox_w0(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                              uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return c0;
}
__device__ __forceinline__ float draw_uniform(unsigned long long seed, int b, int j, int draw) {
  const uint32_t w = philox_w0((uint32_t)b, (uint32_t)j, (uint32_t)draw, 0u, (uint32_t)seed, (uint32_t)(seed >> 32));
  return (float)(w >> 8) * 0x1p-24f;
}
constexpr int kDrawSelect = 0, kDrawAccept = 16, kDrawResidual = 32, kDrawBonus = 33;
constexpr int kDrawKeep = 34, kDrawOutside = 35;   // truncated alphabet: keep Y', replace it

// ------------------------------------------------------------------ element IO

template <int DT>
struct Elt;
template <>
struct Elt<MDS_F32> {
  static constexpr int VE = 4;  // logits per 16-byte unit
  __device__ static __forceinline__ void unit(const char* row, int u, float* v) {
    const float4 x = *reinterpret_cast<const float4*>(row + 16 * u);
    v[0] = x.x;
    v[1] = x.y;
    v[2] = x.z;
    v[3] = x.w;
  }
  __device__ static __forceinline__ float global(const char* row, int x) {
    return __ldg(reinterpret_cast<const float*>(row) + x);
  }
  __device__ static __forceinline__ void unit_global(const char* at, float* v) {
    const float4 x = __ldg(reinterpret_cast<const float4*>(at));
    v[0] = x.x;
    v[1] = x.y;
    v[2] = x.z;
    v[3] = x.w;
  }
  __device__ static __forceinline__ void unpack(const uint4& x, float* v) {
    v[0] = __uint_as_float(x.x);
    v[1] = __uint_as_float(x.y);
    v[2] = __uint_as_float(x.z);
    v[3] = __uint_as_float(x.w);
  }
};
template <>
struct Elt<MDS_BF16> {
  static constexpr int VE = 8;
  __device__ static __forceinline__ void unit(const char* row, int u, float* v) {
    const uint4 x = *reinterpret_cast<const uint4*>(row + 16 * u);
    v[0] = __uint_as_float(x.x << 16);
    v[1] = __uint_as_float(x.x & 0xffff0000u);
    v[2] = __uint_as_float(x.y << 16);
    v[3] = __uint_as_float(x.y & 0xffff0000u);
    v[4] = __uint_as_float(x.z << 16);
    v[5] = __uint_as_float(x.z & 0xffff0000u);
    v[6] = __uint_as_float(x.w << 16);
    v[7] = __uint_as_float(x.w & 0xffff0000u);
  }
  __device__ static __forceinline__ float global(const char* row, int x) {
    return __uint_as_float((uint32_t)__ldg(reinterpret_cast<const unsigned short*>(row) + x) << 16);
  }
  __device__ static __forceinline__ void unpack(const uint4& x, float* v) {
    v[0] = __uint_as_float(x.x << 16);
    v[1] = __uint_as_float(x.x & 0xffff0000u);
    v[2] = __uint_as_float(x.y << 16);
    v[3] = __uint_as_float(x.y & 0xffff0000u);
    v[4] = __uint_as_float(x.z << 16);
    v[5] = __uint_as_float(x.z & 0xffff0000u);
    v[6] = __uint_as_float(x.w << 16);
    v[7] = __uint_as_float(x.w & 0xffff0000u);
  }
  __device__ static __forceinline__ void unit_global(const char* at, float* v) {
    const uint4 x = __ldg(reinterpret_cast<const uint4*>(at));
    v[0] = __uint_as_float(x.x << 16);
    v[1] = __uint_as_float(x.x & 0xffff0000u);
    v[2] = __uint_as_float(x.y << 16);
    v[3] = __uint_as_float(x.y & 0xffff0000u);
    v[4] = __uint_as_float(x.z << 16);
    v[5] = __uint_as_float(x.z & 0xffff0000u);
    v[6] = __uint_as_float(x.w << 16);
    v[7] = __uint_as_float(x.w & 0xffff0000u);
  }
};

// Probability of a logit under a row's statistics.  The same expression is
// used for in-pass values and point lookups so both give identical bits.
// Exponents: a term is 2^fma(l, c, -round(M c)) (one rounding, l c exact
// inside the FMA); a partial sum moves from reference m to M by the factor
// 2^(round(m c) - round(M c)), so every term of a row shares one reference.
__device__ __forceinline__ float prob_of(float l, float M, float c, float invZ) {
  return __fmul_rn(ex2(__fmaf_rn(l, c, -__fmul_rn(M, c))), invZ);
}

// ------------------------------------------------------------------ shared state

struct Cand {  // candidate for Omega_1: larger key first, then smaller token id
  float key;
  int id;
  float a, b;   // the stage input laws at this token
};
#define CAND_NONE Cand{kNegInf, 0x7fffffff, 0.f, 0.f}
__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

struct State {
  // rows of the current depth
  int nrows;
  int model_row[MDS_MAX_K];   // row index of each (remapped) draft model, -1 if not loaded
  const char* gptr[kMaxRows];
  float M[kMaxRows], c[kMaxRows], invZ[kMaxRows];
  // walk
  int nv;                     // valid branches
  int vbr[MDS_MAX_K];         // valid branch ids, ascending
  int X[MDS_MAX_K];           // their tokens at this depth
  int vrow[MDS_MAX_K];        // row of each valid branch's draft model
  // outcome of the depth
  int Y, accepted;
  float qY, pIY;
  int next_b;
  int Zslot;
  int tok_j[32];
  // cluster exchange (double-buffered) and its gathered copy
  float xch[2][kXch];
  float gat[kMaxCluster * kXch];
  // block reduction scratch
  float red[kWarps * 3 * kMaxRows];
  float wthr[kWarps];        // per warp: bound on the target logits outside its list
  float wtau[kWarps];        // per warp: largest target logit dropped at a merge
  Cand wcand[kWarps * kTop];
  Cand blk[kTop];
  Cand fin[kTop];
  // WIS state: generic coefficient per row, special tokens, current stage
  float gamma[kMaxRows];
  int nspec;
  int spec_id[kMaxSpecial];
  float spec_val[kMaxSpecial];
  int om[MDS_MAX_S];
  float om_x[MDS_MAX_S], om_q[MDS_MAX_S], om_a[MDS_MAX_S], om_b[MDS_MAX_S];
  float lp_rs[kMaxPairs], lp_fl[kMaxPairs], lp_fh[kMaxPairs];
  float A2, B2;
  // WIS candidate list bookkeeping
  float pc[kMaxRows];        // complement exp mass per row
  int ncand, cand_all, fast_ok;
  float cand_q;
  float cand_tau;            // every target logit outside the list is <= cand_tau
  // truncated alphabet: kept inputs (list lane, row) and the depth's outcome
  int k_lane[MDS_MAX_K], k_row[MDS_MAX_K];
  int o0_n, o0_all, o0_Yp;
  float o0_cut, o0_pa, o0_R;
  // SpecTr: inverse residual masses of rejected rounds
  float sp_invR[MDS_MAX_K];
  int sp_rows[MDS_MAX_K];
  // IS: quadrature grid
  int is_mlo, is_n;
  int is_cnt[kMaxRows];
  // CDF search
  int owner, seg;
  float run;
  // streaming: one ring per warp, one mbarrier per stage
  uint64_t wbar[kWarps][kWStages];
  int wapp[kWarps];          // tokens each warp set aside (may exceed kWarpApp: overflow)
  float thr_cta;
};

// ------------------------------------------------------------------ reductions

__device__ __forceinline__ void combine_ms(float& m, float& s, float m2, float s2, float c) {
  const float M = fmaxf(m, m2);
  const float a = (m == kNegInf) ? 0.f : __fmul_rn(s, ex2(__fsub_rn(__fmul_rn(m, c), __fmul_rn(M, c))));
  const float b = (m2 == kNegInf) ? 0.f : __fmul_rn(s2, ex2(__fsub_rn(__fmul_rn(m2, c), __fmul_rn(M, c))));
  m = M;
  s = __fadd_rn(a, b);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Every CTA contributes n floats (S.xch[buf][0..n)); afterwards S.gat[r*n+i]
// holds CTA r's values.  One cluster barrier; the two halves of S.xch
// alternate so a later exchange never overwrites values still being read.
__device__ __forceinline__ void cluster_gather(State& S, int n, int& buf, int cn) {
  __syncthreads();
  if (cn > 1) {
    cluster_sync_all();
    for (int idx = threadIdx.x; idx < cn * n; idx += kThreads) {
      const int r = idx / n, i = idx - r * n;
      S.gat[idx] = ld_dsmem(&S.xch[buf][i], (uint32_t)r);
    }
  } else {
    for (int idx = threadIdx.x; idx < n; idx += kThreads) S.gat[idx] = S.xch[buf][idx];
  }
  __syncthreads();
  buf ^= 1;
}

// Warp-wide merge of per-lane sorted candidate lists (best first, kTop each,
// unused slots CAND_NONE).  Lane 0 writes the warp's best `rounds` entries,
// in order, to out[0..rounds) and CAND_NONE to out[rounds..kTop); the a and b
// masses of every entry not popped are summed (fixed order) into rest_a /
// rest_b on every lane.  Deterministic: ties break on the id.
__device__ void warp_merge(Cand (&top)[kTop], Cand* out, int rounds, float& rest_a, float& rest_b) {
  const int lane = threadIdx.x & 31;
#pragma unroll 1
  for (int t = 0; t < kTop; ++t) {
    if (t >= rounds) {
      if (lane == 0) out[t] = CAND_NONE;
      continue;
    }
    float bk = top[0].key;
    int bid = top[0].id;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float ok = __shfl_xor_sync(0xffffffffu, bk, o);
      const int oid = __shfl_xor_sync(0xffffffffu, bid, o);
      if (better(ok, oid, bk, bid)) {
        bk = ok;
        bid = oid;
      }
    }
    const bool mine = (top[0].id == bid && top[0].key == bk && bid != 0x7fffffff);
    const unsigned who = __ballot_sync(0xffffffffu, mine);
    const int src = who ? __ffs(who) - 1 : 0;
    const float wa = __shfl_sync(0xffffffffu, top[0].a, src);
    const float wb = __shfl_sync(0xffffffffu, top[0].b, src);
    if (mine) {
#pragma unroll
      for (int i = 0; i < kTop - 1; ++i) top[i] = top[i + 1];
      top[kTop - 1] = CAND_NONE;
    }
    if (lane == 0) out[t] = who ? Cand{bk, bid, wa, wb} : CAND_NONE;
  }
  float ra = 0.f, rb = 0.f;
#pragma unroll
  for (int i = 0; i < kTop; ++i) {
    ra = __fadd_rn(ra, top[i].a);
    rb = __fadd_rn(rb, top[i].b);
  }
  rest_a = warp_sum(ra);
  rest_b = warp_sum(rb);
}

// Pair {u, v}, u != v, of tokens below SM: its index in the lexicographic
// order of (i, j), i < j < SM.
__host__ __device__ constexpr int pidx(int u, int v, int SM) {
  return (u < v) ? u * (2 * SM - u - 1) / 2 + (v - u - 1) : v * (2 * SM - v - 1) / 2 + (u - v - 1);
}
// Lower token of pair e in that order.
__host__ __device__ constexpr int pidx_lo(int e, int SM) {
  int i = 0, n = SM - 1;
  while (e >= n) {
    e -= n;
    ++i;
    --n;
  }
  return i;
}
static_assert(pidx(0, 1, 8) == 0 && pidx(1, 2, 8) == 7 && pidx(5, 3, 8) == pidx(3, 5, 8) && pidx(6, 7, 8) == 27 &&
                  pidx(3, 4, 5) == 9 && pidx_lo(pidx(3, 6, 8), 8) == 3 && pidx_lo(pidx(2, 4, 5), 5) == 2,
              "pair indexing");

// Insert into a sorted (best first) candidate list; whatever drops out adds
// its a and b to the running Omega_2 masses.
__device__ __forceinline__ void cand_insert(Cand (&top)[kTop], const Cand& c, float& ra, float& rb) {
  if (better(c.key, c.id, top[kTop - 1].key, top[kTop - 1].id)) {
    ra = __fadd_rn(ra, top[kTop - 1].a);
    rb = __fadd_rn(rb, top[kTop - 1].b);
    top[kTop - 1] = c;
#pragma unroll
    for (int t = kTop - 1; t > 0; --t) {
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

// ------------------------------------------------------------------ the kernel

// Unit lu of row r in the current ring stage (rows of the pass in mask order).
template <int DT>
struct StageLoad {
  const char* base;
  uint32_t mask;
  int cb;
  int lu;
  __device__ __forceinline__ void operator()(int r, float* v) const {
    Elt<DT>::unit(base + __popc(mask & ((1u << r) - 1u)) * cb, lu, v);
  }
};
// Unit gu of row r straight from global memory (logits past V read -inf);
// one 16-byte load when the rows are 16-byte aligned and the unit is whole.
template <int DT>
struct GlobalLoad {
  const char* const* gptr;
  int tok0, V, gu;
  bool aligned;
  __device__ __forceinline__ void operator()(int r, float* v) const {
    const int t0 = tok0 + gu * Elt<DT>::VE;
    if (aligned && t0 + Elt<DT>::VE <= V) {
      Elt<DT>::unit_global(gptr[r] + (size_t)t0 * (16 / Elt<DT>::VE), v);
      return;
    }
#pragma unroll
    for (int e = 0; e < Elt<DT>::VE; ++e) v[e] = (t0 + e < V) ? Elt<DT>::global(gptr[r], t0 + e) : kNegInf;
  }
};

template <int DT, int SCHEME>
struct Kernel {
  using E = Elt<DT>;
  static constexpr int VE = E::VE;

  const Params& p;
  State& S;
  char* ring;          // streaming rings: kWarps x kWStages stages
  uint32_t* bitmap;    // one bit per 16-byte unit of this CTA's slice that holds a special token
  float* segsum;       // per-segment residual sums
  float* chksum;       // per-chunk (32 segments) residual sums
  float* segref;       // bonus draw: each segment sum's reference (round(max * c))
  float* isW;          // IS: weights [rows][kIsNodesMax]
  float* isT;          // IS: nodes t_n
  char* cl_base;       // WIS: this CTA's buffered tokens and their logits per row,
                       //      two alternating copies of [cap_cta] ids + [rows][cap_cta] logits
  int* ap_id;          // WIS: tokens each warp set aside during the stats pass ...
  float* ap_l;         //      ... and their logits per row [rows][kWarps * kWarpApp]
  int* cs_id;          // WIS: every CTA's kept tokens (rank order) ...
  float* cs_l;         //      ... their logits [rows][stage]
  float* cs_x;         //      ... and the target's scaled log-ratio
  int* cm_id;          // WIS: the cluster's merged candidates (token order) ...
  float* cm_e;         //      ... exp values per row [rows][cap]
  float* cm_a;         //      ... current law value of special tokens
  int* cm_sp;          //      ... special flag
  int rank, cn, tok0, nvalid, Uv, nseg, nsegv, bm_words;   // nseg: layout (slice); nsegv: written (valid units)
  int xbuf;
  int clbuf;           // which copy of the CTA list the next candidate pass publishes
  uint32_t wphase;     // parity of each stage of this warp's ring
  int bail;            // this warp's ring gave up on a copy: it streams nothing more

  __device__ float prob_row(int r, int x) const {
    return prob_of(E::global(S.gptr[r], x), S.M[r], S.c[r], S.invZ[r]);
  }

  // ---------------------------------------------------------------- streaming engine
  // The CTA's slice is cut into chunks of su units (a multiple of 32, one
  // ring stage) taken round-robin by the warps (warp w: chunks w, w + kWarps,
  // ...), each walked in groups of 32, one unit per lane:
  // fn(gu, valid, L) is called by all 32 lanes together, gu the unit's index
  // in the slice (a group starts at a multiple of 32) and L(r, v) loading
  // unit gu of row r.  With 16-byte aligned rows the rows of `mask` flow
  // through the warp's own ring of kWStages stages (cp.async.bulk issued by
  // lane 0 up to kWStages stages ahead, completion counted on the stage's
  // mbarrier); otherwise (rows not 16-byte aligned, rows in mapped host
  // memory, or a stage too small for a group of every row), units are loaded
  // straight from global memory.  No block barrier is
  // taken inside a pass, nor at its end: a caller synchronises the block
  // before reading what other warps wrote.  Every wait is bounded.
  __device__ __forceinline__ int stage_units(int nrm) const {
    return ((p.ring_bytes / kWarps / kWStages) / (16 * nrm)) & ~31;
  }

  // Issue this warp's k-th stage: chunk c = warp + k * kWarps of su units.
  __device__ __forceinline__ void issue_stage(int k, uint32_t mask, int su) {
    const int warp = threadIdx.x >> 5;
    const int stage = k % kWStages;
    char* dst = ring + (size_t)(warp * kWStages + stage) * (p.ring_bytes / kWarps / kWStages);
    const int cu0 = (warp + k * kWarps) * su;
    const int bytes = (min(cu0 + su, Uv) - cu0) * 16;
    mbar_expect_tx(&S.wbar[warp][stage], (uint32_t)(bytes * __popc(mask)));
    int pos = 0;
    for (int r = 0; r < S.nrows; ++r) {
      if (!(mask >> r & 1u)) continue;
      bulk_copy(dst + pos * su * 16, S.gptr[r] + ((size_t)tok0 + (size_t)cu0 * VE) * p.esize, (uint32_t)bytes,
                &S.wbar[warp][stage]);
      ++pos;
    }
  }

  template <class FN>
  __device__ void stream(uint32_t mask, FN&& fn) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nrm = __popc(mask);
    const int su = stage_units(nrm);
    if (!p.tma_ok || !p.bulk_ok || su < 32) {
      for (int g = warp * 32; g < Uv; g += kWarps * 32) {
        const int gu = g + lane;
        fn(gu, gu < Uv, GlobalLoad<DT>{S.gptr, tok0, p.V, gu, p.tma_ok != 0});
      }
      return;
    }
    const int nchunk = (Uv + su - 1) / su;
    const int nk = (nchunk - warp + kWarps - 1) / kWarps;   // this warp's chunks: warp, warp + kWarps, ...
    if (nk <= 0 || bail) return;
    if (lane == 0) {
      fence_proxy_async();
      for (int k = 0; k < nk && k < kWStages; ++k) issue_stage(k, mask, su);
    }
    __syncwarp();
    for (int k = 0; k < nk; ++k) {
      const int stage = k % kWStages;
      const char* base = ring + (size_t)(warp * kWStages + stage) * (p.ring_bytes / kWarps / kWStages);
      long long spins = 0;
      bool ok = true;
      while (!mbar_try_wait(&S.wbar[warp][stage], (wphase >> stage) & 1u)) {
        if (++spins > kWaitLimit) {
          ok = false;
          break;
        }
      }
      if (!__all_sync(0xffffffffu, ok)) {
        // A copy never landed: flag the launch (every sequence still to be
        // written is then marked -1), issue nothing more from this warp and
        // give the copies already issued one more bounded wait before the
        // warp's ring is left for good.
        if (lane == 0) {
          atomicOr(p.status, MDS_ST_TIMEOUT);
          for (int kk = k; kk < nk && kk < k + kWStages; ++kk) {
            const int st = kk % kWStages;
            for (long long w = 0; w <= kWaitLimit && !mbar_try_wait(&S.wbar[warp][st], (wphase >> st) & 1u); ++w) {
            }
          }
        }
        __syncwarp();
        bail = 1;
        return;
      }
      wphase ^= 1u << stage;
      const int cu0 = (warp + k * kWarps) * su, cu1 = min(cu0 + su, Uv);
      for (int g = cu0; g < cu1; g += 32) {
        const int gu = g + lane;
        fn(gu, gu < cu1, StageLoad<DT>{base, mask, su * 16, g - cu0 + lane});
      }
      __syncwarp();
      if (lane == 0 && k + kWStages < nk) {
        fence_proxy_async();
        issue_stage(k + kWStages, mask, su);
      }
      __syncwarp();
    }
  }

  // ---------------------------------------------------------------- softmax statistics
  // Candidate order: larger target logit first, then smaller token id.
  __device__ __forceinline__ static bool cand_before(float la, int ia, float lb, int ib) {
    return la > lb || (la == lb && ia < ib);
  }

  // Warp-wide: raise `theta` to the kListN-th largest target logit among the
  // warp's set-aside list and the tokens of the current group flagged in
  // `aside` (bisection on order-preserving keys), drop the list entries at
  // or below it (their exp values join the warp's pruned sums: reference
  // max pm, sum ps, both warp-uniform; the reference only grows and every
  // logit of the list is <= the warp's running max of its row) and unflag
  // the group's tokens at or below it.  Fewer than kListN entries remain,
  // so the flagged tokens fit.  Returns the new length.
  template <int R>
  __device__ int prune_warp_list(int napp, float& theta, uint32_t& aside, const float (&v0)[VE], const float (&m)[R],
                                 const float (&cr)[R], float (&pm)[R], float (&ps)[R], int* wa_id, float* wa_l) {
    const int lane = threadIdx.x & 31;
    constexpr int kPer = kWarpApp / 32;
    unsigned lk[kPer], gk[VE];
#pragma unroll
    for (int k = 0; k < kPer; ++k) lk[k] = (k * 32 + lane < napp) ? ord_key(wa_l[k * 32 + lane]) : 0u;
#pragma unroll
    for (int e = 0; e < VE; ++e) gk[e] = ((aside >> e) & 1u) ? ord_key(v0[e]) : 0u;
    // the largest key with at least kListN keys >= it (0: fewer keys); the
    // low 16 bits of a key are zero for bf16 logits
    unsigned t = 0u;
#pragma unroll 1
    for (int bit = 31; bit >= (DT == MDS_BF16 ? 16 : 0); --bit) {
      const unsigned c = t | (1u << bit);
      int cnt = 0;
#pragma unroll
      for (int k = 0; k < kPer; ++k) cnt += (lk[k] >= c) ? 1 : 0;
#pragma unroll
      for (int e = 0; e < VE; ++e) cnt += (gk[e] >= c) ? 1 : 0;
      if (__reduce_add_sync(0xffffffffu, cnt) >= kListN) t = c;
    }
    if (t != 0u) theta = fmaxf(theta, ord_val(t));
    napp = drop_warp_list<R>(napp, theta, m, cr, pm, ps, wa_id, wa_l);
#pragma unroll
    for (int e = 0; e < VE; ++e)
      if (!(v0[e] > theta)) aside &= ~(1u << e);
    return napp;
  }

  // Warp-wide: drop the entries of the warp's list at or below `theta` (their
  // exp values join the pruned sums) and compact the rest in order.
  template <int R>
  __device__ int drop_warp_list(int napp, float theta, const float (&m)[R], const float (&cr)[R], float (&pm)[R],
                                float (&ps)[R], int* wa_id, float* wa_l) {
    const int lane = threadIdx.x & 31;
    constexpr int kPer = kWarpApp / 32;
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float wm = m[r];
#pragma unroll
      for (int o = 16; o; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
      if (wm > pm[r]) {
        ps[r] = (pm[r] == kNegInf) ? 0.f : __fmul_rn(ps[r], ex2(__fsub_rn(__fmul_rn(pm[r], cr[r]), __fmul_rn(wm, cr[r]))));
        pm[r] = wm;
      }
    }
    float add[R];
#pragma unroll
    for (int r = 0; r < R; ++r) add[r] = 0.f;
    int outp = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      // entries move only towards the front: read this slice, then write it
      const int i = k * 32 + lane;
      const bool present = i < napp;
      int id = 0;
      float l[R];
#pragma unroll
      for (int r = 0; r < R; ++r) l[r] = kNegInf;
      if (present) {
        id = wa_id[i];
#pragma unroll
        for (int r = 0; r < R; ++r) l[r] = wa_l[r * kWarps * kWarpApp + i];
      }
      const bool keep = present && l[0] > theta;
      const uint32_t bal = __ballot_sync(0xffffffffu, keep);
      __syncwarp();
      if (keep) {
        const int pos = outp + __popc(bal & ((1u << lane) - 1u));
        wa_id[pos] = id;
#pragma unroll
        for (int r = 0; r < R; ++r) wa_l[r * kWarps * kWarpApp + pos] = l[r];
      } else if (present) {
#pragma unroll
        for (int r = 0; r < R; ++r)
          if (l[r] > kNegInf) add[r] = __fadd_rn(add[r], ex2(__fmaf_rn(l[r], cr[r], -__fmul_rn(pm[r], cr[r]))));
      }
      outp += __popc(bal);
      __syncwarp();
    }
#pragma unroll
    for (int r = 0; r < R; ++r) ps[r] = __fadd_rn(ps[r], warp_sum(add[r]));
    return outp;
  }

  // One streaming pass over rows [r0, r0 + R): per thread an online max and a
  // sum of exp((l - m) c) per row, rescaled once per unit.  With CAND (WIS,
  // R = all rows) the pass also finds the kListN largest target logits of the
  // sequence (ties: smaller token id first), which are kept out of the sums:
  // each warp sets aside every token above `theta`, which starts at the
  // kListN-th largest of the threads' target maxima over a sample and
  // rises to the kListN-th largest target logit the warp holds whenever its
  // list fills; the CTA keeps the first kListN of its warps' lists and the
  // cluster the first kListN of its CTAs' lists.  Every pruned or never
  // set-aside token has a target logit <= tau, the last kept one.  One
  // cluster exchange gives every CTA M and Z of each row, the candidate list
  // (by token id, exp values per row) and the complement's exp mass per row
  // (S.pc), so Omega_2 masses need no 1 - sum.
  template <int R, bool CAND>
  __device__ void stats_pass(int r0) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float m[R], sc[R], cr[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      m[r] = kNegInf;
      sc[r] = 0.f;
      cr[r] = S.c[r0 + r];
    }
    int napp = 0;                       // this warp's set-aside tokens (warp-uniform)
    float pm[R], ps[R];                 // pruned set-aside tokens: reference max and sum (warp-uniform)
#pragma unroll
    for (int r = 0; r < R; ++r) {
      pm[r] = kNegInf;
      ps[r] = 0.f;
    }
    // The filter's starting threshold: the kListN-th largest of the threads'
    // target maxima over a sample of the CTA's slice (one 128-byte line in
    // kSampleStride, plain loads).  Those maxima are kThreads distinct
    // tokens, so the threshold is at most the CTA's kListN-th largest target
    // logit: every token at or below it can be in no list.
    float theta = kNegInf;              // warp-uniform
    if constexpr (CAND) {
      float mx = kNegInf;
      constexpr int kBatch = 16;        // loads in flight per thread
      // sample: 8 consecutive units (one 128-byte line) out of every
      // 8 * kSampleStride, so the sample touches only its own lines
      auto sample_unit = [&](int i) { return (i >> 3) * (8 * kSampleStride) + (i & 7); };
      for (int i0 = threadIdx.x * 8; sample_unit(i0) < Uv; i0 += kThreads * kBatch) {
        if (p.tma_ok) {
          // whole, 16-byte aligned units: raw loads first, then the maxima
          uint4 raw[kBatch];
#pragma unroll
          for (int b = 0; b < kBatch; ++b) {
            const int u = sample_unit(i0 + (b & 7) + (b >> 3) * kThreads * 8);
            raw[b] = (u < Uv) ? __ldg(reinterpret_cast<const uint4*>(S.gptr[r0] + ((size_t)tok0 + (size_t)u * VE) * p.esize))
                              : make_uint4(0u, 0u, 0u, 0u);   // skipped below
          }
#pragma unroll
          for (int b = 0; b < kBatch; ++b) {
            if (sample_unit(i0 + (b & 7) + (b >> 3) * kThreads * 8) >= Uv) continue;
            float v[VE];
            E::unpack(raw[b], v);
#pragma unroll
            for (int e = 0; e < VE; ++e) mx = fmaxf(mx, v[e]);
          }
        } else {
          for (int b = 0; b < kBatch; ++b) {
            const int u = sample_unit(i0 + (b & 7) + (b >> 3) * kThreads * 8);
            if (u >= Uv) continue;
            float v[VE];
            GlobalLoad<DT>{S.gptr, tok0, p.V, u, false}(r0, v);
#pragma unroll
            for (int e = 0; e < VE; ++e) mx = fmaxf(mx, v[e]);
          }
        }
      }
      static_assert(kWarps * 3 * kMaxRows >= kThreads, "scratch for the thread maxima");
      S.red[threadIdx.x] = mx;
      if (threadIdx.x == 0) S.wthr[0] = kNegInf;
      __syncthreads();
      if (mx > kNegInf) {
        int rk = 0;   // rank among the threads' maxima (larger first, then lower thread)
        for (int j = 0; j < kThreads; ++j) {
          const float o = S.red[j];
          rk += (o > mx || (o == mx && j < (int)threadIdx.x)) ? 1 : 0;
        }
        if (rk == kListN - 1) S.wthr[0] = mx;
      }
      __syncthreads();
      theta = S.wthr[0];
      __syncthreads();   // S.red and S.wthr are rewritten after the pass
    }
    int* wa_id = ap_id + warp * kWarpApp;
    float* wa_l = ap_l + warp * kWarpApp;   // row r at wa_l[r * kWarps * kWarpApp + i]
    const uint32_t mask = ((1u << R) - 1u) << r0;
    stream(mask, [&](int gu, bool valid, const auto& L) {
      // row 0 first: its values decide which tokens are set aside
      float v0[VE];
      if (valid) {
        L(r0, v0);
      } else {
#pragma unroll
        for (int e = 0; e < VE; ++e) v0[e] = kNegInf;
      }
      const int t0 = tok0 + gu * VE;
      (void)t0;
      float mu0 = v0[0];
#pragma unroll
      for (int e = 1; e < VE; ++e) mu0 = fmaxf(mu0, v0[e]);
      uint32_t aside = 0u;
      if constexpr (CAND) {
        if (mu0 > theta) {   // only then can a token of the unit pass
#pragma unroll
          for (int e = 0; e < VE; ++e)
            if (t0 + e < p.V && v0[e] > theta) aside |= 1u << e;
        }
      }
      // sums of the tokens not set aside (one rescale per unit and row)
#pragma unroll
      for (int r = 0; r < R; ++r) {
        float v[VE];
        float mu = mu0;
        if (r == 0) {
#pragma unroll
          for (int e = 0; e < VE; ++e) v[e] = v0[e];
        } else {
          if (valid) {
            L(r0 + r, v);
          } else {
#pragma unroll
            for (int e = 0; e < VE; ++e) v[e] = kNegInf;
          }
          mu = v[0];
#pragma unroll
          for (int e = 1; e < VE; ++e) mu = fmaxf(mu, v[e]);
        }
        if (mu > m[r]) {
          sc[r] = (m[r] == kNegInf) ? 0.f : __fmul_rn(sc[r], ex2(__fsub_rn(__fmul_rn(m[r], cr[r]), __fmul_rn(mu, cr[r]))));
          m[r] = mu;
        }
        if (m[r] > kNegInf) {   // exp of -inf is 0; only -inf - -inf must be avoided
          const float mc = __fmul_rn(m[r], cr[r]);
          if (!aside) {
#pragma unroll
            for (int e = 0; e < VE; ++e) sc[r] = __fadd_rn(sc[r], ex2(__fmaf_rn(v[e], cr[r], -mc)));
          } else {
#pragma unroll
            for (int e = 0; e < VE; ++e) {
              const float t = ex2(__fmaf_rn(v[e], cr[r], -mc));
              sc[r] = __fadd_rn(sc[r], ((aside >> e) & 1u) ? 0.f : t);
            }
          }
        }
      }
      if constexpr (CAND) {
        if (__any_sync(0xffffffffu, aside != 0u)) {
          const int nadd = __reduce_add_sync(0xffffffffu, __popc(aside));
          if (napp + nadd > kWarpApp) {
            const uint32_t before = aside;
            napp = prune_warp_list<R>(napp, theta, aside, v0, m, cr, pm, ps, wa_id, wa_l);
            const uint32_t back = before & ~aside;   // unflagged by the raised theta: sum them now
            if (back) {
#pragma unroll
              for (int r = 0; r < R; ++r) {
                float v[VE];
                if (r == 0) {
#pragma unroll
                  for (int e = 0; e < VE; ++e) v[e] = v0[e];
                } else {
                  L(r0 + r, v);
                }
#pragma unroll
                for (int e = 0; e < VE; ++e)
                  if (((back >> e) & 1u) && v[e] > kNegInf)
                    sc[r] = __fadd_rn(sc[r], ex2(__fmaf_rn(v[e], cr[r], -__fmul_rn(m[r], cr[r]))));
              }
            }
          }
          // append in lane order, each lane its flagged tokens in token order;
          // the other rows' logits are re-read from the unit
          const int cnt = __popc(aside);
          int incl = cnt;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
          }
          if (aside) {
            int pos = napp + incl - cnt;
#pragma unroll
            for (int e = 0; e < VE; ++e)
              if ((aside >> e) & 1u) {
                wa_id[pos] = t0 + e;
                wa_l[pos] = v0[e];
                ++pos;
              }
            float vr[VE];
#pragma unroll
            for (int r = 1; r < R; ++r) {
              L(r0 + r, vr);
              int q = napp + incl - cnt;
#pragma unroll
              for (int e = 0; e < VE; ++e)
                if ((aside >> e) & 1u) wa_l[r * kWarps * kWarpApp + q++] = vr[e];
            }
          }
          napp += __shfl_sync(0xffffffffu, incl, 31);
        }
      }
    });
    if constexpr (CAND) {
      __syncwarp();
      if (napp > kListN) {   // at most kListN entries per warp for the CTA merge
        uint32_t none = 0u;
        float nv[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) nv[e] = kNegInf;
        napp = prune_warp_list<R>(napp, theta, none, nv, m, cr, pm, ps, wa_id, wa_l);
      }
    }
    // block: combine (max, sum) per row
#pragma unroll
    for (int r = 0; r < R; ++r) {
      float mm = m[r], ss = sc[r];
      if (CAND && lane == 0) combine_ms(mm, ss, pm[r], ps[r], cr[r]);
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, mm, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, ss, o);
        combine_ms(mm, ss, m2, s2, cr[r]);
      }
      if (lane == 0) {
        S.red[(warp * kMaxRows + r) * 2] = mm;
        S.red[(warp * kMaxRows + r) * 2 + 1] = ss;
      }
    }
    if (CAND && lane == 0) {
      S.wapp[warp] = napp;
      S.wthr[warp] = theta;   // every token of the warp outside its list has a target logit <= theta
    }
    __syncthreads();
    constexpr int nx = CAND ? 3 * R + 2 : 2 * R;
    constexpr int sx = CAND ? 3 : 2;   // exchange stride per row: max, complement sum[, list sum]
    if (threadIdx.x < R) {
      const int r = threadIdx.x;
      float mm = kNegInf, ss = 0.f;
      for (int w = 0; w < kWarps; ++w)
        combine_ms(mm, ss, S.red[(w * kMaxRows + r) * 2], S.red[(w * kMaxRows + r) * 2 + 1], cr[r]);
      S.xch[xbuf][sx * r] = mm;
      S.xch[xbuf][sx * r + 1] = ss;
    }
    if constexpr (CAND) {
      __syncthreads();
      // CTA list: the first kListN of the warps' lists (entry t: warp t / 32,
      // slot t % 32); the others join the CTA's complement sums, the kept ones
      // its list sums (both relative to the CTA's row max)
      float pr_s[R], kp_s[R];
#pragma unroll
      for (int r = 0; r < R; ++r) {
        pr_s[r] = 0.f;
        kp_s[r] = 0.f;
      }
      int* cl_id = reinterpret_cast<int*>(cl_base) + clbuf * kListN * (1 + p.rows_max);
      float* cl_l = reinterpret_cast<float*>(cl_id + kListN);
      float tau_t = kNegInf;   // largest target logit this thread drops
      {
        const int w = threadIdx.x >> 5, slot = threadIdx.x & 31;
        static_assert(kListN == 32 && kWarps * 32 == kThreads, "one warp-list entry per thread");
        if (slot < S.wapp[w]) {
          const int i = w * kWarpApp + slot;
          const float l0 = ap_l[i];
          const int id = ap_id[i];
          int rk = 0;
          for (int w2 = 0; w2 < kWarps; ++w2) {
            const int n2 = S.wapp[w2];
            for (int j = 0; j < n2; ++j)
              rk += cand_before(ap_l[w2 * kWarpApp + j], ap_id[w2 * kWarpApp + j], l0, id) ? 1 : 0;
          }
#pragma unroll
          for (int r = 0; r < R; ++r) {
            const float l = ap_l[r * kWarps * kWarpApp + i];
            const float ev = (l > kNegInf) ? ex2(__fmaf_rn(l, cr[r], -__fmul_rn(S.xch[xbuf][sx * r], cr[r]))) : 0.f;
            if (rk < kListN)
              kp_s[r] = ev;
            else
              pr_s[r] = ev;
          }
          if (rk < kListN) {
            cl_id[rk] = id;
#pragma unroll
            for (int r = 0; r < R; ++r) cl_l[r * kListN + rk] = ap_l[r * kWarps * kWarpApp + i];
          } else {
            tau_t = l0;
          }
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) tau_t = fmaxf(tau_t, __shfl_xor_sync(0xffffffffu, tau_t, o));
      int nk = 0;
      for (int w = 0; w < kWarps; ++w) nk += S.wapp[w];
      nk = min(nk, kListN);
#pragma unroll
      for (int r = 0; r < R; ++r) {
        pr_s[r] = warp_sum(pr_s[r]);
        kp_s[r] = warp_sum(kp_s[r]);
      }
      __syncthreads();   // S.red reads above are done; cl_* written
#pragma unroll
      for (int r = 0; r < R; ++r)
        if (lane == 0) {
          S.red[(warp * kMaxRows + r) * 2] = pr_s[r];
          S.red[(warp * kMaxRows + r) * 2 + 1] = kp_s[r];
        }
      if (lane == 0) S.wtau[warp] = tau_t;
      __syncthreads();
      if (threadIdx.x < R) {
        const int r = threadIdx.x;
        float ss = S.xch[xbuf][sx * r + 1], bs = 0.f;
        for (int w = 0; w < kWarps; ++w) {
          ss = __fadd_rn(ss, S.red[(w * kMaxRows + r) * 2]);
          bs = __fadd_rn(bs, S.red[(w * kMaxRows + r) * 2 + 1]);
        }
        S.xch[xbuf][sx * r + 1] = ss;
        S.xch[xbuf][sx * r + 2] = bs;
      }
      if (threadIdx.x == 0) {
        float tc = kNegInf;
        for (int w = 0; w < kWarps; ++w) tc = fmaxf(tc, fmaxf(S.wthr[w], S.wtau[w]));
        S.xch[xbuf][3 * R] = __int_as_float(nk);
        S.xch[xbuf][3 * R + 1] = tc;   // bound on every target logit of this CTA outside its list
      }
    }
    cluster_gather(S, nx, xbuf, cn);   // also publishes cl_* to the cluster
    // every CTA: M, Z and the complement sum of each row (rank order)
    if (threadIdx.x < R) {
      const int r = threadIdx.x;
      float mm = kNegInf;
      for (int q = 0; q < cn; ++q) mm = fmaxf(mm, S.gat[q * nx + sx * r]);
      float ss = 0.f, zz = 0.f;
      if (mm > kNegInf)
        for (int q = 0; q < cn; ++q) {
          const float mq = S.gat[q * nx + sx * r];
          if (!(mq > kNegInf)) continue;
          const float f = ex2(__fsub_rn(__fmul_rn(mq, cr[r]), __fmul_rn(mm, cr[r])));
          const float sq = S.gat[q * nx + sx * r + 1];
          ss = __fadd_rn(ss, __fmul_rn(sq, f));
          zz = __fadd_rn(zz, __fmul_rn(CAND ? __fadd_rn(sq, S.gat[q * nx + sx * r + 2]) : sq, f));
        }
      if (!(mm > kNegInf) || mm != mm) {
        atomicOr(p.status, MDS_ST_NONFINITE);
        mm = 0.f;
      }
      S.M[r0 + r] = mm;
      S.pc[r0 + r] = ss;
      finish_row(r0 + r, zz);
    }
    if constexpr (!CAND) {
      if (threadIdx.x == 0) S.ncand = -1;
      __syncthreads();
      return;
    } else {
      __syncthreads();
      // stage every CTA's list (rank order)
      int ntot = 0;
      for (int q = 0; q < cn; ++q) ntot += __float_as_int(S.gat[q * nx + 3 * R]);
      {
        int base = 0;
        for (int q = 0; q < cn; ++q) {
          const int c = __float_as_int(S.gat[q * nx + 3 * R]);
          const int* qid = reinterpret_cast<const int*>(cl_base) + clbuf * kListN * (1 + p.rows_max);
          const float* ql = reinterpret_cast<const float*>(qid + kListN);
          for (int i = threadIdx.x; i < c; i += kThreads) {
            if (cn > 1) {
              cs_id[base + i] = __float_as_int(ld_dsmem(reinterpret_cast<const float*>(qid) + i, (uint32_t)q));
              for (int r = 0; r < R; ++r) cs_l[r * p.cand_stage + base + i] = ld_dsmem(ql + r * kListN + i, (uint32_t)q);
            } else {
              cs_id[base + i] = qid[i];
              for (int r = 0; r < R; ++r) cs_l[r * p.cand_stage + base + i] = ql[r * kListN + i];
            }
          }
          base += c;
        }
      }
      __syncthreads();
      // the cluster list: the first kListN staged entries, by token id; the
      // others join the complement.  Ranks first (candidate order), then
      // each kept entry's position among the kept by token id.
      const int n = min(ntot, kListN);
      int* rank = reinterpret_cast<int*>(cs_x);
      for (int i = threadIdx.x; i < ntot; i += kThreads) {
        const float l0 = cs_l[i];
        const int id = cs_id[i];
        int rk = 0;
        for (int j = 0; j < ntot; ++j) rk += cand_before(cs_l[j], cs_id[j], l0, id) ? 1 : 0;
        rank[i] = rk;
      }
      __syncthreads();
      float add[R];
#pragma unroll
      for (int r = 0; r < R; ++r) add[r] = 0.f;
      float tau_t2 = kNegInf;
      for (int i = threadIdx.x; i < ntot; i += kThreads) {
        if (rank[i] < kListN) {
          const int id = cs_id[i];
          int pos = 0;
          for (int j = 0; j < ntot; ++j) pos += (rank[j] < kListN && cs_id[j] < id) ? 1 : 0;
          cm_id[pos] = id;
#pragma unroll
          for (int r = 0; r < R; ++r) {
            const float l = cs_l[r * p.cand_stage + i];
            cm_e[r * p.cand_cap + pos] = (l > kNegInf) ? ex2(__fmaf_rn(l, cr[r], -__fmul_rn(S.M[r0 + r], cr[r]))) : 0.f;
          }
          cm_sp[pos] = 0;
          cm_a[pos] = 0.f;
        } else {
          tau_t2 = fmaxf(tau_t2, cs_l[i]);
#pragma unroll
          for (int r = 0; r < R; ++r) {
            const float l = cs_l[r * p.cand_stage + i];
            if (l > kNegInf) add[r] = __fadd_rn(add[r], ex2(__fmaf_rn(l, cr[r], -__fmul_rn(S.M[r0 + r], cr[r]))));
          }
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) tau_t2 = fmaxf(tau_t2, __shfl_xor_sync(0xffffffffu, tau_t2, o));
      if (lane == 0) S.wtau[warp] = tau_t2;
#pragma unroll
      for (int r = 0; r < R; ++r) {
        add[r] = warp_sum(add[r]);
        if (lane == 0) S.red[warp * R + r] = add[r];
      }
      __syncthreads();
      if (threadIdx.x < R) {
        const int r = threadIdx.x;
        float ss = S.pc[r0 + r];
        for (int w = 0; w < kWarps; ++w) ss = __fadd_rn(ss, S.red[w * R + r]);
        S.pc[r0 + r] = ss;
      }
      if (threadIdx.x == 0) {
        // every token outside the list has a target logit <= tau
        float tau = kNegInf;
        for (int q = 0; q < cn; ++q) tau = fmaxf(tau, S.gat[q * nx + 3 * R + 1]);
        for (int w = 0; w < kWarps; ++w) tau = fmaxf(tau, S.wtau[w]);
        S.ncand = n;
        S.cand_all = (n == p.V) ? 1 : 0;
        S.cand_q = (tau > kNegInf) ? ex2(__fmaf_rn(tau, cr[0], -__fmul_rn(S.M[r0], cr[0]))) : 0.f;
        S.cand_tau = tau;
      }
      clbuf ^= 1;
      __syncthreads();
    }
  }

  __device__ __forceinline__ void finish_row(int r, float Z) {
    if (!(Z > 0.f) || !(Z < kPosInf) || Z != Z) {
      atomicOr(p.status, MDS_ST_NONFINITE);
      Z = 1.f;
    }
    S.invZ[r] = __frcp_rn(Z);
  }

  // Statistics of every row loaded at this depth (candidates for WIS and the
  // truncated alphabet).
  __device__ void depth_stats(bool cand) {
    const int nr = S.nrows;
    if constexpr (SCHEME == MDS_WIS0) {
      // the truncated draft laws p_d 1[Omega_0] / p_d(Omega_0) do not involve
      // the draft rows' normalisers: only the target row is streamed
      if (p.cand_cap > 0) {
        stats_pass<1, true>(0);
        return;
      }
    }
    if (cand && nr <= kFastRows && p.cand_cap > 0) {
      switch (nr) {
        case 2: stats_pass<2, true>(0); return;
        case 3: stats_pass<3, true>(0); return;
        case 4: stats_pass<4, true>(0); return;
        default: break;
      }
    }
    for (int r0 = 0; r0 < nr; r0 += 4) {
      switch (min(4, nr - r0)) {
        case 1: stats_pass<1, false>(r0); break;
        case 2: stats_pass<2, false>(r0); break;
        case 3: stats_pass<3, false>(r0); break;
        default: stats_pass<4, false>(r0); break;
      }
    }
  }

  // ---------------------------------------------------------------- residual / CDF sampling
  // Inverse-CDF draw over this sequence's vocabulary from the nonnegative
  // weights rf(gu, L, r[VE]) in token order: the smallest token whose running
  // sum exceeds u * (total).  A streaming pass over the rows in `mask` forms
  // the sum of every 32-unit segment (lane partial sums, warp inclusive
  // scan); segments are added in order per CTA and CTAs in rank order; the
  // owner CTA re-reads its one segment from global memory and re-walks the
  // same sums.  Returns the token (cluster-uniform) and the total mass.
  template <class RF>
  __device__ int sample_cdf(uint32_t mask, const RF& rf, float u01, float* total) {
    const int lane = threadIdx.x & 31;
    stream(mask, [&](int gu, bool valid, const auto& L) {
      float part = 0.f;
      if (valid) {
        float r[VE];
        rf(gu, L, r);
#pragma unroll
        for (int e = 0; e < VE; ++e) part = __fadd_rn(part, r[e]);
      }
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float t = __shfl_up_sync(0xffffffffu, part, o);
        if (lane >= o) part = __fadd_rn(part, t);
      }
      if (lane == 31) segsum[gu >> 5] = part;   // groups start at multiples of 32 units
    });
    __syncthreads();   // every warp's segment sums
    return cdf_search(rf, u01, total);
  }

  // The search of an inverse-CDF draw once segsum[] holds every segment's
  // weight (this CTA's slice, token order): the smallest token whose running
  // sum exceeds u * (total over the cluster).  rf(gu, L, r) gives the
  // weights of unit gu for the re-walk of the owning segment.
  template <class RF>
  __device__ int cdf_search(const RF& rf, float u01, float* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // chunks of 32 segments: inclusive scans by the warps (their last value
    // is the chunk's sum), chunks added in order by thread 0
    const int nchk = (nsegv + 31) / 32;
    for (int k = warp; k < nchk; k += kWarps) {
      const int g = k * 32 + lane;
      float v = g < nsegv ? segsum[g] : 0.f;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v = __fadd_rn(v, t);
      }
      if (lane == 31) chksum[k] = v;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.f;
      for (int k = 0; k < nchk; ++k) tot = __fadd_rn(tot, chksum[k]);
      S.xch[xbuf][0] = tot;
    }
    cluster_gather(S, 1, xbuf, cn);
    float R = 0.f;
    for (int q = 0; q < cn; ++q) R = __fadd_rn(R, S.gat[q]);
    *total = R;
    if (!(R > 0.f)) return -1;
    const float T = __fmul_rn(u01, R);
    if (threadIdx.x == 0) {
      // owner CTA: first whose cumulative total exceeds T (else the last with mass)
      float run = 0.f;
      int owner = -1, last = -1;
      float run_owner = 0.f, run_last = 0.f;
      for (int q = 0; q < cn; ++q) {
        const float tq = S.gat[q];
        if (tq > 0.f) {
          last = q;
          run_last = run;
        }
        if (owner < 0 && __fadd_rn(run, tq) > T) {
          owner = q;
          run_owner = run;
        }
        run = __fadd_rn(run, tq);
      }
      if (owner < 0) {
        owner = last;
        run_owner = run_last;
      }
      S.owner = owner;
      S.run = run_owner;
    }
    __syncthreads();
    const int owner = S.owner;
    if (rank == owner) {
      if (threadIdx.x == 0) {
        // chunk: the first whose running total exceeds T (else the last with mass)
        float run = S.run;
        int k = -1, klast = -1;
        float run_k = 0.f, run_last = 0.f;
        for (int h = 0; h < nchk; ++h) {
          if (chksum[h] > 0.f) {
            klast = h;
            run_last = run;
          }
          if (k < 0 && __fadd_rn(run, chksum[h]) > T) {
            k = h;
            run_k = run;
          }
          run = __fadd_rn(run, chksum[h]);
        }
        if (k < 0) {
          k = klast;
          run_k = run_last;
        }
        S.seg = k;
        S.run = run_k;
      }
      __syncthreads();
      if (warp == 0) {
        // segment inside the chunk: the same scan as the chunk's sum
        const int k = S.seg;
        const float base = S.run;
        const int g = k * 32 + lane;
        const float sv = (k >= 0 && g < nsegv) ? segsum[g] : 0.f;
        float v = sv;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float t = __shfl_up_sync(0xffffffffu, v, o);
          if (lane >= o) v = __fadd_rn(v, t);
        }
        const float vprev = __shfl_up_sync(0xffffffffu, v, 1);
        const unsigned hit = __ballot_sync(0xffffffffu, __fadd_rn(base, v) > T);
        const unsigned pos = __ballot_sync(0xffffffffu, sv > 0.f);
        const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
        if (lane == l) {
          S.seg = k * 32 + l;
          S.run = (l > 0) ? __fadd_rn(base, vprev) : base;
        }
      }
      __syncthreads();
      if (warp == 0) {
        const int g = S.seg;
        const float base = S.run;
        const int gu = g * 32 + lane;
        float r[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) r[e] = 0.f;
        float part = 0.f;
        if (gu < Uv) {
          rf(gu, GlobalLoad<DT>{S.gptr, tok0, p.V, gu, p.tma_ok != 0}, r);
#pragma unroll
          for (int e = 0; e < VE; ++e) part = __fadd_rn(part, r[e]);
        }
        float P = part;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float t = __shfl_up_sync(0xffffffffu, P, o);
          if (lane >= o) P = __fadd_rn(P, t);
        }
        const float Pprev = __shfl_up_sync(0xffffffffu, P, 1);
        const unsigned hit = __ballot_sync(0xffffffffu, __fadd_rn(base, P) > T);
        const unsigned pos = __ballot_sync(0xffffffffu, part > 0.f);
        const int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
        if (lane == l) {
          float acc = (l > 0) ? __fadd_rn(base, Pprev) : base;
          int e_hit = -1, e_last = -1;
#pragma unroll
          for (int e = 0; e < VE; ++e) {
            if (r[e] > 0.f) e_last = e;
            acc = __fadd_rn(acc, r[e]);
            if (e_hit < 0 && acc > T && r[e] > 0.f) e_hit = e;
          }
          if (e_hit < 0) e_hit = e_last < 0 ? 0 : e_last;
          const int tok = min(tok0 + gu * VE + e_hit, p.V - 1);
          for (int q = 0; q < cn; ++q) {
            if (cn > 1)
              st_dsmem(&S.Zslot, (uint32_t)q, tok);
            else
              S.Zslot = tok;
          }
        }
      }
    }
    if (cn > 1)
      cluster_sync_all();
    else
      __syncthreads();
    const int z = S.Zslot;
    __syncthreads();
    return z;
  }

  // Bonus draw (depth L): one pass over the target row gives its max, its
  // sum and the segment sums of the inverse-CDF draw from q.  Each warp takes
  // every exponent against its own running maximum (a warp-uniform
  // reference), so the same values feed the lane sums and the segment
  // sums; a segment sum keeps its reference and becomes q mass once M and Z
  // are known.
  __device__ int bonus_pass(float u01, float* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const float c = S.c[0];
    float wmax = kNegInf, wref = kNegInf;   // warp-uniform; wref = round(wmax c)
    float sc = 0.f;                         // this lane's sum, relative to wref
    stream(1u, [&](int gu, bool valid, const auto& L) {
      float v[VE];
      if (valid) {
        L(0, v);
      } else {
#pragma unroll
        for (int e = 0; e < VE; ++e) v[e] = kNegInf;
      }
      float wm = v[0];
#pragma unroll
      for (int e = 1; e < VE; ++e) wm = fmaxf(wm, v[e]);
#pragma unroll
      for (int o = 16; o; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
      if (wm > wmax) {
        const float nref = __fmul_rn(wm, c);
        sc = (wmax == kNegInf) ? 0.f : __fmul_rn(sc, ex2(__fsub_rn(wref, nref)));
        wmax = wm;
        wref = nref;
      }
      float part = 0.f;
      if (wmax > kNegInf) {
#pragma unroll
        for (int e = 0; e < VE; ++e) part = __fadd_rn(part, ex2(__fmaf_rn(v[e], c, -wref)));
      }
      sc = __fadd_rn(sc, part);
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float t = __shfl_up_sync(0xffffffffu, part, o);
        if (lane >= o) part = __fadd_rn(part, t);
      }
      if (lane == 31) {
        segsum[gu >> 5] = part;
        segref[gu >> 5] = wref;
      }
    });
    // M and Z: warps (one reference each), then the CTA, then the cluster
    const float ss = warp_sum(sc);
    if (lane == 0) {
      S.red[warp * 2] = wmax;
      S.red[warp * 2 + 1] = ss;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float mm = kNegInf, zz = 0.f;
      for (int w = 0; w < kWarps; ++w) combine_ms(mm, zz, S.red[w * 2], S.red[w * 2 + 1], c);
      S.xch[xbuf][0] = mm;
      S.xch[xbuf][1] = zz;
    }
    cluster_gather(S, 2, xbuf, cn);
    if (threadIdx.x == 0) {
      float mm = kNegInf, zz = 0.f;
      for (int q = 0; q < cn; ++q) combine_ms(mm, zz, S.gat[2 * q], S.gat[2 * q + 1], c);
      if (!(mm > kNegInf) || mm != mm) {
        atomicOr(p.status, MDS_ST_NONFINITE);
        mm = 0.f;
      }
      S.M[0] = mm;
      finish_row(0, zz);
    }
    __syncthreads();
    // segment sums -> q mass
    const float mc = __fmul_rn(S.M[0], c), iz = S.invZ[0];
    for (int g = threadIdx.x; g < nsegv; g += kThreads)
      segsum[g] = (segref[g] > kNegInf) ? __fmul_rn(__fmul_rn(segsum[g], ex2(__fsub_rn(segref[g], mc))), iz) : 0.f;
    __syncthreads();
    return cdf_search(
        [&](int, const auto& L, float* r) {
          float v[VE];
          L(0, v);
#pragma unroll
          for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
        },
        u01, total);
  }

  // ---------------------------------------------------------------- schemes

  // Generic draft-law value a_k = sum_r gamma_r p_r(k) from per-row probabilities.
  __device__ __forceinline__ float generic_a(const float* pr) const {
    float a = 0.f;
    for (int r = 1; r < S.nrows; ++r)
      if (S.gamma[r] != 0.f) a = __fmaf_rn(S.gamma[r], pr[r], a);
    return a;
  }
  __device__ float special_lookup(int tok, float fallback) const {
    for (int i = 0; i < S.nspec; ++i)
      if (S.spec_id[i] == tok) return S.spec_val[i];
    return fallback;
  }
  __device__ float a_at(int tok) const {  // point value of the current stage input law
    float pr[kMaxRows];
    for (int r = 1; r < S.nrows; ++r) pr[r] = (S.gamma[r] != 0.f) ? prob_row(r, tok) : 0.f;
    return special_lookup(tok, generic_a(pr));
  }

  // ---------------------------------------------------------------- WIS: the stage LP
  // Maximum flow of one stage on the pair/token network, in the fixed order
  // (a) direct pass over pairs (i, j), i < j, lexicographically: each gives
  // what it can to token i, then to token j; (b) breadth-first augmenting
  // paths in token space (sources: tokens of pairs with supply left, each
  // with the first such pair; u -> v when pair {u, v} gives flow to u;
  // levels in increasing token order, a token's parent the first frontier
  // token reaching it; the path ends at the first token with demand left);
  // (c) the caller splits leftover pair mass 1/2 - 1/2.  Residuals <= eps
  // count as zero.  SM is the compile-time token capacity (5 covers s <= 5
  // in registers; 8 covers every s); all state lives in registers indexed
  // by compile-time constants.  Single thread.
  template <int SM>
  __device__ __forceinline__ void lp_flow(int s, float (&rd)[SM], float (&RS)[SM * (SM - 1) / 2],
                                          float (&FL)[SM * (SM - 1) / 2], float (&FH)[SM * (SM - 1) / 2], float eps) {
    constexpr int P = SM * (SM - 1) / 2;
#pragma unroll
    for (int i = 0; i < SM; ++i) {
#pragma unroll
      for (int j = i + 1; j < SM; ++j) {
        if (j >= s) continue;
        const int e = pidx(i, j, SM);
        if (RS[e] > eps && rd[i] > eps) {
          const float d = fminf(RS[e], rd[i]);
          FL[e] = __fadd_rn(FL[e], d);
          RS[e] = __fsub_rn(RS[e], d);
          rd[i] = __fsub_rn(rd[i], d);
        }
        if (RS[e] > eps && rd[j] > eps) {
          const float d = fminf(RS[e], rd[j]);
          FH[e] = __fadd_rn(FH[e], d);
          RS[e] = __fsub_rn(RS[e], d);
          rd[j] = __fsub_rn(rd[j], d);
        }
      }
    }
    for (int it = 0; it < kLpMaxAugment; ++it) {
      // demands first: with none left (or, below, no supply left) no
      // augmenting path exists
      uint32_t dm = 0u;
#pragma unroll
      for (int t = 0; t < SM; ++t)
        if (t < s && rd[t] > eps) dm |= 1u << t;
      if (!dm) return;
      // adjacency (u -> v when pair {u,v} gives flow to u), sources
      uint32_t adj[SM];
#pragma unroll
      for (int t = 0; t < SM; ++t) adj[t] = 0u;
      uint32_t srcm = 0u, par = 0u;
      unsigned long long srcp = 0ull;
#pragma unroll
      for (int i = 0; i < SM; ++i) {
#pragma unroll
        for (int j = i + 1; j < SM; ++j) {
          if (j >= s) continue;
          const int e = pidx(i, j, SM);
          if (FL[e] > eps) adj[i] |= 1u << j;
          if (FH[e] > eps) adj[j] |= 1u << i;
          if (RS[e] > eps) {
            if (!(srcm >> i & 1u)) {
              srcm |= 1u << i;
              srcp |= (unsigned long long)e << (5 * i);
            }
            if (!(srcm >> j & 1u)) {
              srcm |= 1u << j;
              srcp |= (unsigned long long)e << (5 * j);
            }
          }
        }
      }
      if (!srcm) return;
      uint32_t visited = srcm, frontier = srcm, hit = srcm & dm;
      for (int level = 0; level < SM && !hit && frontier; ++level) {
        uint32_t nxt = 0u;
#pragma unroll
        for (int u = 0; u < SM; ++u) {
          if (!(frontier >> u & 1u)) continue;
          const uint32_t nb = adj[u] & ~(visited | nxt);
#pragma unroll
          for (int v = 0; v < SM; ++v)
            if (nb >> v & 1u) par |= (uint32_t)(u + 1) << (4 * v);
          nxt |= nb;
        }
        visited |= nxt;
        frontier = nxt;
        hit = nxt & dm;
      }
      if (!hit) return;
      const int sink = __ffs(hit) - 1;
      // bottleneck along the path sink <- ... <- t0
      float delta = 0.f;
#pragma unroll
      for (int k = 0; k < SM; ++k)
        if (k == sink) delta = rd[k];
      int t = sink, t0 = sink;
      for (int g = 0; g < SM; ++g) {
        const int u = (int)((par >> (4 * t)) & 15u) - 1;
        if (u < 0) {
          t0 = t;
          break;
        }
        const int e = pidx(u, t, SM);
        float fl = 0.f;
#pragma unroll
        for (int k = 0; k < P; ++k)
          if (k == e) fl = (u < t) ? FL[k] : FH[k];
        delta = fminf(delta, fl);
        t = u;
      }
      const int e0 = (int)((srcp >> (5 * t0)) & 31ull);
      const bool lo0 = pidx_lo(e0, SM) == t0;
#pragma unroll
      for (int k = 0; k < P; ++k)
        if (k == e0) delta = fminf(delta, RS[k]);
      // push
#pragma unroll
      for (int k = 0; k < P; ++k) {
        if (k == e0) {
          RS[k] = __fsub_rn(RS[k], delta);
          if (lo0)
            FL[k] = __fadd_rn(FL[k], delta);
          else
            FH[k] = __fadd_rn(FH[k], delta);
        }
      }
      t = sink;
      for (int g = 0; g < SM; ++g) {
        const int u = (int)((par >> (4 * t)) & 15u) - 1;
        if (u < 0) break;
        const int e = pidx(u, t, SM);
        const bool ulo = u < t;
#pragma unroll
        for (int k = 0; k < P; ++k) {
          if (k == e) {
            if (ulo) {
              FL[k] = __fsub_rn(FL[k], delta);
              FH[k] = __fadd_rn(FH[k], delta);
            } else {
              FH[k] = __fsub_rn(FH[k], delta);
              FL[k] = __fadd_rn(FL[k], delta);
            }
          }
        }
        t = u;
      }
#pragma unroll
      for (int k = 0; k < SM; ++k)
        if (k == sink) rd[k] = __fsub_rn(rd[k], delta);
    }
    atomicOr(p.status, MDS_ST_LP_CAP);
  }

  // Solve one stage given Omega_1 in S.om (increasing token ids; entries
  // past s ignored) with q, a, b at those tokens in S.om_q / S.om_a / S.om_b
  // and the Omega_2 masses: writes p_I on Omega_1 to S.om_x and returns the
  // stage output for the ordered inputs (A, B) and uniform u.  Single thread.
  // Pair state: registers for SM = 5, the shared LP scratch for SM = 8.
  template <int SM>
  __device__ __forceinline__ int stage_solve_t(int s, float A2, float B2, int A, int Btok, float u) {
    constexpr int P = SM * (SM - 1) / 2;
    if constexpr (SM == 5) {
      float RS[P], FL[P], FH[P];
      return stage_solve_body<SM>(s, A2, B2, A, Btok, u, RS, FL, FH);
    } else {
      static_assert(P == kMaxPairs, "pair state");
      return stage_solve_body<SM>(s, A2, B2, A, Btok, u, S.lp_rs, S.lp_fl, S.lp_fh);
    }
  }

  template <int SM>
  __device__ __forceinline__ int stage_solve_body(int s, float A2, float B2, int A, int Btok, float u,
                                                  float (&RS)[SM * (SM - 1) / 2], float (&FL)[SM * (SM - 1) / 2],
                                                  float (&FH)[SM * (SM - 1) / 2]) {
    float ak[SM], bk[SM], x[SM], rd[SM];
    float eps = 0.f;
#pragma unroll
    for (int t = 0; t < SM; ++t) {
      ak[t] = S.om_a[t];
      bk[t] = S.om_b[t];
      const float qk = S.om_q[t];
      x[t] = __fadd_rn(__fadd_rn(__fmul_rn(ak[t], bk[t]), __fmul_rn(ak[t], B2)), __fmul_rn(bk[t], A2));
      rd[t] = (t < s) ? fmaxf(0.f, __fsub_rn(qk, x[t])) : 0.f;
      if (t < s) eps = __fadd_rn(eps, __fadd_rn(qk, x[t]));
    }
    eps = __fmul_rn(eps, kLpEpsRel);
#pragma unroll
    for (int i = 0; i < SM; ++i) {
#pragma unroll
      for (int j = i + 1; j < SM; ++j) {
        const int e = pidx(i, j, SM);
        RS[e] = (j < s) ? __fadd_rn(__fmul_rn(ak[i], bk[j]), __fmul_rn(ak[j], bk[i])) : 0.f;
        FL[e] = 0.f;
        FH[e] = 0.f;
      }
    }
    lp_flow<SM>(s, rd, RS, FL, FH, eps);
    // p_I on Omega_1: base + flow + half of the pair mass left over
#pragma unroll
    for (int i = 0; i < SM; ++i) {
#pragma unroll
      for (int j = i + 1; j < SM; ++j) {
        if (j >= s) continue;
        const int e = pidx(i, j, SM);
        const float half = __fmul_rn(0.5f, RS[e]);
        x[i] = __fadd_rn(x[i], __fadd_rn(FL[e], half));
        x[j] = __fadd_rn(x[j], __fadd_rn(FH[e], half));
      }
    }
#pragma unroll
    for (int t = 0; t < SM; ++t) S.om_x[t] = x[t];
    // the stage output for the ordered inputs (A, B): only the weight of
    // the pair {A, B} is needed
    if (A == Btok) return A;
    int pa = -1, pb = -1;
#pragma unroll
    for (int t = 0; t < SM; ++t) {
      if (t < s && S.om[t] == A) pa = t;
      if (t < s && S.om[t] == Btok) pb = t;
    }
    if (pa >= 0 && pb >= 0) {
      const int lo = min(pa, pb), hi = max(pa, pb);
      const int e = pidx(lo, hi, SM);
      float fl = 0.f, rs = 0.f, alo = 0.f, ahi = 0.f, blo = 0.f, bhi = 0.f;
#pragma unroll
      for (int k = 0; k < SM * (SM - 1) / 2; ++k)
        if (k == e) {
          fl = FL[k];
          rs = RS[k];
        }
#pragma unroll
      for (int t = 0; t < SM; ++t) {
        if (t == lo) {
          alo = ak[t];
          blo = bk[t];
        }
        if (t == hi) {
          ahi = ak[t];
          bhi = bk[t];
        }
      }
      const float m = __fadd_rn(__fmul_rn(alo, bhi), __fmul_rn(ahi, blo));
      const float wlo = m > 0.f ? __fdiv_rn(__fadd_rn(fl, __fmul_rn(0.5f, rs)), m) : 0.5f;
      const float wa = (pa < pb) ? wlo : __fsub_rn(1.f, wlo);
      return (u < wa) ? A : Btok;
    }
    if (pa >= 0) return A;
    if (pb >= 0) return Btok;
    return (u < 0.5f) ? A : Btok;
  }

  // s > 5 is rare (the paper's runs use s = 5 or 7): keep its larger state
  // out of the inlined hot path.
  __device__ __noinline__ int stage_solve_wide(int s, float A2, float B2, int A, int Btok, float u) {
    return stage_solve_t<MDS_MAX_S>(s, A2, B2, A, Btok, u);
  }
  __device__ __forceinline__ int stage_solve(int s, float A2, float B2, int A, int Btok, float u) {
    return (s <= 5) ? stage_solve_t<5>(s, A2, B2, A, Btok, u) : stage_solve_wide(s, A2, B2, A, Btok, u);
  }

  // Law update shared by both paths: generic coefficients gamma.
  __device__ void gamma_update(int rb, float A2, float B2) {
    const float hB = __fmul_rn(0.5f, B2), hA = __fmul_rn(0.5f, A2);
    for (int r = 1; r < S.nrows; ++r) S.gamma[r] = __fmul_rn(hB, S.gamma[r]);
    S.gamma[rb] = __fadd_rn(S.gamma[rb], hA);
  }

  // Omega_1 = the first s merged entries sorted by id (a and b travel with
  // the ids; past s: id INT_MAX), written to S.om / S.om_a / S.om_b.
  // 19-comparator sorting network for 8 entries.  Single thread.
  __device__ __forceinline__ void omega1_sorted(const Cand* fin, int s) {
    int om[MDS_MAX_S];
    float ak[MDS_MAX_S], bk[MDS_MAX_S];
#pragma unroll
    for (int t = 0; t < MDS_MAX_S; ++t) {
      om[t] = (t < s) ? fin[t].id : 0x7fffffff;
      ak[t] = (t < s) ? fin[t].a : 0.f;
      bk[t] = (t < s) ? fin[t].b : 0.f;
    }
#define MDS_CX(i, j)                 \
  if (om[j] < om[i]) {               \
    const int ti = om[i];            \
    om[i] = om[j];                   \
    om[j] = ti;                      \
    const float ta = ak[i];          \
    ak[i] = ak[j];                   \
    ak[j] = ta;                      \
    const float tb = bk[i];          \
    bk[i] = bk[j];                   \
    bk[j] = tb;                      \
  }
    MDS_CX(0, 2) MDS_CX(1, 3) MDS_CX(4, 6) MDS_CX(5, 7) MDS_CX(0, 4) MDS_CX(1, 5) MDS_CX(2, 6) MDS_CX(3, 7)
    MDS_CX(0, 1) MDS_CX(2, 3) MDS_CX(4, 5) MDS_CX(6, 7) MDS_CX(2, 4) MDS_CX(3, 5) MDS_CX(1, 4) MDS_CX(3, 6)
    MDS_CX(1, 2) MDS_CX(3, 4) MDS_CX(5, 6)
#undef MDS_CX
#pragma unroll
    for (int t = 0; t < MDS_MAX_S; ++t) {
      S.om[t] = om[t];
      S.om_a[t] = ak[t];
      S.om_b[t] = bk[t];
    }
  }

  // ---------------------------------------------------------------- WIS: full-vocabulary stage
  // Used when the candidate list cannot certify Omega_1.  The law lives in
  // S.gamma + the special table + this CTA's bitmap.
  __device__ int wis_stage_full(int A, int Btok, int rb, float u) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int s = min(p.wis_s, p.V);
    Cand top[kTop];
#pragma unroll
    for (int t = 0; t < kTop; ++t) top[t] = CAND_NONE;
    float suma = 0.f, sumb = 0.f;   // masses of tokens dropped from this thread's list
    const int nr = S.nrows;
    uint32_t mask = 1u | (1u << rb);
    for (int r = 1; r < nr; ++r)
      if (S.gamma[r] != 0.f) mask |= 1u << r;
    stream(mask, [&](int gu, bool valid, const auto& L) {
      if (!valid) return;
      const int uu = gu;
      const int tbase = tok0 + uu * VE;
      float q[VE], a[VE], bb[VE];
      {
        float v[VE];
        L(0, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = 0.f;
      for (int r = 1; r < nr; ++r) {
        const float g = S.gamma[r];
        if (g == 0.f && r != rb) continue;
        float v[VE];
        L(r, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float pr = prob_of(v[e], S.M[r], S.c[r], S.invZ[r]);
          if (g != 0.f) a[e] = __fmaf_rn(g, pr, a[e]);
          if (r == rb) bb[e] = pr;
        }
      }
      if ((bitmap[uu >> 5] >> (uu & 31)) & 1u) {   // the unit holds a special token
#pragma unroll
        for (int e = 0; e < VE; ++e) a[e] = special_lookup(tbase + e, a[e]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        if (tbase + e >= p.V) break;
        cand_insert(top, Cand{__fmaf_rn(-a[e], bb[e], q[e]), tbase + e, a[e], bb[e]}, suma, sumb);
      }
    });
    // merge: lanes -> warp -> CTA -> cluster, popping s entries at each level;
    // every entry not popped adds its a and b to the Omega_2 masses
    {
      float ra, rbs;
      warp_merge(top, S.wcand + warp * kTop, s, ra, rbs);
      suma = warp_sum(suma);
      sumb = warp_sum(sumb);
      if (lane == 0) {
        S.red[warp * 2] = __fadd_rn(suma, ra);
        S.red[warp * 2 + 1] = __fadd_rn(sumb, rbs);
      }
    }
    __syncthreads();
    const int nx = 4 * kTop + 2;
    if (warp == 0) {
#pragma unroll
      for (int t = 0; t < kTop; ++t) top[t] = (lane < kWarps) ? S.wcand[lane * kTop + t] : CAND_NONE;
      float ra, rbs;
      warp_merge(top, S.blk, s, ra, rbs);
      __syncwarp();
      if (lane == 0) {
        float sa = ra, sb = rbs;
        for (int w = 0; w < kWarps; ++w) {
          sa = __fadd_rn(sa, S.red[w * 2]);
          sb = __fadd_rn(sb, S.red[w * 2 + 1]);
        }
        for (int t = 0; t < kTop; ++t) {
          S.xch[xbuf][4 * t] = S.blk[t].key;
          S.xch[xbuf][4 * t + 1] = __int_as_float(S.blk[t].id);
          S.xch[xbuf][4 * t + 2] = S.blk[t].a;
          S.xch[xbuf][4 * t + 3] = S.blk[t].b;
        }
        S.xch[xbuf][4 * kTop] = sa;
        S.xch[xbuf][4 * kTop + 1] = sb;
      }
    }
    cluster_gather(S, nx, xbuf, cn);
    if (warp == 0) {
#pragma unroll
      for (int t = 0; t < kTop; ++t) {
        const float* g = &S.gat[lane * nx + 4 * t];
        top[t] = (lane < cn) ? Cand{g[0], __float_as_int(g[1]), g[2], g[3]} : CAND_NONE;
      }
      float ra, rbs;
      warp_merge(top, S.fin, s, ra, rbs);
      // q at Omega_1 (lanes in parallel)
      if (lane < s) {
        int id = S.fin[lane].id;
        if (id < 0 || id >= p.V) id = 0;   // only with non-finite keys (status already set)
        S.fin[lane].id = id;
        S.om_q[lane] = prob_row(0, id);
      }
      __syncwarp();
      if (lane == 0) {
        float sa = 0.f, sb = 0.f;
        for (int q = 0; q < cn; ++q) {
          sa = __fadd_rn(sa, S.gat[q * nx + 4 * kTop]);
          sb = __fadd_rn(sb, S.gat[q * nx + 4 * kTop + 1]);
        }
        sa = __fadd_rn(sa, ra);
        sb = __fadd_rn(sb, rbs);
        // Omega_1 by token id; q follows its token through the sort
        float qf[MDS_MAX_S];
#pragma unroll
        for (int k = 0; k < MDS_MAX_S; ++k) qf[k] = S.om_q[k];
        omega1_sorted(S.fin, s);
#pragma unroll
        for (int t = 0; t < MDS_MAX_S; ++t) {
          float qv = 0.f;
#pragma unroll
          for (int k = 0; k < MDS_MAX_S; ++k)
            if (k < s && S.fin[k].id == S.om[t]) qv = qf[k];
          S.om_q[t] = qv;
        }
        S.Y = stage_solve(s, sa, sb, A, Btok, u);
        S.A2 = sa;
        S.B2 = sb;
      }
      __syncwarp();
      // law update: special tokens outside Omega_1 (lanes), gamma, Omega_1 values
      const float A2 = S.A2, B2 = S.B2;
      for (int i = lane; i < S.nspec; i += 32) {
        const int tokn = S.spec_id[i];
        bool in1 = false;
        for (int t = 0; t < s; ++t) in1 |= (S.om[t] == tokn);
        if (!in1)
          S.spec_val[i] = __fmul_rn(0.5f, __fadd_rn(__fmul_rn(S.spec_val[i], B2), __fmul_rn(prob_row(rb, tokn), A2)));
      }
      __syncwarp();
      if (lane == 0) {
        gamma_update(rb, A2, B2);
        for (int t = 0; t < s; ++t) {
          int i = 0;
          while (i < S.nspec && S.spec_id[i] != S.om[t]) ++i;
          if (i == S.nspec && S.nspec < kMaxSpecial) {
            S.spec_id[i] = S.om[t];
            ++S.nspec;
          }
          if (i < kMaxSpecial) S.spec_val[i] = S.om_x[t];
        }
      }
    }
    __syncthreads();
    if (threadIdx.x < s) {
      const int loc = S.om[threadIdx.x] - tok0;
      if (loc >= 0 && loc < p.slice) atomicOr(&bitmap[(loc / VE) >> 5], 1u << ((loc / VE) & 31));
    }
    __syncthreads();
    return S.Y;
  }

  // One stage on the candidate list (at most 32 entries, by token id), by
  // warp 0 of every CTA, one entry per lane.  Returns false (and changes
  // nothing) if the list cannot certify Omega_1.
  __device__ bool wis_stage_fast(int A, int Btok, int rb, float u) {
    static_assert(kListN <= 32, "one list entry per lane");
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int s = min(p.wis_s, p.V);
    const int n = S.ncand;
    if (warp == 0) {
      const float iz0 = S.invZ[0], izb = S.invZ[rb];
      const bool have = lane < n;
      float q = 0.f, a = 0.f, b = 0.f, key = kNegInf;
      if (have) {
        q = __fmul_rn(cm_e[lane], iz0);
        if (cm_sp[lane]) {
          a = cm_a[lane];
        } else {
          for (int r = 1; r < S.nrows; ++r)
            if (S.gamma[r] != 0.f) a = __fmaf_rn(S.gamma[r], __fmul_rn(cm_e[r * p.cand_cap + lane], S.invZ[r]), a);
        }
        b = __fmul_rn(cm_e[rb * p.cand_cap + lane], izb);
        key = __fadd_rn(__fmaf_rn(-a, b, q), 0.f);   // -0 -> +0: keys compare as floats
      }
      // Omega_1: s rounds of a warp max over order-preserving keys, ties to
      // the lower lane (the lower token id)
      unsigned kk = have ? ord_key(key) : 0u;
      uint32_t selm = 0u;
      float kth = kNegInf;
      for (int t = 0; t < s; ++t) {
        const unsigned km = __reduce_max_sync(0xffffffffu, kk);
        const uint32_t who = __ballot_sync(0xffffffffu, km != 0u && kk == km);
        if (!who) break;
        const int wl = __ffs(who) - 1;
        selm |= 1u << wl;
        if (lane == wl) kk = 0u;
        kth = ord_val(km);
      }
      const bool sel = (selm >> lane) & 1u;
      // certification: s entries, and the s-th key above every key outside
      // the list (each such key is <= its q <= q(tau))
      const float qout = __fmul_rn(__fmul_rn(S.cand_q, iz0), 1.0001f);
      const bool ok = __popc(selm) == s && (S.cand_all || kth > qout);
      const float ra = warp_sum((have && !sel) ? a : 0.f);
      const float rbm = warp_sum((have && !sel) ? b : 0.f);
      if (!ok) {
        if (lane == 0) S.fast_ok = 0;
      } else {
        // Omega_1 by token id = the selected lanes in increasing order
        const int rk = __popc(selm & ((1u << lane) - 1u));
        if (lane >= s && lane < MDS_MAX_S) {   // slots past s are ignored by the solve; keep them defined
          S.om[lane] = -1;
          S.om_q[lane] = 0.f;
          S.om_a[lane] = 0.f;
          S.om_b[lane] = 0.f;
        }
        if (sel) {
          S.om[rk] = cm_id[lane];
          S.om_q[rk] = q;
          S.om_a[rk] = a;
          S.om_b[rk] = b;
        }
        __syncwarp();
        if (lane == 0) {
          // Omega_2 masses: complement (generic law) + list entries outside Omega_1
          float sa = 0.f;
          for (int r = 1; r < S.nrows; ++r)
            if (S.gamma[r] != 0.f) sa = __fmaf_rn(S.gamma[r], __fmul_rn(S.pc[r], S.invZ[r]), sa);
          const float sb = __fadd_rn(__fmul_rn(S.pc[rb], izb), rbm);
          sa = __fadd_rn(sa, ra);
          S.Y = stage_solve(s, sa, sb, A, Btok, u);
          S.A2 = sa;
          S.B2 = sb;
          S.fast_ok = 1;
        }
        __syncwarp();
        // law update on the list: Omega_1 takes its x, other specials mix
        const float A2 = S.A2, B2 = S.B2;
        if (sel) {
          cm_a[lane] = S.om_x[rk];
          cm_sp[lane] = 1;
        } else if (have && cm_sp[lane]) {
          cm_a[lane] = __fmul_rn(0.5f, __fadd_rn(__fmul_rn(a, B2), __fmul_rn(b, A2)));
        }
        __syncwarp();
        if (lane == 0) gamma_update(rb, A2, B2);
      }
    }
    __syncthreads();
    return S.fast_ok != 0;
  }

  // Move the list's special tokens into the table + bitmap form used by the
  // full-vocabulary stages, the residual and the point lookups.
  __device__ void wis_list_to_table() {
    if (threadIdx.x == 0) {
      int k = 0;
      for (int i = 0; i < S.ncand && k < kMaxSpecial; ++i)
        if (cm_sp[i]) {
          S.spec_id[k] = cm_id[i];
          S.spec_val[k] = cm_a[i];
          ++k;
        }
      S.nspec = k;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < bm_words; i += kThreads) bitmap[i] = 0u;   // overwrites the list
    __syncthreads();
    for (int i = threadIdx.x; i < S.nspec; i += kThreads) {
      const int loc = S.spec_id[i] - tok0;
      if (loc >= 0 && loc < p.slice) atomicOr(&bitmap[(loc / VE) >> 5], 1u << ((loc / VE) & 31));
    }
    __syncthreads();
  }

  // ---------------------------------------------------------------- plain IS
  __device__ void is_prepare() {
    // rows present and their branch counts
    if (threadIdx.x == 0) {
      for (int r = 0; r < kMaxRows; ++r) S.is_cnt[r] = 0;
      for (int i = 0; i < S.nv; ++i) S.is_cnt[S.vrow[i]]++;
    }
    __syncthreads();
    // range of rho = q / p_r over tokens with q > 0 and p_r > 0
    float lo = kPosInf, hi = 0.f;
    uint32_t mask = 1u;
    for (int r = 1; r < S.nrows; ++r)
      if (S.is_cnt[r]) mask |= 1u << r;
    stream(mask, [&](int, bool valid, const auto& L) {
      if (!valid) return;
      float q[VE];
      {
        float v[VE];
        L(0, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
      }
      for (int r = 1; r < S.nrows; ++r) {
        if (!S.is_cnt[r]) continue;
        float v[VE];
        L(r, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float pr = prob_of(v[e], S.M[r], S.c[r], S.invZ[r]);
          if (pr > 0.f && q[e] > 0.f) {
            const float rho = __fdiv_rn(q[e], pr);
            lo = fminf(lo, rho);
            hi = fmaxf(hi, rho);
          }
        }
      }
    });
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) {
      S.red[warp * 2] = lo;
      S.red[warp * 2 + 1] = hi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w = 0; w < kWarps; ++w) {
        lo = fminf(lo, S.red[w * 2]);
        hi = fmaxf(hi, S.red[w * 2 + 1]);
      }
      S.xch[xbuf][0] = lo;
      S.xch[xbuf][1] = hi;
    }
    cluster_gather(S, 2, xbuf, cn);
    if (threadIdx.x == 0) {
      float rlo = kPosInf, rhi = 0.f;
      for (int q = 0; q < cn; ++q) {
        rlo = fminf(rlo, S.gat[2 * q]);
        rhi = fmaxf(rhi, S.gat[2 * q + 1]);
      }
      rlo = fmaxf(rlo, 1e-37f);
      rhi = fmaxf(rhi, rlo);
      const float h = p.is_h;
      const float ulo = -logf((float)S.nv * rhi) - 40.f;
      const float uhi = logf(40.f / rlo);
      const int mlo = (int)floorf(ulo / h);
      int mhi = (int)ceilf(uhi / h);
      if (mhi - mlo + 1 > kIsNodesMax) mhi = mlo + kIsNodesMax - 1;
      S.is_mlo = mlo;
      S.is_n = mhi - mlo + 1;
      if (p.dbg_exps && rank == 0) {
        // the node sums below: one exponential per node, token and draft row
        int rows = 0;
        for (int r = 1; r < S.nrows; ++r) rows += S.is_cnt[r] ? 1 : 0;
        atomicAdd(p.dbg_exps, (unsigned long long)S.is_n * (unsigned long long)p.V * (unsigned long long)rows);
      }
    }
    __syncthreads();
    const int nn = S.is_n;
    for (int n = threadIdx.x; n < nn; n += kThreads) isT[n] = ex2(__fmul_rn((float)(S.is_mlo + n) * p.is_h, kLog2e));
    __syncthreads();
    // M_r(t_n) = sum_x p_r(x) exp(-t_n rho_r(x)), node chunks of kIsChunk
    for (int r = 1; r < S.nrows; ++r) {
      if (!S.is_cnt[r]) continue;
      for (int n0 = 0; n0 < nn; n0 += kIsChunk) {
        float acc[kIsChunk];
        float tl[kIsChunk];
#pragma unroll
        for (int i = 0; i < kIsChunk; ++i) {
          acc[i] = 0.f;
          tl[i] = (n0 + i < nn) ? __fmul_rn(isT[n0 + i], -kLog2e) : 0.f;
        }
        stream(1u | (1u << r), [&](int, bool valid, const auto& L) {
          if (!valid) return;
          float q[VE], pr[VE];
          {
            float v[VE];
            L(0, v);
#pragma unroll
            for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
            L(r, v);
#pragma unroll
            for (int e = 0; e < VE; ++e) pr[e] = prob_of(v[e], S.M[r], S.c[r], S.invZ[r]);
          }
#pragma unroll
          for (int e = 0; e < VE; ++e) {
            if (!(pr[e] > 0.f)) continue;
            const float rho = __fdiv_rn(q[e], pr[e]);
#pragma unroll
            for (int i = 0; i < kIsChunk; ++i) acc[i] = __fmaf_rn(pr[e], ex2(__fmul_rn(tl[i], rho)), acc[i]);
          }
        });
#pragma unroll
        for (int i = 0; i < kIsChunk; ++i) {
          const float v = warp_sum(acc[i]);
          if (lane == 0) S.red[warp * kIsChunk + i] = v;
        }
        __syncthreads();
        if (threadIdx.x < kIsChunk) {
          float v = 0.f;
          for (int w = 0; w < kWarps; ++w) v = __fadd_rn(v, S.red[w * kIsChunk + threadIdx.x]);
          S.xch[xbuf][threadIdx.x] = v;
        }
        cluster_gather(S, kIsChunk, xbuf, cn);
        if (threadIdx.x < kIsChunk && n0 + threadIdx.x < nn) {
          float v = 0.f;
          for (int q = 0; q < cn; ++q) v = __fadd_rn(v, S.gat[q * kIsChunk + threadIdx.x]);
          isW[r * kIsNodesMax + n0 + threadIdx.x] = v;  // M_r(t_n) for now
        }
        __syncthreads();
      }
    }
    // weights W_r(n) = h t_n c_r M_r^(c_r - 1) prod_{r' != r} M_r'^(c_r')
    for (int n = threadIdx.x; n < nn; n += kThreads) {
      float Mv[kMaxRows];
      for (int r = 1; r < S.nrows; ++r) Mv[r] = S.is_cnt[r] ? isW[r * kIsNodesMax + n] : 1.f;
      const float base = __fmul_rn(p.is_h, isT[n]);
      for (int r = 1; r < S.nrows; ++r) {
        if (!S.is_cnt[r]) continue;
        float w = __fmul_rn(base, (float)S.is_cnt[r]);
        for (int k = 1; k < S.is_cnt[r]; ++k) w = __fmul_rn(w, Mv[r]);
        for (int r2 = 1; r2 < S.nrows; ++r2) {
          if (r2 == r || !S.is_cnt[r2]) continue;
          for (int k = 0; k < S.is_cnt[r2]; ++k) w = __fmul_rn(w, Mv[r2]);
        }
        isW[r * kIsNodesMax + n] = w;
      }
    }
    __syncthreads();
  }

  // p_I(x) / q(x) = sum_r sum_n W_r(n) exp(-t_n rho_r(x)), compensated sum over nodes.
  __device__ float is_ratio_sum(const float* rho_r) const {
    float sum = 0.f, comp = 0.f;
    const int nn = S.is_n;
    for (int r = 1; r < S.nrows; ++r) {
      if (!S.is_cnt[r]) continue;
      const float rl = __fmul_rn(rho_r[r], -kLog2e);
      const float* W = isW + r * kIsNodesMax;
      for (int n = 0; n < nn; ++n) {
        const float term = __fmul_rn(W[n], ex2(__fmul_rn(isT[n], rl)));
        const float y = __fsub_rn(term, comp);
        const float t = __fadd_rn(sum, y);
        comp = __fsub_rn(__fsub_rn(t, sum), y);
        sum = t;
      }
    }
    return sum;
  }

  // ---------------------------------------------------------------- importance steps
  __device__ void single_importance() {
    if (threadIdx.x == 0) {
      S.Y = S.X[0];
      S.qY = prob_row(0, S.Y);
      S.pIY = prob_row(S.vrow[0], S.Y);
    }
  }

  __device__ void wis_importance(int b, int j) {
    if (threadIdx.x == 0) {
      for (int r = 0; r < kMaxRows; ++r) S.gamma[r] = 0.f;
      S.gamma[S.vrow[0]] = 1.f;
      S.nspec = 0;
    }
    bool fast = S.ncand >= 0;
    if (!fast)   // with a list the bitmap region still holds it; cleared on conversion
      for (int i = threadIdx.x; i < bm_words; i += kThreads) bitmap[i] = 0u;
    __syncthreads();
    int A = S.X[0];
    for (int m = 1; m < S.nv; ++m) {
      const float u = draw_uniform(p.seed, b, j, kDrawSelect + m - 1);
      if (fast) {
        fast = wis_stage_fast(A, S.X[m], S.vrow[m], u);
        if (fast) {
          A = S.Y;
          continue;
        }
        wis_list_to_table();
      }
      A = wis_stage_full(A, S.X[m], S.vrow[m], u);
    }
    if (fast) wis_list_to_table();
    if (threadIdx.x == 0) {
      S.Y = A;
      S.qY = prob_row(0, A);
      S.pIY = a_at(A);
    }
  }

  __device__ void is_importance(int b, int j) {
    if (threadIdx.x == 0) {
      // weights rho_i = q(X_i)/p_i(X_i); I = first i with running sum > u * total
      float rho[MDS_MAX_K], tot = 0.f;
      int inf_i = -1;
      for (int i = 0; i < S.nv; ++i) {
        const float pv = prob_row(S.vrow[i], S.X[i]);
        const float qv = prob_row(0, S.X[i]);
        rho[i] = pv > 0.f ? __fdiv_rn(qv, pv) : 0.f;
        if (!(pv > 0.f) && inf_i < 0) inf_i = i;
        tot = __fadd_rn(tot, rho[i]);
      }
      int I = S.nv - 1;
      if (inf_i >= 0) {
        I = inf_i;
      } else {
        const float T = __fmul_rn(draw_uniform(p.seed, b, j, kDrawSelect), tot);
        float run = 0.f;
        for (int i = 0; i < S.nv; ++i) {
          run = __fadd_rn(run, rho[i]);
          if (run > T) {
            I = i;
            break;
          }
        }
      }
      S.Y = S.X[I];
    }
    __syncthreads();
    is_prepare();
    if (threadIdx.x == 0) {
      const int y = S.Y;
      const float qv = prob_row(0, y);
      float rr[kMaxRows];
      for (int r = 1; r < S.nrows; ++r) {
        const float pv = S.is_cnt[r] ? prob_row(r, y) : 0.f;
        rr[r] = pv > 0.f ? __fdiv_rn(qv, pv) : kPosInf;
      }
      S.qY = qv;
      S.pIY = __fmul_rn(qv, is_ratio_sum(rr));
    }
  }

  // ---------------------------------------------------------------- one sequence
  // ---------------------------------------------------------------- truncated alphabet
  // Warp-wide inverse CDF over one weight per lane (lane order is the list's
  // token-id order): the smallest lane whose running sum exceeds u * total,
  // the last lane with positive weight if rounding leaves none, -1 if the
  // total is not positive.
  __device__ __forceinline__ int lane_cdf(float w, float u01, float* total) const {
    const int lane = threadIdx.x & 31;
    float c = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, c, o);
      if (lane >= o) c = __fadd_rn(c, t);
    }
    const float tot = __shfl_sync(0xffffffffu, c, 31);
    *total = tot;
    if (!(tot > 0.f)) return -1;
    const unsigned who = __ballot_sync(0xffffffffu, c > __fmul_rn(u01, tot));
    if (who) return __ffs(who) - 1;
    return 31 - __clz(__ballot_sync(0xffffffffu, w > 0.f));
  }

  // One depth of the truncated-alphabet scheme (Section 4, read together with
  // the non-iid appendix's remark on keeping only the inputs in Omega_0).
  // Omega_0 = the target tokens above the (M+1)-th largest target logit.  The
  // candidate list holds every token above cand_tau, so the cut is exact when
  // the list's (M+1)-th entry is >= cand_tau (or the list holds the whole
  // vocabulary, or every token outside it is -inf); otherwise the tokens above
  // cand_tau form Omega_0 and the status says so.  Warp 0 runs the WIS stages
  // on Omega_0, one list entry per lane, against q~ = q / p_a with the kept
  // inputs' draft laws restricted to Omega_0 and renormalised, then
  // Algorithm 1 against q~ (a lane-level inverse CDF for the residual).  The
  // result Y' is kept with probability p_a; otherwise a streaming draw over
  // the tokens outside Omega_0 in proportion to q replaces it.  Every CTA of
  // the cluster computes the same warp-0 result from the same list.
  __device__ int wis0_step(int b, int j, float* qYo, float* pIYo, int* Yo, float* Ro) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (warp == 0) {
      const unsigned FULL = 0xffffffffu;
      const int n = max(0, S.ncand);
      const bool have = lane < n;
      const int id = have ? cm_id[lane] : 0;
      const float l = have ? E::global(S.gptr[0], id) : kNegInf;
      int rk = 0;   // rank in the list by (larger logit, then lower id)
      for (int t = 0; t < 32; ++t) {
        const float lt = __shfl_sync(FULL, l, t);
        const int it = __shfl_sync(FULL, id, t);
        rk += (t < n && cand_before(lt, it, l, id)) ? 1 : 0;
      }
      const int M = p.omega0;
      const bool all0 = M >= p.V;
      float cut = kNegInf;
      bool cert;
      if (all0) {
        cert = S.cand_all != 0;
      } else {
        const unsigned who = __ballot_sync(FULL, have && rk == M);
        if (who) cut = __shfl_sync(FULL, l, __ffs(who) - 1);
        const float tau = S.cand_tau;
        cert = S.cand_all || (who ? cut >= tau : !(tau > kNegInf));
        if (!cert) cut = fmaxf(cut, tau);
      }
      const bool in0 = have && (all0 || l > cut);
      const int n0 = __popc(__ballot_sync(FULL, in0));
      const float q = in0 ? prob_of(l, S.M[0], S.c[0], S.invZ[0]) : 0.f;
      const float pa = warp_sum(q);
      const float qt = (in0 && pa > 0.f) ? __fdiv_rn(q, pa) : 0.f;
      // draft laws of this depth's rows restricted to Omega_0, renormalised:
      // point loads of the draft logits at Omega_0, exponents against their
      // own maximum (the rows' full normalisers cancel)
      for (int r = 1; r < S.nrows; ++r) {
        const float lr = in0 ? E::global(S.gptr[r], id) : kNegInf;
        float ref = lr;
#pragma unroll
        for (int o = 16; o; o >>= 1) ref = fmaxf(ref, __shfl_xor_sync(FULL, ref, o));
        const float cr = S.c[r];
        const float e = (in0 && ref > kNegInf) ? ex2(__fmaf_rn(lr, cr, -__fmul_rn(ref, cr))) : 0.f;
        const float P = warp_sum(e);
        if (lane == 0 && rank == 0 && P != P) atomicOr(p.status, MDS_ST_NONFINITE);
        cm_e[r * p.cand_cap + lane] = (P > 0.f) ? __fdiv_rn(e, P) : 0.f;
      }
      __syncwarp();
      // kept inputs: valid branches (branch order) whose token lies in Omega_0
      int nk = 0;
      for (int i = 0; i < S.nv; ++i) {
        const unsigned w = __ballot_sync(FULL, in0 && id == S.X[i]);
        if (!w) continue;
        const int li = __ffs(w) - 1;
        if (!(cm_e[S.vrow[i] * p.cand_cap + li] > 0.f)) continue;   // impossible draw: dropped
        if (lane == 0) {
          S.k_lane[nk] = li;
          S.k_row[nk] = S.vrow[i];
        }
        ++nk;
      }
      __syncwarp();
      int yl = -1, Yl = -1;
      float qY = 0.f, pIY = 0.f, R = 0.f;
      if (n0 > 0 && nk == 0) {
        float t;
        yl = lane_cdf(qt, draw_uniform(p.seed, b, j, kDrawResidual), &t);
      } else if (n0 > 0) {
        float a = cm_e[S.k_row[0] * p.cand_cap + lane];
        int A = S.k_lane[0];
        const int s = min(p.wis_s, n0);
        for (int m = 1; m < nk; ++m) {
          const int Bl = S.k_lane[m];
          const float bb = cm_e[S.k_row[m] * p.cand_cap + lane];
          const float u = draw_uniform(p.seed, b, j, kDrawSelect + m - 1);
          // Omega_1: the s largest keys q~ - a b in Omega_0, ties to the lower id
          unsigned kk = in0 ? ord_key(__fadd_rn(__fmaf_rn(-a, bb, qt), 0.f)) : 0u;
          uint32_t selm = 0u;
          for (int t = 0; t < s; ++t) {
            const unsigned km = __reduce_max_sync(FULL, kk);
            const uint32_t who = __ballot_sync(FULL, km != 0u && kk == km);
            if (!who) break;
            const int wl = __ffs(who) - 1;
            selm |= 1u << wl;
            if (lane == wl) kk = 0u;
          }
          const bool sel = (selm >> lane) & 1u;
          const int sn = __popc(selm);
          const float A2 = warp_sum((in0 && !sel) ? a : 0.f);
          const float B2 = warp_sum((in0 && !sel) ? bb : 0.f);
          const int rk1 = __popc(selm & ((1u << lane) - 1u));
          if (lane >= sn && lane < MDS_MAX_S) {
            S.om[lane] = -1;
            S.om_q[lane] = 0.f;
            S.om_a[lane] = 0.f;
            S.om_b[lane] = 0.f;
          }
          if (sel) {
            S.om[rk1] = id;
            S.om_q[rk1] = qt;
            S.om_a[rk1] = a;
            S.om_b[rk1] = bb;
          }
          __syncwarp();
          if (lane == 0) S.Y = stage_solve(sn, A2, B2, cm_id[A], cm_id[Bl], u);
          __syncwarp();
          const int Yt = S.Y;
          A = max(0, __ffs(__ballot_sync(FULL, in0 && id == Yt)) - 1);   // Yt is A's or B's token
          a = sel ? S.om_x[rk1] : (in0 ? __fmul_rn(0.5f, __fadd_rn(__fmul_rn(a, B2), __fmul_rn(bb, A2))) : 0.f);
          __syncwarp();
        }
        Yl = A;
        qY = __shfl_sync(FULL, qt, A);
        pIY = __shfl_sync(FULL, a, A);
        const float ratio = pIY > 0.f ? __fdiv_rn(qY, pIY) : kPosInf;
        if (draw_uniform(p.seed, b, j, kDrawAccept) < fminf(1.f, ratio)) {
          yl = A;
        } else {
          const float ures = draw_uniform(p.seed, b, j, kDrawResidual);
          yl = lane_cdf(in0 ? fmaxf(0.f, __fsub_rn(qt, a)) : 0.f, ures, &R);
          if (yl < 0) {   // only by rounding: sample q~
            if (lane == 0 && rank == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
            float t;
            yl = lane_cdf(qt, ures, &t);
          }
        }
      }
      if (lane == 0) {
        if (!cert && rank == 0) atomicOr(p.status, MDS_ST_OMEGA0);
        S.o0_n = n0;
        S.o0_all = (all0 && S.cand_all) ? 1 : 0;
        S.o0_cut = cut;
        S.o0_pa = pa;
        S.o0_R = R;
        S.o0_Yp = (yl >= 0) ? cm_id[yl] : -1;
        S.Y = (Yl >= 0) ? cm_id[Yl] : -1;
        S.qY = qY;
        S.pIY = pIY;
      }
    }
    __syncthreads();
    *Yo = S.Y;
    *qYo = S.qY;
    *pIYo = S.pIY;
    *Ro = S.o0_R;
    const int Yp = S.o0_Yp;
    if (S.o0_n > 0 && (S.o0_all || draw_uniform(p.seed, b, j, kDrawKeep) < S.o0_pa)) return Yp;
    // replace: a draw over the tokens outside Omega_0 in proportion to q
    const float cut = S.o0_cut;
    const bool all0 = S.o0_all != 0;
    float tot;
    int Z = sample_cdf(
        1u,
        [&](int, const auto& L, float* r) {
          float v[VE];
          L(0, v);
#pragma unroll
          for (int e = 0; e < VE; ++e) r[e] = (all0 || v[e] > cut) ? 0.f : prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
        },
        draw_uniform(p.seed, b, j, kDrawOutside), &tot);
    if (Z < 0) {   // no target mass outside Omega_0
      if (Yp >= 0) return Yp;
      if (threadIdx.x == 0 && rank == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
      Z = sample_cdf(
          1u,
          [&](int, const auto& L, float* r) {
            float v[VE];
            L(0, v);
#pragma unroll
            for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
          },
          draw_uniform(p.seed, b, j, kDrawOutside), &tot);
    }
    return Z;
  }

  __device__ __forceinline__ void run_sequence(int b) {
    const int K = p.K, L = p.L, V = p.V;
    const int tid = threadIdx.x;
    unsigned valid = (K >= 32) ? 0xffffffffu : ((1u << K) - 1u);
    int acc_len = L;
    for (int j = 0; j <= L; ++j) {
      const bool bonus = (j == L);
      if (threadIdx.x < 32) {   // tokens of every branch at this depth, one lane each
        const int k = threadIdx.x;
        S.tok_j[k] = (!bonus && k < K) ? p.tokens[((size_t)b * K + k) * L + j] : 0;
      }
      __syncthreads();
      if (tid == 0) {
        // plan the rows of this depth
        const int kstar = __ffs(valid) - 1;
        for (int m = 0; m < MDS_MAX_K; ++m) S.model_row[m] = -1;
        S.gptr[0] = p.target + ((((size_t)b * K + kstar) * (L + 1) + j) * (size_t)V) * p.esize;
        float tq = p.temps[(size_t)b * (1 + K)];
        int nr = 1;
        S.nv = 0;
        if (!bonus) {
          for (int k = 0; k < K; ++k) {
            if (!(valid >> k & 1u)) continue;
            const int m = p.model_of[k];
            if (S.model_row[m] < 0) {
              S.model_row[m] = nr;
              S.gptr[nr] = p.drafts[k] + (((size_t)b * L + j) * (size_t)V) * p.esize;
              float td = p.temps[(size_t)b * (1 + K) + 1 + k];
              if (!(td > 0.f) || !(td < kPosInf)) {
                atomicOr(p.status, MDS_ST_BADTEMP);
                td = 1.f;
              }
              S.c[nr] = __fdiv_rn(kLog2e, td);
              ++nr;
            }
            const int i = S.nv++;
            S.vbr[i] = k;
            int x = S.tok_j[k];
            if (x < 0 || x >= V) {
              atomicOr(p.status, MDS_ST_BADTOKEN);
              x = 0;
            }
            S.X[i] = x;
            S.vrow[i] = S.model_row[m];
          }
        }
        if (!(tq > 0.f) || !(tq < kPosInf)) {
          atomicOr(p.status, MDS_ST_BADTEMP);
          tq = 1.f;
        }
        S.c[0] = __fdiv_rn(kLog2e, tq);
        S.nrows = nr;
      }
      __syncthreads();
      if (!bonus) depth_stats((SCHEME == MDS_WIS && S.nv > 1) || SCHEME == MDS_WIS0);
      int Z;
      float qY = 0.f, pIY = 0.f, Rdiag = 0.f;
      int Ydiag = -1;
      if (bonus) {
        float tot;
        Z = bonus_pass(draw_uniform(p.seed, b, j, kDrawBonus), &tot);
        Rdiag = tot;
      } else if constexpr (SCHEME == MDS_SPECTR) {
        Z = spectr(b, j, &qY, &pIY, &Ydiag, &Rdiag);
      } else if constexpr (SCHEME == MDS_WIS0) {
        Z = wis0_step(b, j, &qY, &pIY, &Ydiag, &Rdiag);
      } else {
        // importance step -> Y and the law p_I (kept in S for the residual)
        int Y;
        if constexpr (SCHEME == MDS_WIS) {
          if (S.nv > 1)
            wis_importance(b, j);
          else
            single_importance();
        } else if constexpr (SCHEME == MDS_IS) {
          if (S.nv > 1)
            is_importance(b, j);
          else
            single_importance();
        } else {
          single_importance();
        }
        __syncthreads();
        Y = S.Y;
        qY = S.qY;
        pIY = S.pIY;
        Ydiag = Y;
        // Algorithm 1 on Y
        const float uacc = draw_uniform(p.seed, b, j, kDrawAccept);
        const float ratio = pIY > 0.f ? __fdiv_rn(qY, pIY) : kPosInf;
        const bool acc = uacc < fminf(1.f, ratio);
        if (acc && !p.acc_prob) {
          Z = Y;
        } else {
          // the residual mass R = sum max(0, q - p_I) and, after a rejection,
          // the draw from it; with acc_prob an accepted depth computes R too
          // (1 - R = sum min(q, p_I), the depth's acceptance probability)
          const float ures = acc ? 0.f : draw_uniform(p.seed, b, j, kDrawResidual);
          float tot;
          bool done = false;
          if constexpr (SCHEME == MDS_WIS) {
            if (S.nv > 1) {
              uint32_t mask = 1u;
              for (int r = 1; r < S.nrows; ++r)
                if (S.gamma[r] != 0.f) mask |= 1u << r;
              Z = sample_cdf(mask, [&](int gu, const auto& L, float* r) { residual_wis(gu, L, r); }, ures, &tot);
              done = true;
            }
          }
          if constexpr (SCHEME == MDS_IS) {
            if (S.nv > 1) {
              uint32_t mask = 1u;
              int rows = 0;
              for (int r = 1; r < S.nrows; ++r)
                if (S.is_cnt[r]) {
                  mask |= 1u << r;
                  ++rows;
                }
              if (p.dbg_exps && rank == 0 && tid == 0)   // p_I at every token: one exponential per node and row
                atomicAdd(p.dbg_exps, (unsigned long long)S.is_n * (unsigned long long)p.V * (unsigned long long)rows);
              Z = sample_cdf(mask, [&](int, const auto& L, float* r) { residual_is(L, r); }, ures, &tot);
              done = true;
            }
          }
          if (!done) {
            const int r1 = S.vrow[0];
            Z = sample_cdf(
                1u | (1u << r1),
                [&](int, const auto& L, float* r) {
                  float v[VE], w[VE];
                  L(0, v);
                  L(r1, w);
#pragma unroll
                  for (int e = 0; e < VE; ++e)
                    r[e] = fmaxf(0.f, __fsub_rn(prob_of(v[e], S.M[0], S.c[0], S.invZ[0]),
                                                prob_of(w[e], S.M[r1], S.c[r1], S.invZ[r1])));
                },
                ures, &tot);
          }
          Rdiag = tot;
          if (acc) {
            Z = Y;
          } else if (Z < 0) {
            if (tid == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
            Z = sample_cdf(
                1u,
                [&](int, const auto& L, float* r) {
                  float v[VE];
                  L(0, v);
#pragma unroll
                  for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
                },
                ures, &tot);
          }
        }
      }
      // outputs and the walk
      if (rank == 0 && tid == 0) {
        p.out_tokens[(size_t)b * (L + 1) + j] = Z;
        if (p.out_diag) {
          float* dg = p.out_diag + ((size_t)b * (L + 1) + j) * 4;
          dg[0] = qY;
          dg[1] = pIY;
          dg[2] = Rdiag;
          dg[3] = (float)Ydiag;
        }
      }
      if (bonus) {
        acc_len = L;
        break;
      }
      unsigned nvld = 0u;
      for (int i = 0; i < S.nv; ++i)
        if (S.X[i] == Z) nvld |= 1u << S.vbr[i];
      __syncthreads();
      if (!nvld) {
        acc_len = j;
        break;
      }
      valid = nvld;
    }
    if (rank == 0 && tid == 0) {
      if (*reinterpret_cast<volatile unsigned*>(p.status) & MDS_ST_TIMEOUT) {
        abandon(b);   // a ring wait gave up during the launch: this walk is not trusted
      } else {
        p.out_accept[b] = acc_len;
        for (int j = acc_len + 1; j <= L; ++j) p.out_tokens[(size_t)b * (L + 1) + j] = -1;
      }
    }
  }

  // Outputs of a sequence the launch gives up on: accept length -1, every
  // token -1 (the diagnostics are left as they are).
  __device__ void abandon(int b) const {
    p.out_accept[b] = -1;
    for (int j = 0; j <= p.L; ++j) p.out_tokens[(size_t)b * (p.L + 1) + j] = -1;
  }

  // residual weight max(0, q - p_I) for WIS (generic gamma law + special table)
  template <class LD>
  __device__ __forceinline__ void residual_wis(int gu, const LD& L, float* r) const {
    const int tbase = tok0 + gu * VE;
    float q[VE], a[VE];
    {
      float v[VE];
      L(0, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
        a[e] = 0.f;
      }
    }
    for (int rr = 1; rr < S.nrows; ++rr) {
      const float g = S.gamma[rr];
      if (g == 0.f) continue;
      float v[VE];
      L(rr, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = __fmaf_rn(g, prob_of(v[e], S.M[rr], S.c[rr], S.invZ[rr]), a[e]);
    }
    if ((bitmap[gu >> 5] >> (gu & 31)) & 1u) {   // the unit holds a special token
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = special_lookup(tbase + e, a[e]);
    }
#pragma unroll
    for (int e = 0; e < VE; ++e) r[e] = fmaxf(0.f, __fsub_rn(q[e], a[e]));
  }

  // residual weight max(0, q - p_I) for plain IS (Laplace identity)
  template <class LD>
  __device__ __forceinline__ void residual_is(const LD& L, float* r) const {
    float q[VE];
    {
      float v[VE];
      L(0, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
    }
    float rho[VE][kMaxRows];
    for (int rr = 1; rr < S.nrows; ++rr) {
      if (!S.is_cnt[rr]) continue;
      float v[VE];
      L(rr, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const float pv = prob_of(v[e], S.M[rr], S.c[rr], S.invZ[rr]);
        rho[e][rr] = pv > 0.f ? __fdiv_rn(q[e], pv) : kPosInf;
      }
    }
#pragma unroll
    for (int e = 0; e < VE; ++e) {
      if (!(q[e] > 0.f)) {
        r[e] = 0.f;
        continue;
      }
      const float pI = __fmul_rn(q[e], is_ratio_sum(rho[e]));
      r[e] = fmaxf(0.f, __fsub_rn(q[e], pI));
    }
  }

  // Sequential rejection over the valid drafts (baseline).  Returns Z.
  // *Rd: the product of the rounds' residual masses, the probability that
  // every round rejects (1 - the depth's acceptance probability); with
  // acc_prob the rounds after an acceptance are computed for it too, without
  // changing the token.
  __device__ int spectr(int b, int j, float* qY, float* pIY, int* Yd, float* Rd) {
    const int nv = S.nv;
    int zacc = -1;
    float prodR = 1.f;
    for (int i = 0; i < nv; ++i) {
      // point value of the running target at X_i (the accept test, until a
      // round accepts)
      if (threadIdx.x == 0) S.sp_rows[i] = S.vrow[i];
      if (threadIdx.x == 0 && zacc < 0) {
        const int x = S.X[i];
        float qi = prob_row(0, x);
        for (int k = 0; k < i; ++k) {
          const float pk = prob_row(S.sp_rows[k], x);
          if (S.sp_invR[k] > 0.f) qi = __fmul_rn(fmaxf(0.f, __fsub_rn(qi, pk)), S.sp_invR[k]);
        }
        const float pv = prob_row(S.vrow[i], x);
        const float ratio = pv > 0.f ? __fdiv_rn(qi, pv) : kPosInf;
        const float u = draw_uniform(p.seed, b, j, kDrawAccept + i);
        if (i == 0) {
          S.qY = qi;
          S.pIY = pv;
        }
        S.accepted = (u < fminf(1.f, ratio)) ? 1 : 0;
      }
      __syncthreads();
      *qY = S.qY;
      *pIY = S.pIY;
      *Yd = S.X[0];
      if (zacc < 0 && S.accepted) {
        zacc = S.X[i];
        if (!p.acc_prob) {
          __syncthreads();
          *Rd = 0.f;
          return zacc;
        }
      }
      // residual mass of this round
      float part = 0.f;
      const int ri = S.sp_rows[i];
      uint32_t mask = 1u | (1u << ri);
      for (int k = 0; k < i; ++k) mask |= 1u << S.sp_rows[k];
      stream(mask, [&](int, bool valid, const auto& L) {
        if (!valid) return;
        float r[VE];
        spectr_target(L, i, r);
        float w[VE];
        L(ri, w);
#pragma unroll
        for (int e = 0; e < VE; ++e) part += fmaxf(0.f, __fsub_rn(r[e], prob_of(w[e], S.M[ri], S.c[ri], S.invZ[ri])));
      });
      part = warp_sum(part);
      const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
      if (lane == 0) S.red[warp] = part;
      __syncthreads();
      if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < kWarps; ++w) t = __fadd_rn(t, S.red[w]);
        S.xch[xbuf][0] = t;
      }
      cluster_gather(S, 1, xbuf, cn);
      if (threadIdx.x == 0) {
        float R = 0.f;
        for (int q = 0; q < cn; ++q) R = __fadd_rn(R, S.gat[q]);
        S.sp_invR[i] = R > 0.f ? __frcp_rn(R) : 0.f;
        S.red[kWarps] = R;
      }
      __syncthreads();
      prodR = __fmul_rn(prodR, S.red[kWarps]);
      __syncthreads();
    }
    *Rd = prodR;
    if (zacc >= 0) return zacc;
    float tot;
    uint32_t mask = 1u;
    for (int k = 0; k < nv; ++k) mask |= 1u << S.sp_rows[k];
    const int z = sample_cdf(mask, [&](int, const auto& L, float* r) { spectr_target(L, nv, r); },
                             draw_uniform(p.seed, b, j, kDrawResidual), &tot);
    return z;
  }

  // running target after `rounds` rejected rounds, for one unit
  template <class LD>
  __device__ __forceinline__ void spectr_target(const LD& L, int rounds, float* r) const {
    float v[VE];
    L(0, v);
#pragma unroll
    for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
    for (int k = 0; k < rounds; ++k) {
      if (!(S.sp_invR[k] > 0.f)) continue;
      const int rk = S.sp_rows[k];
      float w[VE];
      L(rk, w);
#pragma unroll
      for (int e = 0; e < VE; ++e)
        r[e] = __fmul_rn(fmaxf(0.f, __fsub_rn(r[e], prob_of(w[e], S.M[rk], S.c[rk], S.invZ[rk]))), S.sp_invR[k]);
    }
  }
};

template <int DT, int SCHEME>
__global__ void __launch_bounds__(kThreads, SCHEME == MDS_IS ? 1 : 2) verify_kernel(const __grid_constant__ Params p) {
  extern __shared__ __align__(128) char dsm[];
  __shared__ State S;
  Kernel<DT, SCHEME> k{p, S};
  k.rank = (int)cluster_rank();
  k.cn = p.cn;
  k.tok0 = k.rank * p.slice;
  k.nvalid = max(0, min(p.slice, p.V - k.tok0));
  k.Uv = (k.nvalid + Kernel<DT, SCHEME>::VE - 1) / Kernel<DT, SCHEME>::VE;
  k.nseg = (p.slice / Kernel<DT, SCHEME>::VE + 31) / 32;   // same in every CTA: peers map the same offsets
  k.nsegv = (k.Uv + 31) / 32;                                // segments the residual pass writes
  k.bm_words = (p.slice / Kernel<DT, SCHEME>::VE + 31) / 32;   // one bit per 16-byte unit
  // dynamic shared memory: ring | segment sums | chunk sums | segment references | scheme region
  //   IS : nodes t_n | weights W_r(n)
  //   WIS: CTA list (two copies) | warp lists = staging list | merged list, the
  //        last aliased later by the special-token bitmap (only the CTA list
  //        is ever read by other CTAs)
  k.ring = dsm;
  k.segsum = reinterpret_cast<float*>(dsm + p.ring_bytes);
  k.chksum = k.segsum + ((k.nseg + 3) & ~3);
  k.segref = k.chksum + ((((k.nseg + 31) / 32) + 3) & ~3);
  {
    char* c = reinterpret_cast<char*>(k.segref + ((k.nseg + 3) & ~3));
    k.isT = reinterpret_cast<float*>(c);
    k.isW = k.isT + kIsNodesMax;
    k.cl_base = c;
    c += (size_t)2 * kListN * (1 + p.rows_max) * 4;
    // the warps' set-aside lists and the staging list share one region: the
    // lists are compacted into the CTA list before anything is staged
    char* st = c;
    k.ap_id = reinterpret_cast<int*>(st);
    k.ap_l = reinterpret_cast<float*>(st + (size_t)kWarps * kWarpApp * 4);
    k.cs_id = reinterpret_cast<int*>(c);
    c += (size_t)p.cand_stage * 4;
    k.cs_l = reinterpret_cast<float*>(c);
    c += (size_t)p.cand_stage * p.rows_max * 4;
    k.cs_x = reinterpret_cast<float*>(c);
    c += (size_t)p.cand_stage * 4;
    if (p.cand_cap > 0) c = st + max(c - st, (ptrdiff_t)kWarps * kWarpApp * 4 * (1 + p.rows_max));
    k.bitmap = reinterpret_cast<uint32_t*>(c);
    k.cm_id = reinterpret_cast<int*>(c);
    c += (size_t)p.cand_cap * 4;
    k.cm_e = reinterpret_cast<float*>(c);
    c += (size_t)p.cand_cap * p.rows_max * 4;
    k.cm_a = reinterpret_cast<float*>(c);
    c += (size_t)p.cand_cap * 4;
    k.cm_sp = reinterpret_cast<int*>(c);
  }
  k.xbuf = 0;
  k.clbuf = 0;
  k.wphase = 0u;
  k.bail = 0;
  if (threadIdx.x == 0) {
    for (int w = 0; w < kWarps; ++w)
      for (int i = 0; i < kWStages; ++i) mbar_init(&S.wbar[w][i]);
    mbar_init_fence();
  }
  __syncthreads();
  // A peer's shared memory may be accessed only once every CTA of the
  // cluster is running: one cluster barrier before the first remote store.
  if (p.cn > 1) cluster_sync_all();
  for (;;) {
    if (k.rank == 0 && threadIdx.x == 0) {
      int b = (int)(atomicAdd(p.queue, 1u) - p.ticket0);
      if (b < p.B && (*reinterpret_cast<volatile unsigned*>(p.status) & MDS_ST_TIMEOUT)) {
        k.abandon(b);   // after a ring wait gave up, the remaining sequences are only marked
        b = -1;
      }
      if (p.cn > 1) {
        for (int q = 0; q < p.cn; ++q) st_dsmem(&S.next_b, (uint32_t)q, b);
      } else {
        S.next_b = b;
      }
    }
    if (p.cn > 1)
      cluster_sync_all();
    else
      __syncthreads();
    const int b = *(volatile int*)&S.next_b;
    __syncthreads();
    if (b >= p.B) break;
    if (b < 0) {
      // every CTA of the cluster has read S.next_b before rank 0 writes it again
      if (p.cn > 1) cluster_sync_all();
      continue;
    }
    k.run_sequence(b);
  }
}

}  // namespace

size_t smem_bytes(const Params& p) {
  const int VE = 16 / p.esize;
  const int nseg = (p.slice / VE + 31) / 32;
  size_t bytes = (size_t)p.ring_bytes + (size_t)((nseg + 3) & ~3) * 4 * 2 + (size_t)((((nseg + 31) / 32) + 3) & ~3) * 4;
  if (p.scheme == MDS_IS) bytes += (size_t)kIsNodesMax * 4 * (1 + p.rows_max);
  if (p.scheme == MDS_WIS || p.scheme == MDS_WIS0) {
    const size_t bm = (size_t)((p.slice / VE + 31) / 32) * 4;
    const size_t cm = (size_t)p.cand_cap * 4 * (3 + p.rows_max);
    size_t stg = (size_t)p.cand_stage * 4 * (2 + p.rows_max);
    const size_t app = (size_t)kWarps * kWarpApp * 4 * (1 + p.rows_max);
    if (p.cand_cap > 0 && app > stg) stg = app;
    bytes += (size_t)2 * kListN * 4 * (1 + p.rows_max) + stg +
             (bm > cm ? bm : cm);
  }
  return bytes;
}

using KernelFn = void (*)(Params);

static KernelFn kernel_for(int dtype, int scheme) {
  if (dtype == MDS_F32) {
    switch (scheme) {
      case MDS_IS: return verify_kernel<MDS_F32, MDS_IS>;
      case MDS_WIS: return verify_kernel<MDS_F32, MDS_WIS>;
      case MDS_SPECTR: return verify_kernel<MDS_F32, MDS_SPECTR>;
      case MDS_WIS0: return verify_kernel<MDS_F32, MDS_WIS0>;
      default: return verify_kernel<MDS_F32, MDS_SINGLE>;
    }
  }
  switch (scheme) {
    case MDS_IS: return verify_kernel<MDS_BF16, MDS_IS>;
    case MDS_WIS: return verify_kernel<MDS_BF16, MDS_WIS>;
    case MDS_SPECTR: return verify_kernel<MDS_BF16, MDS_SPECTR>;
    case MDS_WIS0: return verify_kernel<MDS_BF16, MDS_WIS0>;
    default: return verify_kernel<MDS_BF16, MDS_SINGLE>;
  }
}

cudaError_t configure_kernel(int dtype) {
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  for (int scheme = MDS_SINGLE; scheme <= MDS_WIS0; ++scheme) {
    const void* fn = (const void*)kernel_for(dtype, scheme);
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, fn);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

static void fill_config(cudaLaunchConfig_t& cfg, cudaLaunchAttribute* at, const Params& p, int clusters,
                        cudaStream_t stream) {
  cfg = cudaLaunchConfig_t{};
  cfg.gridDim = dim3((unsigned)(clusters * p.cn));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem_bytes(p);
  cfg.stream = stream;
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = (unsigned)p.cn;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
}

int max_active_clusters(const Params& p) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute at[1];
  fill_config(cfg, at, p, 1, nullptr);
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (const void*)kernel_for(p.dtype, p.scheme), &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch(const Params& p, int clusters, cudaStream_t stream) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute at[1];
  fill_config(cfg, at, p, clusters, stream);
  return cudaLaunchKernelEx(&cfg, kernel_for(p.dtype, p.scheme), p);
}

}  // namespace mds
