// Batched multi-draft speculative verification on GB300 (sm_103a).
//
// One thread-block cluster verifies one sequence at a time and loops over
// sequences taken from a work counter (a persistent kernel sized to the
// co-resident clusters).  CTA r of the cluster owns tokens
// [r*slice, (r+1)*slice) of every row.  Per depth j of the walk it
//   1. bulk-copies (cp.async.bulk, mbarrier completion) its slice of the
//      target row and of one row per distinct draft model into shared memory,
//   2. computes the temperature-softmax statistics (max, sum of exp) of each
//      row and combines them across the cluster through distributed shared
//      memory,
//   3. runs the importance step of the selected scheme (Definition 1 /
//      Theorem 1), reading the rows from shared memory,
//   4. applies Algorithm 1 (accept with probability min(1, q(Y)/p_I(Y)), else
//      an inverse-CDF draw from max(0, q - p_I) in token order), and
//   5. advances the walk: continue while the output is one of the valid draft
//      tokens (Problem 1's event Z in S); after L accepted positions draw the
//      bonus token from the target row at depth L.
// Every decision is taken redundantly and identically by every CTA of the
// cluster from cluster-combined values, so control flow stays uniform and
// the cluster barriers always match.  There are no spin-waits across CTAs;
// the only wait is on this CTA's own bulk copies and it is bounded.
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
constexpr int kCandLevels = 4;          // candidate levels: q >= q_max * 2^-(12, 10, 8, 6)
__host__ __device__ constexpr float cand_log2(int level) { return 12.f - 2.f * (float)level; }

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
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
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
};

// Probability of a logit under a row's statistics.  The same expression is
// used for in-pass values and point lookups so both give identical bits.
__device__ __forceinline__ float prob_of(float l, float M, float c, float invZ) {
  return __fmul_rn(ex2(__fmul_rn(__fsub_rn(l, M), c)), invZ);
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
  int tma_bytes;
  // walk
  int nv;                     // valid branches
  int vbr[MDS_MAX_K];         // valid branch ids, ascending
  int X[MDS_MAX_K];           // their tokens at this depth
  int vrow[MDS_MAX_K];        // row of each valid branch's draft model
  // outcome of the depth
  int Y, Z, accepted, flags;
  float qY, pIY, R;
  int next_b;
  int Zslot;
  int tok_j[32];
  // cluster exchange (double-buffered) and its gathered copy
  float xch[2][kXch];
  float gat[kMaxCluster * kXch];
  // block reduction scratch
  float red[kWarps * 2 * kMaxRows];
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
  float W[kMaxPairs];
  float lp_rs[kMaxPairs], lp_fl[kMaxPairs], lp_fh[kMaxPairs], lp_m[kMaxPairs];
  float A2, B2;
  // WIS candidate list bookkeeping
  int wcnt[kWarps];
  float pc[kMaxRows];        // complement exp mass per row
  int ncand, cand_all, fast_ok;
  float cand_q;
  int wlev[kWarps * kCandLevels];
  // SpecTr: inverse residual masses of rejected rounds
  float sp_invR[MDS_MAX_K];
  int sp_rows[MDS_MAX_K];
  // IS: quadrature grid
  int is_mlo, is_n;
  int is_cnt[kMaxRows];
  float rho_min, rho_max;
  // CDF search
  int owner, seg;
  float run, T;
  uint64_t mbar;
};

// ------------------------------------------------------------------ reductions

__device__ __forceinline__ void combine_ms(float& m, float& s, float m2, float s2, float c) {
  const float M = fmaxf(m, m2);
  const float a = (m == kNegInf) ? 0.f : __fmul_rn(s, ex2(__fmul_rn(__fsub_rn(m, M), c)));
  const float b = (m2 == kNegInf) ? 0.f : __fmul_rn(s2, ex2(__fmul_rn(__fsub_rn(m2, M), c)));
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

template <int DT, int SCHEME>
struct Kernel {
  using E = Elt<DT>;
  static constexpr int VE = E::VE;

  const Params& p;
  State& S;
  char* rows;          // rows_max x row_stride
  uint32_t* bitmap;    // special-token bits of this CTA's slice
  float* segsum;       // per-segment residual sums
  float* isW;          // IS: weights [rows][kIsNodesMax]
  float* isT;          // IS: nodes t_n
  int* cl_id;          // WIS: this CTA's candidates (token order) ...
  float* cl_e;         //      ... and their exp values per row [rows][cap_cta]
  int* cm_id;          // WIS: the cluster's merged candidates (token order) ...
  float* cm_e;         //      ... exp values per row [rows][cap]
  float* cm_a;         //      ... current law value of special tokens
  int* cm_sp;          //      ... special flag
  int rank, cn, tok0, nvalid, U, nseg, bm_words;
  int xbuf;
  uint32_t mphase;

  __device__ const char* srow(int r) const { return rows + (size_t)r * p.row_stride; }

  __device__ float prob_row(int r, int x) const {
    return prob_of(E::global(S.gptr[r], x), S.M[r], S.c[r], S.invZ[r]);
  }

  // ---------------------------------------------------------------- loads
  __device__ void load_rows() {
    const int nr = S.nrows;
    const int tid = threadIdx.x;
    const int vbytes = nvalid * p.esize;
    const int tma_bytes = p.tma_ok ? (vbytes & ~15) : 0;
    // padding (tokens past V) reads as -inf; plain loads for what bulk copies skip
    for (int r = 0; r < nr; ++r) {
      char* dst = rows + (size_t)r * p.row_stride;
      const char* src = S.gptr[r] + (size_t)tok0 * p.esize;
      for (int i = tid; i < p.slice - nvalid; i += kThreads) {
        const int t = nvalid + i;
        if (DT == MDS_F32)
          reinterpret_cast<float*>(dst)[t] = kNegInf;
        else
          reinterpret_cast<unsigned short*>(dst)[t] = 0xff80u;
      }
      for (int byte = tma_bytes + tid * p.esize; byte < vbytes; byte += kThreads * p.esize) {
        if (DT == MDS_F32)
          *reinterpret_cast<float*>(dst + byte) = __ldg(reinterpret_cast<const float*>(src + byte));
        else
          *reinterpret_cast<unsigned short*>(dst + byte) = __ldg(reinterpret_cast<const unsigned short*>(src + byte));
      }
    }
    if (tma_bytes > 0) {
      if (tid == 0) {
        fence_proxy_async();
        mbar_expect_tx(&S.mbar, (uint32_t)(tma_bytes * nr));
        for (int r = 0; r < nr; ++r)
          bulk_copy(rows + (size_t)r * p.row_stride, S.gptr[r] + (size_t)tok0 * p.esize, (uint32_t)tma_bytes,
                    &S.mbar);
      }
      long long spins = 0;
      while (!mbar_try_wait(&S.mbar, mphase)) {
        if (++spins > kWaitLimit) {
          if (tid == 0) atomicOr(p.status, MDS_ST_TIMEOUT);
          break;
        }
      }
      mphase ^= 1u;
    }
    __syncthreads();
  }

  // ---------------------------------------------------------------- stats
  // Softmax statistics of every loaded row: M = max logit, Z = sum exp((l-M)/T).
  __device__ void row_stats() {
    const int nr = S.nrows;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int r = 0; r < nr; ++r) {
      const char* row = srow(r);
      const float c = S.c[r];
      float m = kNegInf;
      for (int u = threadIdx.x; u < U; u += kThreads) {
        float v[VE];
        E::unit(row, u, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) m = fmaxf(m, v[e]);
      }
      float s = 0.f;
      if (m != kNegInf) {
        for (int u = threadIdx.x; u < U; u += kThreads) {
          float v[VE];
          E::unit(row, u, v);
#pragma unroll
          for (int e = 0; e < VE; ++e) s += ex2(__fmul_rn(__fsub_rn(v[e], m), c));
        }
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        combine_ms(m, s, m2, s2, c);
      }
      if (lane == 0) {
        S.red[(warp * kMaxRows + r) * 2] = m;
        S.red[(warp * kMaxRows + r) * 2 + 1] = s;
      }
    }
    __syncthreads();
    if (threadIdx.x < nr) {
      const int r = threadIdx.x;
      float m = kNegInf, s = 0.f;
      for (int w = 0; w < kWarps; ++w)
        combine_ms(m, s, S.red[(w * kMaxRows + r) * 2], S.red[(w * kMaxRows + r) * 2 + 1], S.c[r]);
      S.xch[xbuf][2 * r] = m;
      S.xch[xbuf][2 * r + 1] = s;
    }
    cluster_gather(S, 2 * nr, xbuf, cn);
    if (threadIdx.x < nr) {
      const int r = threadIdx.x;
      float m = kNegInf, s = 0.f;
      for (int q = 0; q < cn; ++q) combine_ms(m, s, S.gat[q * 2 * nr + 2 * r], S.gat[q * 2 * nr + 2 * r + 1], S.c[r]);
      if (!(m > kNegInf) || !(s > 0.f) || !(s < kPosInf) || m != m) {
        atomicOr(p.status, MDS_ST_NONFINITE);
        if (m != m || m == kNegInf) m = 0.f;
        if (!(s > 0.f) || s != s) s = 1.f;
      }
      S.M[r] = m;
      S.invZ[r] = __frcp_rn(s);
    }
    __syncthreads();
  }

  // ---------------------------------------------------------------- residual / CDF sampling
  // Inverse-CDF draw over this sequence's vocabulary from the nonnegative
  // weights rf(u, r[VE]) in token order: the smallest token whose running sum
  // exceeds u * (total).  Sums are formed per 32-unit segment (lane partial
  // sums, warp inclusive scan), segments in order per CTA, CTAs in rank order;
  // the search re-walks the same sums.  Returns the token (cluster-uniform)
  // and the total mass in *total.
  template <class RF>
  __device__ int sample_cdf(const RF& rf, float u01, float* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int u0 = warp * 32; u0 < U; u0 += kThreads) {
      const int uu = u0 + lane;
      float part = 0.f;
      if (uu < U) {
        float r[VE];
        rf(uu, r);
#pragma unroll
        for (int e = 0; e < VE; ++e) part = __fadd_rn(part, r[e]);
      }
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float t = __shfl_up_sync(0xffffffffu, part, o);
        if (lane >= o) part = __fadd_rn(part, t);
      }
      if (lane == 31) segsum[u0 >> 5] = part;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.f;
      for (int g = 0; g < nseg; ++g) tot = __fadd_rn(tot, segsum[g]);
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
      int owner = -1;
      float run_owner = 0.f;
      int last = -1;
      float run_last = 0.f;
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
      S.T = T;
    }
    __syncthreads();
    const int owner = S.owner;
    if (rank == owner) {
      if (threadIdx.x == 0) {
        float run = S.run;
        int g = -1, glast = -1;
        float run_g = 0.f, run_last = 0.f;
        for (int h = 0; h < nseg; ++h) {
          if (segsum[h] > 0.f) {
            glast = h;
            run_last = run;
          }
          if (g < 0 && __fadd_rn(run, segsum[h]) > T) {
            g = h;
            run_g = run;
          }
          run = __fadd_rn(run, segsum[h]);
        }
        if (g < 0) {
          g = glast;
          run_g = run_last;
        }
        S.seg = g;
        S.run = run_g;
      }
      __syncthreads();
      if (warp == 0) {
        const int g = S.seg;
        const float base = S.run;
        const int uu = g * 32 + lane;
        float r[VE];
#pragma unroll
        for (int e = 0; e < VE; ++e) r[e] = 0.f;
        float part = 0.f;
        if (uu < U) {
          rf(uu, r);
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
        int l = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : 0);
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
          const int tok = min(tok0 + uu * VE + e_hit, p.V - 1);
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
      // adjacency (u -> v when pair {u,v} gives flow to u), sources, demands
      uint32_t adj[SM];
#pragma unroll
      for (int t = 0; t < SM; ++t) adj[t] = 0u;
      uint32_t srcm = 0u, dm = 0u, par = 0u;
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
#pragma unroll
      for (int t = 0; t < SM; ++t)
        if (t < s && rd[t] > eps) dm |= 1u << t;
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
  // and the Omega_2 masses: writes p_I on Omega_1 to S.om_x and the pair
  // weights to S.W (layout of pidx(., ., SM)), and returns the stage output
  // for the ordered inputs (A, B) and uniform u.  Single thread.
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
#pragma unroll
    for (int i = 0; i < SM; ++i) {
#pragma unroll
      for (int j = i + 1; j < SM; ++j) {
        if (j >= s) continue;
        const int e = pidx(i, j, SM);
        const float m = __fadd_rn(__fmul_rn(ak[i], bk[j]), __fmul_rn(ak[j], bk[i]));
        const float half = __fmul_rn(0.5f, RS[e]);
        const float to_i = __fadd_rn(FL[e], half), to_j = __fadd_rn(FH[e], half);
        x[i] = __fadd_rn(x[i], to_i);
        x[j] = __fadd_rn(x[j], to_j);
        S.W[e] = m > 0.f ? __fdiv_rn(to_i, m) : 0.5f;
      }
    }
#pragma unroll
    for (int t = 0; t < SM; ++t) S.om_x[t] = x[t];
    int pa = -1, pb = -1;
    for (int t = 0; t < s; ++t) {
      if (S.om[t] == A) pa = t;
      if (S.om[t] == Btok) pb = t;
    }
    if (A == Btok) return A;
    if (pa >= 0 && pb >= 0) {
      const int e = pidx(pa, pb, SM);
      const float wa = (pa < pb) ? S.W[e] : __fsub_rn(1.f, S.W[e]);
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
    for (int uu = threadIdx.x; uu < U; uu += kThreads) {
      const int tbase = tok0 + uu * VE;
      if (tbase >= p.V) break;
      float q[VE], a[VE], bb[VE];
      {
        float v[VE];
        E::unit(srow(0), uu, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = 0.f;
      for (int r = 1; r < nr; ++r) {
        const float g = S.gamma[r];
        if (g == 0.f && r != rb) continue;
        float v[VE];
        E::unit(srow(r), uu, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float pr = prob_of(v[e], S.M[r], S.c[r], S.invZ[r]);
          if (g != 0.f) a[e] = __fmaf_rn(g, pr, a[e]);
          if (r == rb) bb[e] = pr;
        }
      }
      const uint32_t bits = (bitmap[(uu * VE) >> 5] >> ((uu * VE) & 31)) & ((1u << VE) - 1u);
      if (bits) {
#pragma unroll
        for (int e = 0; e < VE; ++e)
          if (bits >> e & 1u) a[e] = special_lookup(tbase + e, a[e]);
      }
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        if (tbase + e >= p.V) break;
        cand_insert(top, Cand{__fmaf_rn(-a[e], bb[e], q[e]), tbase + e, a[e], bb[e]}, suma, sumb);
      }
    }
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
      if (loc >= 0 && loc < p.slice) atomicOr(&bitmap[loc >> 5], 1u << (loc & 31));
    }
    __syncthreads();
    return S.Y;
  }

  // ---------------------------------------------------------------- WIS: candidate list
  // Softmax statistics for a WIS depth with more than one valid draft, plus
  // the candidate list C = {k : q_k >= q_max 2^-kCandLog2} gathered to every
  // CTA in token order.  Every stage key q - a b is <= q, so whenever the
  // s-th best key in C exceeds the largest q outside C, Omega_1 lies in C and
  // the stage can run on C alone.  Two cluster exchanges: the row maxima,
  // then the per-CTA exp sums (split into candidates and complement) and the
  // candidate counts.  Units are mapped to warps in contiguous chunks so the
  // candidates come out in token order with a single block barrier.
  __device__ void wis_prepare() {
    const int nr = S.nrows;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // pass A: maxima; then, against this CTA's target max (<= the global
    // max, so these are upper bounds), counts of tokens at each candidate level
    for (int r = 0; r < nr; ++r) {
      float m = kNegInf;
      for (int u = threadIdx.x; u < U; u += kThreads) {
        float v[VE];
        E::unit(srow(r), u, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) m = fmaxf(m, v[e]);
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      if (lane == 0) S.red[warp * kMaxRows + r] = m;
    }
    __syncthreads();
    float mcta = kNegInf;
    for (int w = 0; w < kWarps; ++w) mcta = fmaxf(mcta, S.red[w * kMaxRows]);
    int lc[kCandLevels];
#pragma unroll
    for (int l = 0; l < kCandLevels; ++l) lc[l] = 0;
    if (mcta > kNegInf) {
      const float c0 = S.c[0];
      for (int u = threadIdx.x; u < U; u += kThreads) {
        if (tok0 + u * VE >= p.V) break;
        float v[VE];
        E::unit(srow(0), u, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float x = __fmul_rn(__fsub_rn(v[e], mcta), c0);
#pragma unroll
          for (int l = 0; l < kCandLevels; ++l) lc[l] += (x >= -cand_log2(l)) ? 1 : 0;
        }
      }
    }
#pragma unroll
    for (int l = 0; l < kCandLevels; ++l) lc[l] = __reduce_add_sync(0xffffffffu, lc[l]);
    if (lane == 0)
#pragma unroll
      for (int l = 0; l < kCandLevels; ++l) S.wlev[warp * kCandLevels + l] = lc[l];
    __syncthreads();
    if (threadIdx.x < nr) {
      float m = kNegInf;
      for (int w = 0; w < kWarps; ++w) m = fmaxf(m, S.red[w * kMaxRows + threadIdx.x]);
      S.xch[xbuf][threadIdx.x] = m;
    }
    if (threadIdx.x < kCandLevels) {
      int c = 0;
      for (int w = 0; w < kWarps; ++w) c += S.wlev[w * kCandLevels + threadIdx.x];
      S.xch[xbuf][nr + threadIdx.x] = __int_as_float(c);
    }
    const int n1 = nr + kCandLevels;
    cluster_gather(S, n1, xbuf, cn);
    if (threadIdx.x < nr) {
      float m = kNegInf;
      for (int q = 0; q < cn; ++q) m = fmaxf(m, S.gat[q * n1 + threadIdx.x]);
      if (!(m > kNegInf) || m != m) {
        atomicOr(p.status, MDS_ST_NONFINITE);
        m = 0.f;
      }
      S.M[threadIdx.x] = m;
    }
    // the most permissive level whose bounded counts fit the lists
    int level = -1;
    if (p.cand_cap > 0) {
      for (int l = 0; l < kCandLevels && level < 0; ++l) {
        int tot = 0, worst = 0;
        for (int q = 0; q < cn; ++q) {
          const int c = __float_as_int(S.gat[q * n1 + nr + l]);
          tot += c;
          worst = max(worst, c);
        }
        if (tot <= p.cand_cap && worst <= p.cand_cap_cta) level = l;
      }
    }
    __syncthreads();
    const float xthr = (level >= 0) ? -cand_log2(level) : 0.f;   // level < 0: no list (overflow)
    // pass B over this warp's chunk: exp sums split by candidacy, counts
    const int chunk = ((U + kWarps - 1) / kWarps + 31) & ~31;
    const int ubeg = min(U, warp * chunk), uend = min(U, ubeg + chunk);
    const float M0 = S.M[0], c0 = S.c[0];
    float comp[kFastRows], cand[kFastRows];
#pragma unroll
    for (int r = 0; r < kFastRows; ++r) comp[r] = cand[r] = 0.f;
    int cnt = 0;
    for (int u = ubeg + lane; u < uend; u += 32) {
      float x0[VE];
      {
        float v[VE];
        E::unit(srow(0), u, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) x0[e] = __fmul_rn(__fsub_rn(v[e], M0), c0);
      }
      uint32_t isc = 0u;
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        const bool c = (level >= 0) && (x0[e] >= xthr) && (tok0 + u * VE + e < p.V);
        isc |= (c ? 1u : 0u) << e;
        const float ex = ex2(x0[e]);
        if (c) cand[0] += ex; else comp[0] += ex;
      }
      cnt += __popc(isc);
#pragma unroll
      for (int r = 1; r < kFastRows; ++r) {
        if (r >= nr) break;
        const float Mr = S.M[r], cr = S.c[r];
        float v[VE];
        E::unit(srow(r), u, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) {
          const float ex = ex2(__fmul_rn(__fsub_rn(v[e], Mr), cr));
          if (isc >> e & 1u) cand[r] += ex; else comp[r] += ex;
        }
      }
    }
#pragma unroll
    for (int r = 0; r < kFastRows; ++r) {
      comp[r] = warp_sum(comp[r]);
      cand[r] = warp_sum(cand[r]);
    }
    const int wtot = __reduce_add_sync(0xffffffffu, cnt);
    if (lane == 0) {
      S.wcnt[warp] = wtot;
#pragma unroll
      for (int r = 0; r < kFastRows; ++r) {
        S.red[(warp * kFastRows + r) * 2] = comp[r];
        S.red[(warp * kFastRows + r) * 2 + 1] = cand[r];
      }
    }
    __syncthreads();
    int woff = 0, total = 0;
    for (int w = 0; w < kWarps; ++w) {
      if (w < warp) woff += S.wcnt[w];
      total += S.wcnt[w];
    }
    // candidate write pass (compare-only; exps just for the candidates)
    if (level >= 0 && total <= p.cand_cap_cta && wtot > 0) {
      int run = woff;
      for (int u = ubeg + lane; u - lane < uend; u += 32) {
        float v0[VE];
        uint32_t isc = 0u;
        if (u < uend) {
          E::unit(srow(0), u, v0);
#pragma unroll
          for (int e = 0; e < VE; ++e)
            isc |= ((__fmul_rn(__fsub_rn(v0[e], M0), c0) >= xthr && tok0 + u * VE + e < p.V) ? 1u : 0u) << e;
        }
        const int c = __popc(isc);
        int inc = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int t = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += t;
        }
        if (c) {
          int pos = run + inc - c;
#pragma unroll
          for (int e = 0; e < VE; ++e) {
            if (!(isc >> e & 1u)) continue;
            cl_id[pos] = tok0 + u * VE + e;
            cl_e[pos] = ex2(__fmul_rn(__fsub_rn(v0[e], M0), c0));
            for (int r = 1; r < nr; ++r) {
              float v[VE];
              E::unit(srow(r), u, v);
              cl_e[r * p.cand_cap_cta + pos] = ex2(__fmul_rn(__fsub_rn(v[e], S.M[r]), S.c[r]));
            }
            ++pos;
          }
        }
        run += __shfl_sync(0xffffffffu, inc, 31);
      }
    }
    if (threadIdx.x < kFastRows) {
      float a0 = 0.f, a1 = 0.f;
      for (int w = 0; w < kWarps; ++w) {
        a0 = __fadd_rn(a0, S.red[(w * kFastRows + threadIdx.x) * 2]);
        a1 = __fadd_rn(a1, S.red[(w * kFastRows + threadIdx.x) * 2 + 1]);
      }
      S.xch[xbuf][2 * threadIdx.x] = a0;
      S.xch[xbuf][2 * threadIdx.x + 1] = a1;
    }
    if (threadIdx.x == 0) S.xch[xbuf][2 * kFastRows] = __int_as_float(total);
    const int nx = 2 * kFastRows + 1;
    cluster_gather(S, nx, xbuf, cn);   // also publishes cl_* to the cluster
    // totals, complement masses, the merged list (every CTA, rank order)
    int ntot = 0, overflow = level >= 0 ? 0 : 1;
    for (int q = 0; q < cn; ++q) {
      const int c = __float_as_int(S.gat[q * nx + 2 * kFastRows]);
      if (c > p.cand_cap_cta) overflow = 1;
      ntot += c;
    }
    if (ntot > p.cand_cap) overflow = 1;
    if (threadIdx.x < nr) {
      const int r = threadIdx.x;
      float comp_t = 0.f, cand_t = 0.f;
      for (int q = 0; q < cn; ++q) {
        comp_t = __fadd_rn(comp_t, S.gat[q * nx + 2 * r]);
        cand_t = __fadd_rn(cand_t, S.gat[q * nx + 2 * r + 1]);
      }
      const float Z = __fadd_rn(comp_t, cand_t);
      if (!(Z > 0.f) || !(Z < kPosInf)) atomicOr(p.status, MDS_ST_NONFINITE);
      S.invZ[r] = (Z > 0.f && Z < kPosInf) ? __frcp_rn(Z) : 1.f;
      S.pc[r] = comp_t;                  // complement exp mass (times invZ: probability)
    }
    if (!overflow) {
      int off = 0;
      for (int q = 0; q < cn; ++q) {
        const int c = __float_as_int(S.gat[q * nx + 2 * kFastRows]);
        for (int i = threadIdx.x; i < c; i += kThreads) {
          if (cn > 1) {
            cm_id[off + i] = __float_as_int(ld_dsmem(reinterpret_cast<const float*>(cl_id) + i, (uint32_t)q));
            for (int r = 0; r < nr; ++r)
              cm_e[r * p.cand_cap + off + i] = ld_dsmem(cl_e + r * p.cand_cap_cta + i, (uint32_t)q);
          } else {
            cm_id[off + i] = cl_id[i];
            for (int r = 0; r < nr; ++r) cm_e[r * p.cand_cap + off + i] = cl_e[r * p.cand_cap_cta + i];
          }
          cm_sp[off + i] = 0;
          cm_a[off + i] = 0.f;
        }
        off += c;
      }
    }
    if (threadIdx.x == 0) {
      S.ncand = overflow ? -1 : ntot;
      S.cand_all = (!overflow && ntot == p.V) ? 1 : 0;
      S.cand_q = (level >= 0) ? ex2(xthr) : 0.f;   // every non-candidate has q < cand_q / Z
    }
    __syncthreads();
    // Other CTAs read this CTA's cl_* right after the exchange; the next write
    // to cl_* is a depth later, behind at least one more cluster barrier.
  }

  // One stage on the merged candidate list, by warp 0 of every CTA.
  // Returns false (and changes nothing) if the list cannot certify Omega_1.
  __device__ bool wis_stage_fast(int A, int Btok, int rb, float u) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int s = min(p.wis_s, p.V);
    const int n = S.ncand;
    if (warp == 0) {
      Cand top[kTop];
#pragma unroll
      for (int t = 0; t < kTop; ++t) top[t] = CAND_NONE;
      float suma = 0.f, sumb = 0.f;
      const float iz0 = S.invZ[0], izb = S.invZ[rb];
      for (int i = lane; i < n; i += 32) {
        const float q = __fmul_rn(cm_e[i], iz0);
        float a;
        if (cm_sp[i]) {
          a = cm_a[i];
        } else {
          a = 0.f;
          for (int r = 1; r < S.nrows; ++r)
            if (S.gamma[r] != 0.f) a = __fmaf_rn(S.gamma[r], __fmul_rn(cm_e[r * p.cand_cap + i], S.invZ[r]), a);
        }
        const float b = __fmul_rn(cm_e[rb * p.cand_cap + i], izb);
        cand_insert(top, Cand{__fmaf_rn(-a, b, q), i, a, b}, suma, sumb);   // id: list index (token order)
      }
      float ra, rbs;
      warp_merge(top, S.fin, s, ra, rbs);
      suma = warp_sum(suma);
      sumb = warp_sum(sumb);
      if (lane == 0) {
        // certification: s candidates, and the s-th key above every key
        // outside the list (each such key is <= q < 2^-level / Z)
        const float qout = __fmul_rn(__fmul_rn(S.cand_q, iz0), 1.0001f);
        const bool ok = (n >= s) && (S.cand_all || S.fin[s - 1].key > qout);
        S.fast_ok = ok ? 1 : 0;
        if (ok) {
          // Omega_2 masses: complement (generic law) + candidates outside Omega_1
          float sa = 0.f;
          for (int r = 1; r < S.nrows; ++r)
            if (S.gamma[r] != 0.f) sa = __fmaf_rn(S.gamma[r], __fmul_rn(S.pc[r], S.invZ[r]), sa);
          float sb = __fmul_rn(S.pc[rb], izb);
          sa = __fadd_rn(sa, __fadd_rn(suma, ra));
          sb = __fadd_rn(sb, __fadd_rn(sumb, rbs));
          omega1_sorted(S.fin, s);   // list indices, increasing = token order
          int oi[MDS_MAX_S];
#pragma unroll
          for (int t = 0; t < MDS_MAX_S; ++t) {
            oi[t] = (t < s) ? S.om[t] : -1;
            const int ii = (t < s) ? oi[t] : 0;
            S.om[t] = (t < s) ? cm_id[ii] : -1;      // token ids for the solve
            S.om_q[t] = (t < s) ? __fmul_rn(cm_e[ii], iz0) : 0.f;
          }
          S.Y = stage_solve(s, sa, sb, A, Btok, u);
#pragma unroll
          for (int t = 0; t < MDS_MAX_S; ++t) S.om[t] = oi[t];   // back to list indices
          S.A2 = sa;
          S.B2 = sb;
        }
      }
      __syncwarp();
      if (S.fast_ok) {
        // law update on the list: specials outside Omega_1, then Omega_1
        const float A2 = S.A2, B2 = S.B2;
        for (int i = lane; i < n; i += 32) {
          int t1 = -1;
          for (int t = 0; t < s; ++t)
            if (S.om[t] == i) t1 = t;
          if (t1 >= 0) {
            cm_a[i] = S.om_x[t1];
            cm_sp[i] = 1;
          } else if (cm_sp[i]) {
            const float b = __fmul_rn(cm_e[rb * p.cand_cap + i], izb);
            cm_a[i] = __fmul_rn(0.5f, __fadd_rn(__fmul_rn(cm_a[i], B2), __fmul_rn(b, A2)));
          }
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
      if (loc >= 0 && loc < p.slice) atomicOr(&bitmap[loc >> 5], 1u << (loc & 31));
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
    for (int uu = threadIdx.x; uu < U; uu += kThreads) {
      float q[VE];
      {
        float v[VE];
        E::unit(srow(0), uu, v);
#pragma unroll
        for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
      }
      for (int r = 1; r < S.nrows; ++r) {
        if (!S.is_cnt[r]) continue;
        float v[VE];
        E::unit(srow(r), uu, v);
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
    }
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
      S.rho_min = rlo;
      S.rho_max = rhi;
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
        for (int uu = threadIdx.x; uu < U; uu += kThreads) {
          float q[VE], pr[VE];
          {
            float v[VE];
            E::unit(srow(0), uu, v);
#pragma unroll
            for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
            E::unit(srow(r), uu, v);
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
        }
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
  __device__ void run_sequence(int b) {
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
        S.flags = 0;
        S.R = 0.f;
      }
      __syncthreads();
      load_rows();
      if (SCHEME == MDS_WIS && !bonus && S.nv > 1 && S.nrows <= kFastRows)
        wis_prepare();
      else
        row_stats();
      if (threadIdx.x == 0 && !(SCHEME == MDS_WIS && !bonus && S.nv > 1 && S.nrows <= kFastRows)) S.ncand = -1;
      int Z;
      float qY = 0.f, pIY = 0.f, Rdiag = 0.f;
      int Ydiag = -1;
      if (bonus) {
        float tot;
        Z = sample_cdf(
            [&](int uu, float* r) {
              float v[VE];
              E::unit(srow(0), uu, v);
#pragma unroll
              for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
            },
            draw_uniform(p.seed, b, j, kDrawBonus), &tot);
        Rdiag = tot;
      } else if constexpr (SCHEME == MDS_SPECTR) {
        Z = spectr(b, j, &qY, &pIY, &Ydiag, &Rdiag);
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
        if (uacc < fminf(1.f, ratio)) {
          Z = Y;
        } else {
          const float ures = draw_uniform(p.seed, b, j, kDrawResidual);
          float tot;
          bool done = false;
          if constexpr (SCHEME == MDS_WIS) {
            if (S.nv > 1) {
              Z = sample_cdf([&](int uu, float* r) { residual_wis(uu, r); }, ures, &tot);
              done = true;
            }
          }
          if constexpr (SCHEME == MDS_IS) {
            if (S.nv > 1) {
              Z = sample_cdf([&](int uu, float* r) { residual_is(uu, r); }, ures, &tot);
              done = true;
            }
          }
          if (!done) {
            const int r1 = S.vrow[0];
            Z = sample_cdf(
                [&](int uu, float* r) {
                  float v[VE], w[VE];
                  E::unit(srow(0), uu, v);
                  E::unit(srow(r1), uu, w);
#pragma unroll
                  for (int e = 0; e < VE; ++e)
                    r[e] = fmaxf(0.f, __fsub_rn(prob_of(v[e], S.M[0], S.c[0], S.invZ[0]),
                                                prob_of(w[e], S.M[r1], S.c[r1], S.invZ[r1])));
                },
                ures, &tot);
          }
          Rdiag = tot;
          if (Z < 0) {
            if (tid == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
            Z = sample_cdf(
                [&](int uu, float* r) {
                  float v[VE];
                  E::unit(srow(0), uu, v);
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
      p.out_accept[b] = acc_len;
      for (int j = acc_len + 1; j <= L; ++j) p.out_tokens[(size_t)b * (L + 1) + j] = -1;
    }
  }

  // residual weight max(0, q - p_I) for WIS (generic gamma law + special table)
  __device__ __forceinline__ void residual_wis(int uu, float* r) const {
    const int tbase = tok0 + uu * VE;
    float q[VE], a[VE];
    {
      float v[VE];
      E::unit(srow(0), uu, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) {
        q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
        a[e] = 0.f;
      }
    }
    for (int r = 1; r < S.nrows; ++r) {
      const float g = S.gamma[r];
      if (g == 0.f) continue;
      float v[VE];
      E::unit(srow(r), uu, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) a[e] = __fmaf_rn(g, prob_of(v[e], S.M[r], S.c[r], S.invZ[r]), a[e]);
    }
    const uint32_t bits = (bitmap[(uu * VE) >> 5] >> ((uu * VE) & 31)) & ((1u << VE) - 1u);
    if (bits) {
#pragma unroll
      for (int e = 0; e < VE; ++e)
        if (bits >> e & 1u) a[e] = special_lookup(tbase + e, a[e]);
    }
#pragma unroll
    for (int e = 0; e < VE; ++e) r[e] = fmaxf(0.f, __fsub_rn(q[e], a[e]));
  }

  // residual weight max(0, q - p_I) for plain IS (Laplace identity)
  __device__ __forceinline__ void residual_is(int uu, float* r) const {
    float q[VE];
    {
      float v[VE];
      E::unit(srow(0), uu, v);
#pragma unroll
      for (int e = 0; e < VE; ++e) q[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
    }
    float rho[VE][kMaxRows];
    for (int rr = 1; rr < S.nrows; ++rr) {
      if (!S.is_cnt[rr]) continue;
      float v[VE];
      E::unit(srow(rr), uu, v);
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
  __device__ int spectr(int b, int j, float* qY, float* pIY, int* Yd, float* Rd) {
    const int nv = S.nv;
    for (int i = 0; i < nv; ++i) {
      // point value of the running target at X_i
      if (threadIdx.x == 0) {
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
        S.sp_rows[i] = S.vrow[i];
      }
      __syncthreads();
      *qY = S.qY;
      *pIY = S.pIY;
      *Yd = S.X[0];
      if (S.accepted) {
        const int z = S.X[i];
        __syncthreads();
        return z;
      }
      // residual mass of this round
      float part = 0.f;
      const int ri = S.sp_rows[i];
      for (int uu = threadIdx.x; uu < U; uu += kThreads) {
        float r[VE];
        spectr_target(uu, i, r);
        float w[VE];
        E::unit(srow(ri), uu, w);
#pragma unroll
        for (int e = 0; e < VE; ++e) part += fmaxf(0.f, __fsub_rn(r[e], prob_of(w[e], S.M[ri], S.c[ri], S.invZ[ri])));
      }
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
      }
      __syncthreads();
    }
    float tot;
    const int z = sample_cdf([&](int uu, float* r) { spectr_target(uu, nv, r); },
                             draw_uniform(p.seed, b, j, kDrawResidual), &tot);
    *Rd = tot;
    return z;
  }

  // running target after `rounds` rejected rounds, for one unit
  __device__ __forceinline__ void spectr_target(int uu, int rounds, float* r) const {
    float v[VE];
    E::unit(srow(0), uu, v);
#pragma unroll
    for (int e = 0; e < VE; ++e) r[e] = prob_of(v[e], S.M[0], S.c[0], S.invZ[0]);
    for (int k = 0; k < rounds; ++k) {
      if (!(S.sp_invR[k] > 0.f)) continue;
      const int rk = S.sp_rows[k];
      float w[VE];
      E::unit(srow(rk), uu, w);
#pragma unroll
      for (int e = 0; e < VE; ++e)
        r[e] = __fmul_rn(fmaxf(0.f, __fsub_rn(r[e], prob_of(w[e], S.M[rk], S.c[rk], S.invZ[rk]))), S.sp_invR[k]);
    }
  }
};

template <int DT, int SCHEME>
__global__ void __launch_bounds__(kThreads, SCHEME == MDS_IS ? 1 : 3) verify_kernel(const __grid_constant__ Params p) {
  extern __shared__ __align__(128) char dsm[];
  __shared__ State S;
  Kernel<DT, SCHEME> k{p, S};
  k.rank = (int)cluster_rank();
  k.cn = p.cn;
  k.tok0 = k.rank * p.slice;
  k.nvalid = max(0, min(p.slice, p.V - k.tok0));
  k.U = p.slice / Kernel<DT, SCHEME>::VE;
  k.nseg = (k.U + 31) / 32;
  k.bm_words = (p.slice + 31) / 32;
  // dynamic shared memory: rows | segment sums | scheme region
  //   IS : nodes t_n | weights W_r(n)
  //   WIS: this CTA's candidate list | merged list, aliased later by the
  //        special-token bitmap (the merged list is local; other CTAs only
  //        ever read the CTA list)
  k.rows = dsm;
  k.segsum = reinterpret_cast<float*>(dsm + (size_t)p.rows_max * p.row_stride);
  {
    char* c = reinterpret_cast<char*>(k.segsum + ((k.nseg + 3) & ~3));
    k.isT = reinterpret_cast<float*>(c);
    k.isW = k.isT + kIsNodesMax;
    k.cl_id = reinterpret_cast<int*>(c);
    c += (size_t)p.cand_cap_cta * 4;
    k.cl_e = reinterpret_cast<float*>(c);
    c += (size_t)p.cand_cap_cta * p.rows_max * 4;
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
  k.mphase = 0u;
  if (threadIdx.x == 0) mbar_init(&S.mbar);
  __syncthreads();
  for (;;) {
    if (k.rank == 0 && threadIdx.x == 0) {
      const int b = (int)(atomicAdd(p.queue, 1u) - p.ticket0);
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
    k.run_sequence(b);
  }
}

}  // namespace

size_t smem_bytes(const Params& p) {
  const int VE = 16 / p.esize;
  const int U = p.slice / VE;
  const int nseg = (U + 31) / 32;
  size_t bytes = (size_t)p.rows_max * p.row_stride + (size_t)((nseg + 3) & ~3) * 4;
  if (p.scheme == MDS_IS) bytes += (size_t)kIsNodesMax * 4 * (1 + p.rows_max);
  if (p.scheme == MDS_WIS) {
    const size_t bm = (size_t)((p.slice + 31) / 32) * 4;
    const size_t cm = (size_t)p.cand_cap * 4 * (3 + p.rows_max);
    bytes += (size_t)p.cand_cap_cta * 4 * (1 + p.rows_max) + (bm > cm ? bm : cm);
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
      default: return verify_kernel<MDS_F32, MDS_SINGLE>;
    }
  }
  switch (scheme) {
    case MDS_IS: return verify_kernel<MDS_BF16, MDS_IS>;
    case MDS_WIS: return verify_kernel<MDS_BF16, MDS_WIS>;
    case MDS_SPECTR: return verify_kernel<MDS_BF16, MDS_SPECTR>;
    default: return verify_kernel<MDS_BF16, MDS_SINGLE>;
  }
}

cudaError_t configure_kernel(int dtype) {
  int dev = 0, optin = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  for (int scheme = MDS_SINGLE; scheme <= MDS_SPECTR; ++scheme) {
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
