// Device helpers of the slice-dataflow engine (mds_flow.cu) and the top-k
// kernel (mds_topk.cu): inline PTX wrappers, the counter-based random
// numbers, logit IO, the exponent convention of every probability, and the
// stage maximum flow of the weighted scheme.  Not part of the public ABI.
#pragma once
#include <cuda_bf16.h>

#include <cstdint>

#include "mds_internal.h"

namespace mds {
namespace dev {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kNegInf = -__builtin_huge_valf();
constexpr float kPosInf = __builtin_huge_valf();
constexpr int kLpMaxAugment = 4096;     // augmenting paths one stage LP may take
constexpr float kLpEpsRel = 1e-6f;      // LP residuals below this share of the stage's mass count as zero
constexpr int kMaxPairs = MDS_MAX_S * (MDS_MAX_S - 1) / 2;

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
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count = 1) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_init_fence() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
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
// Bulk copy global -> this CTA's shared memory, completion counted on `bar`.
// Both addresses 16-byte aligned, `bytes` a multiple of 16.
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
// Uniform of draw `draw` at (sequence b, depth j): counter (b, j, draw, 0),
// key (seed low, seed high), value (word0 >> 8) * 2^-24 in [0, 1).
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
  // Largest logit of a unit (NaN entries are ignored unless all are NaN).
  __device__ static __forceinline__ float unit_max(const uint4& x) {
    return fmaxf(fmaxf(__uint_as_float(x.x), __uint_as_float(x.y)), fmaxf(__uint_as_float(x.z), __uint_as_float(x.w)));
  }
  static constexpr uint32_t kNegInfBits = 0xff800000u;   // one logit of -inf
};
template <>
struct Elt<MDS_BF16> {
  static constexpr int VE = 8;
  __device__ static __forceinline__ void unit(const char* row, int u, float* v) {
    const uint4 x = *reinterpret_cast<const uint4*>(row + 16 * u);
    unpack(x, v);
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
    unpack(__ldg(reinterpret_cast<const uint4*>(at)), v);
  }
  // Packed bf16x2 maxima (exact: the maximum of bf16 values is one of them).
  __device__ static __forceinline__ float unit_max(const uint4& x) {
    uint32_t m;
    asm("{\n\t.reg .b32 t0, t1;\n\t"
        "max.bf16x2 t0, %1, %2;\n\t"
        "max.bf16x2 t1, %3, %4;\n\t"
        "max.bf16x2 %0, t0, t1;\n\t}"
        : "=r"(m)
        : "r"(x.x), "r"(x.y), "r"(x.z), "r"(x.w));
    return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
  }
  static constexpr uint32_t kNegInfBits = 0xff80ff80u;   // two logits of -inf
};

// Probability of a logit under a row's statistics (row maximum M, scale
// c = log2(e) / T, inverse normaliser).  The same expression serves every
// in-pass value and point lookup, so both give identical bits.  Exponents:
// a term is 2^fma(l, c, -round(M c)) (one rounding, l c exact inside the
// FMA); a partial sum moves from reference m to M by the factor
// 2^(round(m c) - round(M c)), so every term of a row shares one reference.
__device__ __forceinline__ float prob_of(float l, float M, float c, float invZ) {
  return __fmul_rn(ex2(__fmaf_rn(l, c, -__fmul_rn(M, c))), invZ);
}
// Unnormalised term of a logit against reference m (the row or slice maximum).
__device__ __forceinline__ float exp_term(float l, float m, float c) { return ex2(__fmaf_rn(l, c, -__fmul_rn(m, c))); }
// Factor that moves a sum from reference m to reference M >= m.
__device__ __forceinline__ float ref_shift(float m, float M, float c) {
  return ex2(__fsub_rn(__fmul_rn(m, c), __fmul_rn(M, c)));
}

// Combine two (max, sum) pairs of one row.
__device__ __forceinline__ void combine_ms(float& m, float& s, float m2, float s2, float c) {
  const float M = fmaxf(m, m2);
  const float a = (m == kNegInf) ? 0.f : __fmul_rn(s, ref_shift(m, M, c));
  const float b = (m2 == kNegInf) ? 0.f : __fmul_rn(s2, ref_shift(m2, M, c));
  m = M;
  s = __fadd_rn(a, b);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ------------------------------------------------------------------ stage LP

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

// Maximum flow of one stage of the weighted scheme on the pair/token
// network of its s-variable LP (appendix "Variant of Truncated LP"; the
// non-iid appendix for the pair masses): pair e = {i, j} of Omega_1 (tokens
// in increasing id) has supply RS[e] = a_i b_j + a_j b_i, token t has demand
// rd[t] = (q_t - base_t)+.  The flow is fixed by this order:
//   (a) a direct pass over the pairs (i, j), i < j, lexicographically: each
//       gives what it can to token i (FL), then to token j (FH);
//   (b) breadth-first augmenting paths in token space: sources are the
//       tokens of pairs with supply left, each with the first such pair;
//       u -> v when pair {u, v} gives flow to u; levels in increasing token
//       order, a token's parent the first frontier token reaching it; the
//       path ends at the first token with demand left;
//   (c) the caller splits the leftover pair mass 1/2 - 1/2.
// Residuals <= eps count as zero.  SM is the compile-time token capacity (all
// state in registers indexed by compile-time constants).  One thread.
// Returns false if the augmentation cap was reached.
template <int SM>
__device__ __forceinline__ bool lp_maxflow(int s, float (&rd)[SM], float (&RS)[SM * (SM - 1) / 2],
                                           float (&FL)[SM * (SM - 1) / 2], float (&FH)[SM * (SM - 1) / 2],
                                           float eps) {
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
    if (!dm) return true;
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
    if (!srcm) return true;
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
    if (!hit) return true;
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
  return false;
}

// One stage of the weighted scheme given Omega_1 (om[0..s), increasing
// token ids; entries past s ignored) with q, a, b at those tokens and the
// Omega_2 masses A2 = a(Omega_2), B2 = b(Omega_2).  Writes p_I on Omega_1 to
// om_x and returns the stage output for the ordered inputs (A, B) and
// uniform u: equal inputs give A; inputs both in Omega_1 select A with
// probability w_{AB} (flow plus half the leftover pair mass, over the pair
// mass); exactly one in Omega_1 gives that one; both in Omega_2 select A
// with probability 1/2.  *capped reports an LP that hit its cap.  One thread.
// The pair state (RS, FL, FH) lives where the caller puts it: registers for
// SM = 5, shared memory for larger SM.
template <int SM>
__device__ __forceinline__ int stage_solve(int s, float A2, float B2, int A, int Btok, float u, const int* om,
                                           const float* om_q, const float* om_a, const float* om_b, float* om_x,
                                           bool* capped, float (&RS)[SM * (SM - 1) / 2], float (&FL)[SM * (SM - 1) / 2],
                                           float (&FH)[SM * (SM - 1) / 2]) {
  constexpr int P = SM * (SM - 1) / 2;
  float ak[SM], bk[SM], x[SM], rd[SM];
  float eps = 0.f;
#pragma unroll
  for (int t = 0; t < SM; ++t) {
    ak[t] = om_a[t];
    bk[t] = om_b[t];
    const float qk = om_q[t];
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
  *capped = !lp_maxflow<SM>(s, rd, RS, FL, FH, eps);
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
  for (int t = 0; t < SM; ++t) om_x[t] = x[t];
  if (A == Btok) return A;
  int pa = -1, pb = -1;
#pragma unroll
  for (int t = 0; t < SM; ++t) {
    if (t < s && om[t] == A) pa = t;
    if (t < s && om[t] == Btok) pb = t;
  }
  if (pa >= 0 && pb >= 0) {
    const int lo = min(pa, pb), hi = max(pa, pb);
    const int e = pidx(lo, hi, SM);
    float fl = 0.f, rs = 0.f, alo = 0.f, ahi = 0.f, blo = 0.f, bhi = 0.f;
#pragma unroll
    for (int k = 0; k < P; ++k)
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

}  // namespace dev
}  // namespace mds
