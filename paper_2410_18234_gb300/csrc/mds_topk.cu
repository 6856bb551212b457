// Top-k restricted verification: Section 5 runs every scheme on rows
// restricted to their k most probable tokens (k = 5 and 10, Tables 2 and 3),
// renormalised.  The restriction leaves a depth's laws on the union U of the
// rows' kept tokens, at most (1 + models) * k of them, so one pass over each
// visited row (the top-k selection) is the only full-vocabulary work and the
// scheme itself runs on U:
//   * single draft: Algorithm 1 with p_I the first valid branch's law;
//   * WIS: the pairwise stages (Remark 4) of the variant truncated LP
//     (appendix "Variant of Truncated LP"), Omega_1 the s largest keys
//     q - a b over the whole vocabulary (ties to the lower id): the positive
//     keys of U, then zero keys (tokens outside U and tokens of U with a zero
//     key) by increasing id, then negative keys;
//   * WIS with the sorted rule on Omega_2 (Section 4 Eq. heur, Eq. p_Ieq):
//     the same stages, a pair inside Omega_2 selecting the token earlier in
//     key order; its Omega_2 law needs each token's key-ordered suffix
//     masses, a sum over U;
//   * SpecTr: sequential rejection over the valid drafts.
// Tokens outside U carry zero mass in every law, so the inverse CDFs in
// token-id order (residual, bonus) run over U sorted by id.
//
// One CTA of 256 threads verifies one sequence.  Per depth: warp 0 plans the
// rows (the target row of the lowest valid branch, one draft row per model
// among the valid branches, read from its lowest valid branch; the single
// draft step reads only the first valid branch's).  For each row, every
// thread first takes the maximum of its first units; the k-th largest of
// those maxima bounds the row's k-th logit from below.  Then every thread
// scans its strided share of the row, keeping a sorted list of its 16
// largest (logit, -id) keys at or above that bound, and the warps merge the
// lists into the row's top k.  Warp 0 then computes the kept entries'
// probabilities, the union, the scheme's decision and the walk.
#include "mds_device.cuh"
#include "mds_topk.h"

namespace mds {
namespace topk {
namespace {

using namespace mds::dev;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kKMax = MDS_MAX_TOPK;
constexpr int kRowsMax = 1 + MDS_MAX_K;
constexpr int kEntMax = kRowsMax * kKMax;   // kept entries of one depth, and the largest |U|
constexpr unsigned FULL = 0xffffffffu;
constexpr int kPrefixUnits = 4;             // units per thread behind a row's first logit bound

static_assert(kWarps * kKMax == 4 * 32, "the row merge holds four candidates per lane");
static_assert(kKMax <= 32, "a row's kept entries fit one warp");

struct Shared {
  unsigned long long wk[kWarps][kKMax];   // each warp's top k of a row
  int id[kRowsMax][kKMax];                // each row's kept tokens, decreasing (logit, -id)
  float lg[kRowsMax][kKMax];              // their logits
  float pr[kRowsMax][kKMax];              // their renormalised probabilities
  int n[kRowsMax];                        // kept entries per row
  const char* rowp[kRowsMax];             // row pointers of the depth
  float rowc[kRowsMax];                   // log2(e) / T of each row
  int nrows;
  // the union U of the kept tokens by increasing id, each row's law on it
  int uid[kEntMax];
  float law[kRowsMax][kEntMax];
  float cur[kEntMax];                     // running law (stage output law, SpecTr target)
  float key[kEntMax];                     // stage keys q - a b
  float nxt[kEntMax];                     // the sorted rule's Omega_2 law, before it replaces cur
  unsigned char in1[kEntMax];             // U entry is in Omega_1 of the current stage
  short rank[kEntMax];                    // position in U of each kept entry
  unsigned char dup[kEntMax];             // entry repeats a token of an earlier entry
  int nU;
  // the walk
  int X[MDS_MAX_K], vbr[MDS_MAX_K], vrow[MDS_MAX_K];
  int nv;
  unsigned valid;
  int done;
  // one stage: Omega_1 by increasing id, its values, the pair state
  int om[MDS_MAX_S];
  unsigned char om_in[MDS_MAX_S];         // the Omega_1 token is in U (index om_u)
  short om_u[MDS_MAX_S];
  float om_q[MDS_MAX_S], om_a[MDS_MAX_S], om_b[MDS_MAX_S], om_x[MDS_MAX_S];
  float RS[kMaxPairs], FL[kMaxPairs], FH[kMaxPairs];
  int Y;
  int bcast;                              // warp 0's broadcast word
  float tau0;                             // lower bound on a row's kk-th logit
  // bonus: the target row's kept entries by increasing id
  int bid[kKMax];
  float bw[kKMax];
};

__device__ __forceinline__ unsigned long long max_u64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}
__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = max_u64(v, __shfl_xor_sync(FULL, v, o));
  return v;
}
// A kept entry's key: larger logit first, then lower id.  Never 0 (ids are
// below 2^24), so 0 marks an empty slot.
__device__ __forceinline__ unsigned long long entry_key(float v, int id) {
  return ((unsigned long long)ord_key(v) << 32) | (unsigned long long)(0xffffffffu - (unsigned)id);
}
__device__ __forceinline__ int key_id(unsigned long long k) { return (int)(0xffffffffu - (unsigned)k); }
__device__ __forceinline__ float key_val(unsigned long long k) { return ord_val((unsigned)(k >> 32)); }

// A thread's running list: its 16 largest keys, decreasing; the k-th entry
// and its logit (or the row's known floor, if higher) bound what can still
// enter.  Every array is indexed by
// compile-time constants only (registers).
struct TopList {
  unsigned long long e[kKMax];
  unsigned long long kth;
  float bound;
  float floor;   // a lower bound on the row's kk-th logit known in advance

  __device__ __forceinline__ void reset() {
#pragma unroll
    for (int i = 0; i < kKMax; ++i) e[i] = 0ull;
    kth = 0ull;
    bound = kNegInf;
    floor = kNegInf;
  }
  __device__ __forceinline__ void insert(float v, int id, int kk) {
    unsigned long long x = entry_key(v, id);
    if (!(v >= bound) || x <= kth) return;
#pragma unroll
    for (int i = 0; i < kKMax; ++i) {
      const unsigned long long t = e[i];
      const bool sw = x > t;
      e[i] = sw ? x : t;
      x = sw ? t : x;
    }
#pragma unroll
    for (int i = 0; i < kKMax; ++i)
      if (i == kk - 1) kth = e[i];
    bound = kth ? fmaxf(floor, key_val(kth)) : floor;
  }
  // The values of one unit (n of them, ids base, base + 1, ...): a mask of
  // those at or above the bound, then one insertion site for the (rare) hits.
  template <int N>
  __device__ __forceinline__ void offer(const float (&v)[N], int base, int kk) {
    unsigned m = 0u;
#pragma unroll
    for (int i = 0; i < N; ++i) m |= (v[i] >= bound) ? (1u << i) : 0u;
    while (m) {
      const int i0 = __ffs(m) - 1;
      m &= m - 1u;
      float x = v[0];
#pragma unroll
      for (int i = 1; i < N; ++i)
        if (i == i0) x = v[i];
      insert(x, base + i0, kk);
    }
  }
  __device__ __forceinline__ void pop() {
#pragma unroll
    for (int i = 0; i + 1 < kKMax; ++i) e[i] = e[i + 1];
    e[kKMax - 1] = 0ull;
  }
};

template <int DT>
__device__ __forceinline__ void scan_unit(TopList& T, const uint4& x, int u, int kk) {
  using E = Elt<DT>;
  if (!(E::unit_max(x) >= T.bound)) return;
  float v[E::VE];
  E::unpack(x, v);
  T.offer<E::VE>(v, u * E::VE, kk);
}

// The row's top kk into S.id / S.lg / S.n[r] (all threads; ends synchronised).
template <int DT>
__device__ __noinline__ void select_row(const Params& p, Shared& S, int r, int kk) {
  using E = Elt<DT>;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const char* row = S.rowp[r];
  TopList T;
  T.reset();
  // A lower bound on the row's kk-th logit: the kk-th largest of the threads'
  // maxima over their first units (kk distinct logits reach it), so the
  // full scan below inserts only logits at or above it.
  {
    float mx = kNegInf;
    if (p.vec) {
      const uint4* rv = reinterpret_cast<const uint4*>(row);
      const int nu = (int)(((size_t)p.V * p.esize) / 16);
#pragma unroll
      for (int q = 0; q < kPrefixUnits; ++q)
        if (tid + q * kThreads < nu) mx = fmaxf(mx, E::unit_max(__ldcs(rv + tid + q * kThreads)));
    } else {
#pragma unroll
      for (int q = 0; q < kPrefixUnits; ++q)
        if (tid + q * kThreads < p.V) mx = fmaxf(mx, E::global(row, tid + q * kThreads));
    }
    // kk rounds of a warp maximum over (max, thread) keys, then over the warps'
    unsigned long long mk = (mx == mx && mx > kNegInf) ? entry_key(mx, tid) : 0ull;
    for (int t = 0; t < kk; ++t) {
      const unsigned long long m = warp_max_u64(mk);
      if (mk == m) mk = 0ull;
      if (lane == 0) S.wk[warp][t] = m;
    }
    __syncthreads();
    if (warp == 0) {
      unsigned long long c0, c1, c2, c3;
      const int e0 = lane, e1 = lane + 32, e2 = lane + 64, e3 = lane + 96;
      c0 = (e0 % kKMax < kk) ? S.wk[e0 / kKMax][e0 % kKMax] : 0ull;
      c1 = (e1 % kKMax < kk) ? S.wk[e1 / kKMax][e1 % kKMax] : 0ull;
      c2 = (e2 % kKMax < kk) ? S.wk[e2 / kKMax][e2 % kKMax] : 0ull;
      c3 = (e3 % kKMax < kk) ? S.wk[e3 / kKMax][e3 % kKMax] : 0ull;
      unsigned long long m = 0ull;
      for (int t = 0; t < kk; ++t) {
        m = warp_max_u64(max_u64(max_u64(c0, c1), max_u64(c2, c3)));
        if (m == 0ull) break;
        if (c0 == m) c0 = 0ull;
        if (c1 == m) c1 = 0ull;
        if (c2 == m) c2 = 0ull;
        if (c3 == m) c3 = 0ull;
      }
      // fewer than kk threads saw a logit: no bound
      if (lane == 0) S.tau0 = (m != 0ull) ? key_val(m) : kNegInf;
    }
    __syncthreads();
    T.floor = S.tau0;
    T.bound = S.tau0;
  }
  if (p.vec) {
    // 16-byte units, four in flight per thread
    const uint4* rv = reinterpret_cast<const uint4*>(row);
    const int nu = (int)(((size_t)p.V * p.esize) / 16);
    int u = tid;
    for (; u + 3 * kThreads < nu; u += 4 * kThreads) {
      const uint4 x0 = __ldcs(rv + u), x1 = __ldcs(rv + u + kThreads), x2 = __ldcs(rv + u + 2 * kThreads),
                  x3 = __ldcs(rv + u + 3 * kThreads);
      scan_unit<DT>(T, x0, u, kk);
      scan_unit<DT>(T, x1, u + kThreads, kk);
      scan_unit<DT>(T, x2, u + 2 * kThreads, kk);
      scan_unit<DT>(T, x3, u + 3 * kThreads, kk);
    }
    for (; u < nu; u += kThreads) scan_unit<DT>(T, __ldcs(rv + u), u, kk);
  } else {
    // element loads (rows of any length and alignment), four in flight
    int i = tid;
    for (; i + 3 * kThreads < p.V; i += 4 * kThreads) {
      const float v4[4] = {E::global(row, i), E::global(row, i + kThreads), E::global(row, i + 2 * kThreads),
                           E::global(row, i + 3 * kThreads)};
      unsigned m = 0u;
#pragma unroll
      for (int q = 0; q < 4; ++q) m |= (v4[q] >= T.bound) ? (1u << q) : 0u;
      while (m) {
        const int q0 = __ffs(m) - 1;
        m &= m - 1u;
        const float x = q0 == 0 ? v4[0] : q0 == 1 ? v4[1] : q0 == 2 ? v4[2] : v4[3];
        T.insert(x, i + q0 * kThreads, kk);
      }
    }
    for (; i < p.V; i += kThreads) T.insert(E::global(row, i), i, kk);
  }
  // each warp's top kk: kk rounds of a warp maximum over the lists' heads
  for (int t = 0; t < kk; ++t) {
    const unsigned long long m = warp_max_u64(T.e[0]);
    if (m != 0ull && T.e[0] == m) T.pop();
    if (lane == 0) S.wk[warp][t] = m;
  }
  __syncthreads();
  if (warp == 0) {
    // the row's top kk from the warps' lists, four candidates per lane
    unsigned long long c0, c1, c2, c3;
    {
      const int e0 = lane, e1 = lane + 32, e2 = lane + 64, e3 = lane + 96;
      c0 = (e0 % kKMax < kk) ? S.wk[e0 / kKMax][e0 % kKMax] : 0ull;
      c1 = (e1 % kKMax < kk) ? S.wk[e1 / kKMax][e1 % kKMax] : 0ull;
      c2 = (e2 % kKMax < kk) ? S.wk[e2 / kKMax][e2 % kKMax] : 0ull;
      c3 = (e3 % kKMax < kk) ? S.wk[e3 / kKMax][e3 % kKMax] : 0ull;
    }
    int n = 0;
    for (int t = 0; t < kk; ++t) {
      const unsigned long long best = max_u64(max_u64(c0, c1), max_u64(c2, c3));
      const unsigned long long m = warp_max_u64(best);
      if (m == 0ull) break;
      if (c0 == m) c0 = 0ull;
      if (c1 == m) c1 = 0ull;
      if (c2 == m) c2 = 0ull;
      if (c3 == m) c3 = 0ull;
      if (lane == 0) {
        S.id[r][t] = key_id(m);
        S.lg[r][t] = key_val(m);
      }
      ++n;
    }
    if (lane == 0) S.n[r] = n;
  }
  __syncthreads();
}

// Warp 0: the depth's rows and valid branches (the tree walk's bookkeeping).
__device__ void plan(const Params& p, Shared& S, int b, int j, bool bonus) {
  const int lane = threadIdx.x & 31;
  const int K = p.K;
  const unsigned valid = S.valid;
  const bool v = lane < K && ((valid >> lane) & 1u);
  const int m = v ? (int)p.model_of[lane] : 64 + lane;
  const unsigned same = __match_any_sync(FULL, m);
  const bool first = v && (__ffs(same) - 1) == lane;   // lowest valid branch of its model
  const unsigned fm = __ballot_sync(FULL, first);
  const unsigned vm = __ballot_sync(FULL, v);
  const int myrow = first ? 1 + __popc(fm & ((1u << lane) - 1u)) : 0;
  const int row = __shfl_sync(FULL, myrow, __ffs(same) - 1);
  if (!bonus && v) {
    const int i = __popc(vm & ((1u << lane) - 1u));
    int x = p.tokens[((size_t)b * K + lane) * p.L + j];
    if (x < 0 || x >= p.V) {
      atomicOr(p.status, MDS_ST_BADTOKEN);
      x = 0;
    }
    S.X[i] = x;
    S.vbr[i] = lane;
    S.vrow[i] = row;
  }
  if (!bonus && first) {
    S.rowp[myrow] = p.drafts[lane] + (((size_t)b * p.L + j) * (size_t)p.V) * p.esize;
    float td = p.temps[(size_t)b * (1 + K) + 1 + lane];
    if (!(td > 0.f) || !(td < kPosInf)) {
      atomicOr(p.status, MDS_ST_BADTEMP);
      td = 1.f;
    }
    S.rowc[myrow] = __fdiv_rn(kLog2e, td);
  }
  if (lane == 0) {
    const int kstar = __ffs(valid) - 1;
    S.rowp[0] = p.target + ((((size_t)b * K + kstar) * (p.L + 1) + j) * (size_t)p.V) * p.esize;
    float tq = p.temps[(size_t)b * (1 + K)];
    if (!(tq > 0.f) || !(tq < kPosInf)) {
      atomicOr(p.status, MDS_ST_BADTEMP);
      tq = 1.f;
    }
    S.rowc[0] = __fdiv_rn(kLog2e, tq);
    // the single-draft step reads only the first valid branch's model row (row 1)
    S.nrows = bonus ? 1 : (p.scheme == MDS_SINGLE ? 2 : 1 + __popc(fm));
    S.nv = bonus ? 0 : __popc(vm);
  }
}

// Warp 0: the kept entries' probabilities, exp2((l - M) log2(e) / T) over
// their sum (M the row's largest kept logit).
__device__ void row_probs(const Params& p, Shared& S, int r) {
  const int lane = threadIdx.x & 31;
  const int n = S.n[r];
  const float M = S.lg[r][0], c = S.rowc[r];
  const float t = (lane < n) ? exp_term(S.lg[r][lane], M, c) : 0.f;
  const float Z = warp_sum(t);
  float pr;
  if (!(Z > 0.f) || !(Z < kPosInf)) {
    // no finite kept logit: the row's first kept token takes the mass
    if (lane == 0) atomicOr(p.status, MDS_ST_NONFINITE);
    pr = (lane == 0) ? 1.f : 0.f;
  } else {
    pr = __fmul_rn(t, __frcp_rn(Z));
  }
  if (lane < n) S.pr[r][lane] = pr;
  __syncwarp();
}

// Warp 0: U (the kept tokens of every row, by increasing id) and each row's
// law on it.
__device__ void build_union(Shared& S) {
  const int lane = threadIdx.x & 31;
  const int nr = S.nrows, ne = nr * kKMax;
  for (int e = lane; e < ne; e += 32) {
    const int r = e / kKMax, t = e - r * kKMax;
    unsigned char d = 1;
    if (t < S.n[r]) {
      const int id = S.id[r][t];
      d = 0;
      for (int f = 0; f < e && !d; ++f) {
        const int rf = f / kKMax, tf = f - rf * kKMax;
        d = (tf < S.n[rf] && S.id[rf][tf] == id) ? 1 : 0;
      }
    }
    S.dup[e] = d;
  }
  __syncwarp();
  int cnt = 0;
  for (int e = lane; e < ne; e += 32) {
    const int r = e / kKMax, t = e - r * kKMax;
    if (t >= S.n[r]) continue;
    const int id = S.id[r][t];
    int k = 0;
    for (int f = 0; f < ne; ++f) {
      const int rf = f / kKMax, tf = f - rf * kKMax;
      k += (!S.dup[f] && tf < S.n[rf] && S.id[rf][tf] < id) ? 1 : 0;
    }
    S.rank[e] = (short)k;
    if (!S.dup[e]) {
      S.uid[k] = id;
      ++cnt;
    }
  }
  const int nU = __reduce_add_sync(FULL, cnt);
  for (int i = lane; i < nr * kEntMax; i += 32) {
    const int r = i / kEntMax, u = i - r * kEntMax;
    if (u < nU) S.law[r][u] = 0.f;
  }
  if (lane == 0) S.nU = nU;
  __syncwarp();
  for (int e = lane; e < ne; e += 32) {
    const int r = e / kKMax, t = e - r * kKMax;
    if (t < S.n[r]) S.law[r][S.rank[e]] = S.pr[r][t];
  }
  __syncwarp();
}

// Position of token x in U, or -1.
__device__ __forceinline__ int find_u(const Shared& S, int x) {
  int lo = 0, hi = S.nU;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (S.uid[mid] < x)
      lo = mid + 1;
    else
      hi = mid;
  }
  return (lo < S.nU && S.uid[lo] == x) ? lo : -1;
}
__device__ __forceinline__ float law_at(const Shared& S, const float* w, int x) {
  const int i = find_u(S, x);
  return i >= 0 ? w[i] : 0.f;
}

__device__ __forceinline__ bool better(float ka, int ia, float kb, int ib) {
  return ka > kb || (ka == kb && ia < ib);
}

// Warp 0: inverse CDF over n weights in U order (increasing token id): the
// first index whose running sum exceeds u * total, the last positive weight
// if rounding leaves none, -1 if the total is not positive.  Both passes sum
// in the same order, so the last running sum is the total.
template <class W>
__device__ int warp_cdf(int n, W w, float u01, float* total) {
  const int lane = threadIdx.x & 31;
  float carry = 0.f;
  for (int base = 0; base < n; base += 32) {
    float c = (base + lane < n) ? w(base + lane) : 0.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(FULL, c, o);
      if (lane >= o) c = __fadd_rn(c, t);
    }
    carry = __fadd_rn(carry, __shfl_sync(FULL, c, 31));
  }
  *total = carry;
  if (!(carry > 0.f)) return -1;
  const float thr = __fmul_rn(u01, carry);
  carry = 0.f;
  int last = -1;
  for (int base = 0; base < n; base += 32) {
    const float x = (base + lane < n) ? w(base + lane) : 0.f;
    float c = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(FULL, c, o);
      if (lane >= o) c = __fadd_rn(c, t);
    }
    const unsigned who = __ballot_sync(FULL, __fadd_rn(carry, c) > thr);
    if (who) return base + __ffs(who) - 1;
    const unsigned pos = __ballot_sync(FULL, x > 0.f);
    if (pos) last = base + 31 - __clz(pos);
    carry = __fadd_rn(carry, __shfl_sync(FULL, c, 31));
  }
  return last;
}

// Warp 0: the next Omega_1 entry among U's keys of one sign (sign > 0: key > 0,
// else key < 0) that comes after (lk, lid) in key order.  Returns its index in
// U or -1; *bk / *bid its key and id.
__device__ int next_key(const Shared& S, int sign, float lk, int lid, float* bk_out, int* bid_out) {
  float bk = kNegInf;
  int bid = 0x7fffffff, bi = -1;
  for (int i = threadIdx.x & 31; i < S.nU; i += 32) {
    const float k = S.key[i];
    if (sign > 0 ? !(k > 0.f) : !(k < 0.f)) continue;
    const int id = S.uid[i];
    if (!better(lk, lid, k, id)) continue;
    if (bi < 0 || better(k, id, bk, bid)) {
      bk = k;
      bid = id;
      bi = i;
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float ok = __shfl_xor_sync(FULL, bk, o);
    const int oid = __shfl_xor_sync(FULL, bid, o);
    const int oi = __shfl_xor_sync(FULL, bi, o);
    if (oi >= 0 && (bi < 0 || better(ok, oid, bk, bid))) {
      bk = ok;
      bid = oid;
      bi = oi;
    }
  }
  *bk_out = bk;
  *bid_out = bid;
  return bi;
}

// Warp 0: one pairwise stage of the weighted scheme with input laws
// a = S.cur (the running law) and b = S.law[rb] against q = S.law[0]; ordered
// inputs (A, Btok) and selection uniform u.  Returns the stage's token and
// leaves its output law in S.cur.  With `sorted`, Omega_2 follows the sorted
// rule of the truncated LP (Section 4 Eq. heur and Eq. p_Ieq, the non-iid
// appendix): a pair inside Omega_2 selects the token earlier in key order, so
// p_I(k) = a_k b_k + b_k A_after(k) + a_k B_after(k) with the Omega_2 masses
// of the tokens after k; otherwise the variant's 1/2 rule.
__device__ int wis_stage(const Params& p, Shared& S, int A, int Btok, int rb, float u, bool sorted) {
  const int lane = threadIdx.x & 31;
  const int nU = S.nU;
  const float* q = S.law[0];
  const float* bl = S.law[rb];
  for (int i = lane; i < nU; i += 32) S.key[i] = __fadd_rn(__fmaf_rn(-S.cur[i], bl[i], q[i]), 0.f);
  __syncwarp();
  const int s = min(p.wis_s, p.V);
  // Omega_1 in key order: positive keys, zero keys by id, negative keys
  int taken = 0;
  for (int sign = 1; sign >= -1; sign -= 2) {
    if (sign < 0 && taken < s) {
      // zero keys by increasing id: tokens outside U and tokens of U whose key is 0
      if (lane == 0) {
        int c = 0, ptr = 0, t = taken;
        while (t < s && c < p.V) {
          while (ptr < nU && S.uid[ptr] < c) ++ptr;
          const bool inU = ptr < nU && S.uid[ptr] == c;
          if (!inU || S.key[ptr] == 0.f) {
            S.om[t] = c;
            S.om_in[t] = inU ? 1 : 0;
            S.om_u[t] = (short)(inU ? ptr : -1);
            ++t;
          }
          ++c;
        }
        S.bcast = t;
      }
      __syncwarp();
      taken = S.bcast;
      __syncwarp();
    }
    float lk = kPosInf;
    int lid = -1;
    while (taken < s) {
      float bk;
      int bid;
      const int bi = next_key(S, sign, lk, lid, &bk, &bid);
      if (bi < 0) break;
      if (lane == 0) {
        S.om[taken] = bid;
        S.om_in[taken] = 1;
        S.om_u[taken] = (short)bi;
      }
      lk = bk;
      lid = bid;
      ++taken;
    }
    __syncwarp();
  }
  if (lane == 0) {
    // Omega_1 by increasing id, with q, a, b at its tokens
    for (int x = 1; x < s; ++x)
      for (int y = x; y > 0 && S.om[y] < S.om[y - 1]; --y) {
        const int ti = S.om[y];
        S.om[y] = S.om[y - 1];
        S.om[y - 1] = ti;
        const unsigned char tc = S.om_in[y];
        S.om_in[y] = S.om_in[y - 1];
        S.om_in[y - 1] = tc;
        const short ts = S.om_u[y];
        S.om_u[y] = S.om_u[y - 1];
        S.om_u[y - 1] = ts;
      }
    for (int t = 0; t < MDS_MAX_S; ++t) {
      const bool in = t < s && S.om_in[t];
      const int i = in ? S.om_u[t] : 0;
      if (t >= s) S.om[t] = 0x7fffffff;
      S.om_q[t] = in ? q[i] : 0.f;
      S.om_a[t] = in ? S.cur[i] : 0.f;
      S.om_b[t] = in ? bl[i] : 0.f;
    }
  }
  __syncwarp();
  // Omega_2 masses of the two input laws
  float sa = 0.f, sb = 0.f;
  for (int i = lane; i < nU; i += 32) {
    bool in1 = false;
    for (int t = 0; t < s; ++t) in1 |= (S.om_in[t] && S.om_u[t] == i);
    S.in1[i] = in1 ? 1 : 0;
    if (!in1) {
      sa = __fadd_rn(sa, S.cur[i]);
      sb = __fadd_rn(sb, bl[i]);
    }
  }
  const float A2 = warp_sum(sa), B2 = warp_sum(sb);
  __syncwarp();
  if (sorted) {
    // Omega_2 values of the sorted rule (tokens outside U carry no mass)
    for (int i = lane; i < nU; i += 32) {
      if (S.in1[i]) continue;
      const float ki = S.key[i];
      const int idi = S.uid[i];
      float aa = 0.f, ba = 0.f;
      for (int j = 0; j < nU; ++j)
        if (!S.in1[j] && better(ki, idi, S.key[j], S.uid[j])) {
          aa = __fadd_rn(aa, S.cur[j]);
          ba = __fadd_rn(ba, bl[j]);
        }
      const float ai = S.cur[i], bi = bl[i];
      S.nxt[i] = __fadd_rn(__fadd_rn(__fmul_rn(ai, bi), __fmul_rn(bi, aa)), __fmul_rn(ai, ba));
    }
    __syncwarp();
  }
  if (lane == 0) {
    bool capped = false;
    int y;
    if (s <= 5) {
      float RS[10], FL[10], FH[10];
      y = stage_solve<5>(s, A2, B2, A, Btok, u, S.om, S.om_q, S.om_a, S.om_b, S.om_x, &capped, RS, FL, FH);
    } else {
      y = stage_solve<MDS_MAX_S>(s, A2, B2, A, Btok, u, S.om, S.om_q, S.om_a, S.om_b, S.om_x, &capped, S.RS, S.FL,
                                 S.FH);
    }
    if (capped) atomicOr(p.status, MDS_ST_LP_CAP);
    if (sorted && A != Btok) {
      // both inputs in Omega_2: the one earlier in key order (a token outside U has key 0)
      bool ia = false, ib = false;
      for (int t = 0; t < s; ++t) {
        ia |= (S.om[t] == A);
        ib |= (S.om[t] == Btok);
      }
      if (!ia && !ib) {
        const int ua = find_u(S, A), ub = find_u(S, Btok);
        const float ka = ua >= 0 ? S.key[ua] : 0.f, kb = ub >= 0 ? S.key[ub] : 0.f;
        y = better(ka, A, kb, Btok) ? A : Btok;
      }
    }
    S.Y = y;
  }
  __syncwarp();
  // the stage's output law: p_I on Omega_1 from the LP; on Omega_2 the sorted
  // rule's values or (a B2 + b A2) / 2
  for (int i = lane; i < nU; i += 32) {
    int pos = -1;
    for (int t = 0; t < s; ++t)
      if (S.om_in[t] && S.om_u[t] == i) pos = t;
    S.cur[i] = (pos >= 0) ? S.om_x[pos]
               : sorted   ? S.nxt[i]
                          : __fmul_rn(0.5f, __fadd_rn(__fmul_rn(S.cur[i], B2), __fmul_rn(bl[i], A2)));
  }
  const int y = S.Y;
  __syncwarp();
  return y;
}

// Warp 0: Algorithm 1 on the intermediate token Y with law p_I = a (on U):
// accept with probability min(1, q(Y) / p_I(Y)), otherwise draw from the
// residual max(0, q - p_I) in token-id order.  *R: the residual mass after a
// rejection (and with acc_prob always), else 0.
__device__ int accept_resid(const Params& p, Shared& S, int b, int j, int Y, const float* a, float* R, float* qY,
                            float* pIY) {
  const int lane = threadIdx.x & 31;
  const float* q = S.law[0];
  const float qy = law_at(S, q, Y), py = law_at(S, a, Y);
  const float ratio = py > 0.f ? __fdiv_rn(qy, py) : kPosInf;
  const bool acc = draw_uniform(p.seed, b, j, kDrawAccept) < fminf(1.f, ratio);
  *qY = qy;
  *pIY = py;
  *R = 0.f;
  if (acc && !p.acc_prob) return Y;
  const float ures = acc ? 0.f : draw_uniform(p.seed, b, j, kDrawResidual);
  float tot;
  int z = warp_cdf(S.nU, [&](int i) { return fmaxf(0.f, __fsub_rn(q[i], a[i])); }, ures, &tot);
  *R = tot;
  if (acc) return Y;
  if (z < 0) {
    // only by rounding: sample q
    if (lane == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
    float t;
    z = warp_cdf(S.nU, [&](int i) { return q[i]; }, ures, &t);
  }
  return z >= 0 ? S.uid[z] : (S.nU > 0 ? S.uid[0] : 0);
}

// Warp 0: sequential rejection over the valid drafts (the SpecTr baseline):
// round i accepts X_i with probability min(1, q_i(X_i) / p_i(X_i)); on
// rejection q_{i+1} = max(0, q_i - p_i) / R_i.  If every round rejects, Z is
// drawn from the last target.  *R: prod_i R_i (0 after an acceptance unless
// acc_prob, which computes the later rounds too).
__device__ int spectr(const Params& p, Shared& S, int b, int j, float* R, float* qY, float* pIY) {
  const int lane = threadIdx.x & 31;
  const int nU = S.nU, nv = S.nv;
  for (int i = lane; i < nU; i += 32) S.cur[i] = S.law[0][i];
  __syncwarp();
  float prodR = 1.f;
  int zacc = -1;
  for (int i = 0; i < nv; ++i) {
    const float* pl = S.law[S.vrow[i]];
    if (zacc < 0) {
      const int x = S.X[i];
      const float qi = law_at(S, S.cur, x), pv = law_at(S, pl, x);
      const float ratio = pv > 0.f ? __fdiv_rn(qi, pv) : kPosInf;
      if (i == 0) {
        *qY = qi;
        *pIY = pv;
      }
      if (draw_uniform(p.seed, b, j, kDrawAccept + i) < fminf(1.f, ratio)) {
        zacc = x;
        if (!p.acc_prob) {
          *R = 0.f;
          return zacc;
        }
      }
    }
    float part = 0.f;
    for (int t = lane; t < nU; t += 32) part = __fadd_rn(part, fmaxf(0.f, __fsub_rn(S.cur[t], pl[t])));
    const float Ri = warp_sum(part);
    prodR = __fmul_rn(prodR, Ri);
    if (Ri > 0.f) {
      const float inv = __frcp_rn(Ri);
      for (int t = lane; t < nU; t += 32) S.cur[t] = __fmul_rn(fmaxf(0.f, __fsub_rn(S.cur[t], pl[t])), inv);
    }
    __syncwarp();
  }
  *R = prodR;
  if (zacc >= 0) return zacc;
  float tot;
  int z = warp_cdf(nU, [&](int t) { return S.cur[t]; }, draw_uniform(p.seed, b, j, kDrawResidual), &tot);
  if (z < 0) {
    if (lane == 0) atomicOr(p.status, MDS_ST_ZERO_RESID);
    z = warp_cdf(nU, [&](int t) { return S.law[0][t]; }, draw_uniform(p.seed, b, j, kDrawResidual), &tot);
  }
  return z >= 0 ? S.uid[z] : (S.nU > 0 ? S.uid[0] : 0);
}

// Warp 0: one depth below L: the rows' laws on U, the scheme's token, the walk.
__device__ __noinline__ void decide(const Params& p, Shared& S, int b, int j) {
  const int lane = threadIdx.x & 31;
  for (int r = 0; r < S.nrows; ++r) row_probs(p, S, r);
  build_union(S);
  const int nv = S.nv;
  int Z, Yd;
  float R = 0.f, qY = 0.f, pIY = 0.f;
  if (p.scheme == MDS_SPECTR) {
    Z = spectr(p, S, b, j, &R, &qY, &pIY);
    Yd = S.X[0];
  } else {
    int Y = S.X[0];
    const float* a = S.law[S.vrow[0]];
    if ((p.scheme == MDS_WIS || p.scheme == MDS_WISSORT) && nv > 1) {
      for (int i = lane; i < S.nU; i += 32) S.cur[i] = a[i];
      __syncwarp();
      // every stage's selection uniform at once (lane m - 1 draws stage m's)
      const float ul = (lane + 1 < nv) ? draw_uniform(p.seed, b, j, kDrawSelect + lane) : 0.f;
      const bool sorted = p.scheme == MDS_WISSORT;
      for (int m = 1; m < nv; ++m)
        Y = wis_stage(p, S, Y, S.X[m], S.vrow[m], __shfl_sync(FULL, ul, m - 1), sorted);
      a = S.cur;
    }
    Z = accept_resid(p, S, b, j, Y, a, &R, &qY, &pIY);
    Yd = Y;
  }
  if (lane == 0) {
    p.out_tokens[(size_t)b * (p.L + 1) + j] = Z;
    if (p.out_diag) {
      float* dg = p.out_diag + ((size_t)b * (p.L + 1) + j) * 4;
      dg[0] = qY;
      dg[1] = pIY;
      dg[2] = R;
      dg[3] = (float)Yd;
    }
    unsigned nvm = 0u;
    for (int i = 0; i < nv; ++i)
      if (S.X[i] == Z) nvm |= 1u << S.vbr[i];
    S.valid = nvm;
    if (!nvm) {
      p.out_accept[b] = j;
      S.done = 1;
    }
  }
  __syncwarp();
}

// Warp 0: every draft accepted: the bonus token from the restricted target
// row at depth L, by inverse CDF in token-id order.
__device__ __noinline__ void bonus_step(const Params& p, Shared& S, int b) {
  const int lane = threadIdx.x & 31;
  row_probs(p, S, 0);
  const int n = S.n[0];
  if (lane < n) {
    const int id = S.id[0][lane];
    int k = 0;
    for (int f = 0; f < n; ++f) k += (S.id[0][f] < id) ? 1 : 0;
    S.bid[k] = id;
    S.bw[k] = S.pr[0][lane];
  }
  __syncwarp();
  float Q;
  const int z = warp_cdf(n, [&](int i) { return S.bw[i]; }, draw_uniform(p.seed, b, p.L, kDrawBonus), &Q);
  if (lane == 0) {
    p.out_tokens[(size_t)b * (p.L + 1) + p.L] = z >= 0 ? S.bid[z] : (n > 0 ? S.bid[0] : 0);
    if (p.out_diag) {
      float* dg = p.out_diag + ((size_t)b * (p.L + 1) + p.L) * 4;
      dg[0] = 0.f;
      dg[1] = 0.f;
      dg[2] = Q;
      dg[3] = -1.f;
    }
    p.out_accept[b] = p.L;
    S.done = 1;
  }
  __syncwarp();
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 2) topk_kernel(const Params p) {
  __shared__ Shared S;
  const int b = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int kk = min(p.top_k, p.V);
  for (int j = tid; j <= p.L; j += kThreads) p.out_tokens[(size_t)b * (p.L + 1) + j] = -1;
  if (tid == 0) {
    S.valid = (p.K >= 32) ? FULL : ((1u << p.K) - 1u);
    S.done = 0;
  }
  __syncthreads();
  for (int j = 0; j <= p.L; ++j) {
    const bool bonus = (j == p.L);
    if (warp == 0) plan(p, S, b, j, bonus);
    __syncthreads();
    const int nr = S.nrows;
    for (int r = 0; r < nr; ++r) select_row<DT>(p, S, r, kk);
    if (warp == 0) {
      if (bonus)
        bonus_step(p, S, b);
      else
        decide(p, S, b, j);
    }
    __syncthreads();
    if (S.done) break;
  }
}

template <int DT>
cudaError_t launch_dt(const Params& p, cudaStream_t stream) {
  topk_kernel<DT><<<p.B, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch(const Params& p, cudaStream_t stream) {
  if (p.B <= 0) return cudaSuccess;
  return p.dtype == MDS_F32 ? launch_dt<MDS_F32>(p, stream) : launch_dt<MDS_BF16>(p, stream);
}

int verify(const mds_config& c, int scheme, const int8_t* model_of, bool vec, const void* target_logits,
           const void* const* draft_logits, const int32_t* draft_tokens, const float* temperatures,
           int32_t* out_tokens, int32_t* out_accept_len, float* out_diag, int B, uint64_t seed, unsigned* status,
           cudaStream_t stream) {
  if (!serves(scheme)) return MDS_EUNSUP;
  Params p{};
  p.target = static_cast<const char*>(target_logits);
  for (int k = 0; k < c.K; ++k) {
    p.drafts[k] = static_cast<const char*>(draft_logits[k]);
    p.model_of[k] = model_of[k];
  }
  p.tokens = draft_tokens;
  p.temps = temperatures;
  p.out_tokens = out_tokens;
  p.out_accept = out_accept_len;
  p.out_diag = out_diag;
  p.status = status;
  p.seed = seed;
  p.B = B;
  p.K = c.K;
  p.L = c.L;
  p.V = c.V;
  p.dtype = c.dtype;
  p.esize = c.dtype == MDS_F32 ? 4 : 2;
  p.top_k = c.top_k;
  p.wis_s = c.wis_s;
  p.scheme = scheme;
  p.acc_prob = c.acc_prob;
  p.vec = vec ? 1 : 0;
  const cudaError_t e = launch(p, stream);
  return e == cudaSuccess ? MDS_OK : record_cuda_error(e, "top-k kernel launch");
}

}  // namespace topk
}  // namespace mds
