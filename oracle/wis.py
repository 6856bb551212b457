"""Oracle: weighted importance sampling with the variant truncated LP.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

One pairwise stage takes two independent input tokens A ~ a and B ~ b and
returns Y in {A, B}.  It follows the paper's "Variant of Truncated LP"
(appendix on complexity, Eq. heur2 and the p_I formula after it), written for
independent but non-identical inputs as in the non-iid appendix (ordered
inputs, key q_k - p_{1,k} p_{2,k}):

1. Omega_1 = the s tokens with the largest key  q_k - a_k b_k  (ties: lower
   token id first); Omega_2 = the rest.
2. Fixed weights: a pair with exactly one token in Omega_1 selects that token
   (w = 1 for Omega_1 x Omega_2); a pair of distinct tokens inside Omega_2
   selects either with probability 1/2 (w = 1/2 inside Omega_2).  With
   A2 = sum_{Omega_2} a and B2 = sum_{Omega_2} b this gives, for k in Omega_2,
       p_I(k) = a_k b_k + 1/2 sum_{l in Omega_2, l != k} (a_k b_l + a_l b_k)
              = 1/2 (a_k B2 + b_k A2).
   (Reading: the printed i.i.d. formula sums "i != k" over all of Omega; only
   the reading "i in Omega_2 minus k" is consistent with w = 1 on Omega_1 x
   Omega_2 and makes p_I sum to one.  For a = b = p it is p_k P(Omega_2).)
3. For k in Omega_1:  p_I(k) = base_k + sum_{l in Omega_1} m_kl w_kl  with
       base_k = a_k b_k + a_k B2 + b_k A2,   m_kl = a_k b_l + a_l b_k,
   and the free weights w_kl + w_lk = 1 solve the s-variable LP
       maximise sum_{k in Omega_1} min(q_k, p_I(k))
   (Algorithm 2's LP restricted to Omega_1).  Written as a maximum flow:
   source -> pair {k,l} (capacity m_kl) -> either endpoint -> sink (capacity
   d_k = max(0, q_k - base_k)).  The flow is found by breadth-first
   augmenting paths in a fixed order (below); pair mass left after the flow
   is split 1/2 - 1/2 (reading: the LP optimum is not unique and the paper
   gives no tie-break).  Residual capacities at or below
   eps = 1e-6 * sum_{Omega_1}(q_k + base_k) count as saturated.
4. Selection: A == B -> A; both in Omega_1 -> A with probability w_AB;
   exactly one in Omega_1 -> that one; both in Omega_2 -> A with
   probability 1/2.  The stage's uniform decides: A iff u < w.

K > 2 drafts (Remark 4): stage 1 pairs (X_1, X_2) -> Y_1, stage m pairs
(Y_{m-1}, X_{m+1}) -> Y_m, with a = law of Y_{m-1} and b = law of X_{m+1};
every stage maximises against the same target q (reading).

Flow order (reading; any maximum flow is an LP optimum).  Omega_1 is indexed
by increasing token id; pair (i, j), i < j, are taken lexicographically.
(a) Direct pass: each pair in order gives what it can to its lower-index
    token, then to its higher-index token (each while both the pair's supply
    and the token's remaining demand exceed eps).
(b) Augmenting paths in token space: a token is a source if some pair
    containing it has supply > eps (its source pair: the first such pair);
    token u leads to token v if pair {u, v} currently gives flow > eps to u
    (that flow can be moved to v).  Breadth-first from all sources, level by
    level, tokens in increasing index within a level, each token's parent the
    first frontier token (increasing index) that reaches it; the path ends at
    the first token in that order whose remaining demand exceeds eps.  The
    bottleneck (source pair supply, moved flows, end demand) is pushed and
    the search repeats until no path exists.
(c) Pair mass left over is split 1/2 - 1/2.
Residuals at or below eps = 1e-6 * sum_{Omega_1}(q_k + base_k) count as zero.
"""
import numpy as np

LP_EPS_REL = 1e-6
BAND_KEY = 1e-6
BAND_LP = 0.5      # |r - eps| < BAND_LP * eps flags a near-degenerate LP decision
BAND_SELECT = 1e-6
LP_MAX_AUGMENT = 4096


class Stage:
    """Result of one pairwise stage."""

    __slots__ = ("omega1", "in1", "A2", "B2", "pI", "w", "pair_index", "flow_value", "d", "m")


def _max_flow(d, m_pairs, ends, eps, note):
    """Maximum flow on the pair/token network in the fixed order of the
    module docstring.  Returns (flow [P][2] to (lower, higher) token,
    remaining supply [P])."""
    P = len(m_pairs)
    n = len(d)
    rs = np.array(m_pairs, dtype=np.float64)
    rd = np.array(d, dtype=np.float64)
    f = np.zeros((P, 2), dtype=np.float64)
    pair_of = {}
    for e, (i, j) in enumerate(ends):
        pair_of[(i, j)] = e
        pair_of[(j, i)] = e

    def pos(val):
        note("lp", abs(val - eps), BAND_LP * eps)
        return val > eps

    # (a) direct pass
    for e, (i, j) in enumerate(ends):
        for side, t in ((0, i), (1, j)):
            if pos(rs[e]) and pos(rd[t]):
                delta = min(rs[e], rd[t])
                f[e, side] += delta
                rs[e] -= delta
                rd[t] -= delta
    # (b) augmenting paths in token space
    for _ in range(LP_MAX_AUGMENT):
        src_pair = [-1] * n
        for e, (i, j) in enumerate(ends):
            if pos(rs[e]):
                for t in (i, j):
                    if src_pair[t] < 0:
                        src_pair[t] = e
        parent = [-1] * n
        visited = [src_pair[t] >= 0 for t in range(n)]
        frontier = [t for t in range(n) if visited[t]]
        sink = next((t for t in frontier if pos(rd[t])), -1)
        while sink < 0 and frontier:
            nxt = []
            for u in frontier:
                for v in range(n):
                    if v == u or visited[v] or v in nxt:
                        continue
                    e = pair_of[(u, v)]
                    side_u = 0 if ends[e][0] == u else 1
                    if pos(f[e, side_u]):
                        parent[v] = u
                        nxt.append(v)
            nxt.sort()
            for v in nxt:
                visited[v] = True
            frontier = nxt
            sink = next((t for t in frontier if pos(rd[t])), -1)
        if sink < 0:
            return f, rs
        # path sink <- ... <- t0 (a source); bottleneck
        path = [sink]
        while parent[path[-1]] >= 0:
            path.append(parent[path[-1]])
        path.reverse()
        e0 = src_pair[path[0]]
        delta = min(rs[e0], rd[sink])
        for u, v in zip(path[:-1], path[1:]):
            e = pair_of[(u, v)]
            delta = min(delta, f[e, 0 if ends[e][0] == u else 1])
        rs[e0] -= delta
        f[e0, 0 if ends[e0][0] == path[0] else 1] += delta
        for u, v in zip(path[:-1], path[1:]):
            e = pair_of[(u, v)]
            f[e, 0 if ends[e][0] == u else 1] -= delta
            f[e, 0 if ends[e][0] == v else 1] += delta
        rd[sink] -= delta
    note("lp_cap", 0.0, 1.0)   # iteration cap reached: flag the depth
    return f, rs


def wis_stage(q, a, b, s, note):
    """One pairwise stage (module docstring, steps 1-3)."""
    n = len(q)
    s = min(int(s), n)
    key = q - a * b
    ids = np.arange(n)
    order = np.lexsort((ids, -key))
    if s < n:
        k1, k2 = order[s - 1], order[s]
        gap = key[k1] - key[k2]
        scale = max(q[k1] + a[k1] * b[k1] + q[k2] + a[k2] * b[k2], 1e-30)
        note("key", gap / scale, BAND_KEY)
    omega1 = np.sort(order[:s])
    in1 = np.zeros(n, dtype=bool)
    in1[omega1] = True
    A2 = float(a[~in1].sum())
    B2 = float(b[~in1].sum())
    pI = 0.5 * (a * B2 + b * A2)
    base = np.array([a[k] * b[k] + a[k] * B2 + b[k] * A2 for k in omega1])
    qk = q[omega1]
    d = np.maximum(0.0, qk - base)
    ends = [(i, j) for i in range(s) for j in range(i + 1, s)]
    m_pairs = [a[omega1[i]] * b[omega1[j]] + a[omega1[j]] * b[omega1[i]] for i, j in ends]
    eps = LP_EPS_REL * float(np.sum(qk + base))
    f, rs = _max_flow(d, m_pairs, ends, eps, note)
    x = base.copy()
    w = {}
    pair_index = {}
    for e, (i, j) in enumerate(ends):
        left = rs[e]
        to_i = f[e, 0] + 0.5 * left
        to_j = f[e, 1] + 0.5 * left
        x[i] += to_i
        x[j] += to_j
        w[e] = to_i / m_pairs[e] if m_pairs[e] > 0 else 0.5
        pair_index[(i, j)] = e
    pI[omega1] = x
    st = Stage()
    st.omega1, st.in1, st.A2, st.B2, st.pI, st.w, st.pair_index = omega1, in1, A2, B2, pI, w, pair_index
    st.flow_value = float(sum(f[e, 0] + f[e, 1] for e in range(len(ends))))
    st.d, st.m = d, np.array(m_pairs)
    return st


def stage_select(st, A, B, u, note):
    """Step 4: the stage's output token for ordered inputs (A, B)."""
    if A == B:
        return A
    ia, ib = st.in1[A], st.in1[B]
    if ia and ib:
        pa = int(np.searchsorted(st.omega1, A))
        pb = int(np.searchsorted(st.omega1, B))
        if pa < pb:
            wa = st.w[st.pair_index[(pa, pb)]]
        else:
            wa = 1.0 - st.w[st.pair_index[(pb, pa)]]
        note("select", abs(u - wa), BAND_SELECT)
        return A if u < wa else B
    if ia:
        return A
    if ib:
        return B
    return A if u < 0.5 else B


def wis_select(rec, q, dists, X, us, s):
    """Pairwise stages over the valid drafts (Remark 4).  Returns (Y, p_I)."""
    note = rec.note
    if len(X) == 1:
        return X[0], dists[0]
    A, a = X[0], dists[0]
    for m in range(1, len(X)):
        st = wis_stage(q, a, dists[m], s, note)
        A = stage_select(st, A, X[m], us[m - 1], note)
        a = st.pI
    return A, a


class _NullNote:
    def __call__(self, name, value, threshold):
        pass


def stage_law(q, a, b, s):
    """Convenience for tests: the stage object without margin bookkeeping."""
    return wis_stage(q, a, b, s, _NullNote())
