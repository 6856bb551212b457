"""Oracle: the truncated LP with the sorted rule on Omega_2 (Eq. heur).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  Plain fp64 numpy.

Section 4 ("Faster approximations to linear program", Eq. heur and Eq.
p_Ieq) and Appendix G, Algorithm 2, for two inputs; the non-iid appendix
(App. I) for A ~ a, B ~ b with distinct laws:

1. Sort the vocabulary by the key q_k - a_k b_k, largest first (ties: lower
   token id first).  Omega_1 = the first s tokens, Omega_2 = the rest.
2. Fixed weights: a pair with exactly one token in Omega_1 selects that
   token; a pair inside Omega_2 selects the token that comes first in the
   sorted order (w_ij = 1 for i before j).  Hence, for k in Omega_2,
       p_I(k) = a_k b_k + sum_{j in Omega_2 after k} (a_j b_k + a_k b_j)
   (Eq. p_Ieq; the non-iid appendix's second display).
3. For k in Omega_1 the free weights solve the same s-variable LP as the
   variant (maximise sum_{Omega_1} min(q, p_I)); base_k = a_k b_k + a_k B2 +
   b_k A2 with A2, B2 the Omega_2 masses.  The maximum flow, its fixed order
   and the 1/2 split of leftover pair mass are those of ``wis`` (a reading:
   the LP optimum is not unique).
4. Selection for ordered inputs (A, B): A == B -> A; both in Omega_1 -> A
   with probability w_AB; exactly one in Omega_1 -> that one; both in
   Omega_2 -> the one earlier in the sorted order.

K > 2 drafts: pairwise stages as in Remark 4, stage m pairing (Y_{m-1},
X_{m+1}) with a = the law of Y_{m-1}; the law after a stage is a full vector
(every Omega_2 token's value depends on its rank), unlike the variant's.
"""
import numpy as np

from . import wis as wis_mod


class SortedStage:
    __slots__ = ("order", "rank", "omega1", "in1", "A2", "B2", "pI", "w", "pair_index", "flow_value", "d", "m")


def stage(q, a, b, s, note=None):
    """One pairwise stage of the sorted truncated LP (module docstring)."""
    note = note or (lambda *args: None)
    q, a, b = (np.asarray(x, dtype=np.float64) for x in (q, a, b))
    n = len(q)
    s = min(int(s), n)
    key = q - a * b
    order = np.lexsort((np.arange(n), -key))
    rank = np.empty(n, dtype=np.int64)
    rank[order] = np.arange(n)
    if s < n:
        k1, k2 = order[s - 1], order[s]
        scale = max(q[k1] + a[k1] * b[k1] + q[k2] + a[k2] * b[k2], 1e-30)
        note("key", (key[k1] - key[k2]) / scale, wis_mod.BAND_KEY)
    omega1 = np.sort(order[:s])
    in1 = np.zeros(n, dtype=bool)
    in1[omega1] = True
    A2 = float(a[~in1].sum())
    B2 = float(b[~in1].sum())
    # Omega_2: suffix sums of a and b in sorted order (tokens after k)
    pI = np.zeros(n)
    tail = order[s:]
    a_after = np.concatenate([np.cumsum(a[tail][::-1])[::-1][1:], [0.0]]) if len(tail) else np.zeros(0)
    b_after = np.concatenate([np.cumsum(b[tail][::-1])[::-1][1:], [0.0]]) if len(tail) else np.zeros(0)
    pI[tail] = a[tail] * b[tail] + b[tail] * a_after + a[tail] * b_after
    # Omega_1: the variant's LP on the same base values
    base = np.array([a[k] * b[k] + a[k] * B2 + b[k] * A2 for k in omega1])
    qk = q[omega1]
    d = np.maximum(0.0, qk - base)
    ends = [(i, j) for i in range(s) for j in range(i + 1, s)]
    m_pairs = [a[omega1[i]] * b[omega1[j]] + a[omega1[j]] * b[omega1[i]] for i, j in ends]
    eps = wis_mod.LP_EPS_REL * float(np.sum(qk + base))
    f, rs = wis_mod._max_flow(d, m_pairs, ends, eps, note)
    x = base.copy()
    w, pair_index = {}, {}
    for e, (i, j) in enumerate(ends):
        to_i = f[e, 0] + 0.5 * rs[e]
        to_j = f[e, 1] + 0.5 * rs[e]
        x[i] += to_i
        x[j] += to_j
        w[e] = to_i / m_pairs[e] if m_pairs[e] > 0 else 0.5
        pair_index[(i, j)] = e
    pI[omega1] = x
    st = SortedStage()
    st.order, st.rank, st.omega1, st.in1, st.A2, st.B2, st.pI = order, rank, omega1, in1, A2, B2, pI
    st.w, st.pair_index = w, pair_index
    st.flow_value = float(sum(f[e, 0] + f[e, 1] for e in range(len(ends))))
    st.d, st.m = d, np.array(m_pairs)
    return st


def beta(st, A, B):
    """Law of the stage output for ordered inputs (A, B) (step 4)."""
    if A == B:
        return {A: 1.0}
    ia, ib = st.in1[A], st.in1[B]
    if ia and ib:
        pa = int(np.searchsorted(st.omega1, A))
        pb = int(np.searchsorted(st.omega1, B))
        wa = st.w[st.pair_index[(pa, pb)]] if pa < pb else 1.0 - st.w[st.pair_index[(pb, pa)]]
        return {A: wa, B: 1.0 - wa}
    if ia:
        return {A: 1.0}
    if ib:
        return {B: 1.0}
    return {A: 1.0} if st.rank[A] < st.rank[B] else {B: 1.0}


def select(st, A, B, u, note=None):
    """The stage's output token with the stage's uniform u (A iff u < w)."""
    law = beta(st, A, B)
    if len(law) == 1:
        return next(iter(law))
    wa = law[A]
    if note is not None:
        note("select", abs(u - wa), wis_mod.BAND_SELECT)
    return A if u < wa else B


def sorted_select(rec, q, dists, X, us, s):
    """Pairwise stages over the valid drafts (Remark 4).  Returns (Y, p_I)."""
    if len(X) == 1:
        return X[0], dists[0]
    A, a = X[0], dists[0]
    for m in range(1, len(X)):
        st = stage(q, a, dists[m], s, rec.note)
        A = select(st, A, X[m], us[m - 1], rec.note)
        a = st.pI
    return A, a
