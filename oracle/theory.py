"""Oracle pins: the paper's optimisation problems and closed forms.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Brute-force linear programs on tiny vocabularies (scipy's HiGHS solver) and
the closed forms the paper proves, so that the tests can check one against
the other and the verification oracle against both.
"""
import itertools

import numpy as np
from scipy.optimize import linprog


def _prod_prob(dists, x):
    pr = 1.0
    for xi, p in zip(x, dists):
        pr *= p[xi]
    return pr


def tlsr_optimum(q, dists):
    """Problem 1 (Section 3): the largest Pr(Z in S) over valid token-level
    selection rules P(z | x), for drafts x_i ~ dists[i] independently.

    Variables P(z | x) for every x in Omega^K and z in Omega; constraints
    sum_z P(z|x) = 1 and sum_x P(z|x) Pr(x) = q(z)."""
    V = len(q)
    K = len(dists)
    xs = list(itertools.product(range(V), repeat=K))
    n = len(xs) * V
    c = np.zeros(n)
    A_eq = []
    b_eq = []
    for ix, x in enumerate(xs):
        pr = _prod_prob(dists, x)
        row = np.zeros(n)
        row[ix * V:(ix + 1) * V] = 1.0
        A_eq.append(row)
        b_eq.append(1.0)
        for z in set(x):
            c[ix * V + z] -= pr
    for z in range(V):
        row = np.zeros(n)
        for ix, x in enumerate(xs):
            row[ix * V + z] = _prod_prob(dists, x)
        A_eq.append(row)
        b_eq.append(q[z])
    res = linprog(c, A_eq=np.array(A_eq), b_eq=np.array(b_eq), bounds=(0, 1), method="highs")
    assert res.status == 0, res.message
    return -res.fun


def iws_optimum(q, dists):
    """Theorem 1, Eq. (IS-opt1a): max over importance-weighted selection
    weights beta_y(x) (beta_y(x) = 0 unless y is one of x, sum_y beta_y(x) = 1)
    of sum_y min(q(y), sum_x beta_y(x) Pr(x)).  min() is linearised with
    t_y <= q(y), t_y <= sum_x beta_y(x) Pr(x)."""
    V = len(q)
    K = len(dists)
    xs = list(itertools.product(range(V), repeat=K))
    var = {}
    for ix, x in enumerate(xs):
        for y in sorted(set(x)):
            var[(ix, y)] = len(var)
    nb = len(var)
    n = nb + V
    c = np.zeros(n)
    c[nb:] = -1.0
    A_eq, b_eq, A_ub, b_ub = [], [], [], []
    for ix, x in enumerate(xs):
        row = np.zeros(n)
        for y in set(x):
            row[var[(ix, y)]] = 1.0
        A_eq.append(row)
        b_eq.append(1.0)
    for y in range(V):
        row = np.zeros(n)
        row[nb + y] = 1.0
        for ix, x in enumerate(xs):
            if y in x:
                row[var[(ix, y)]] -= _prod_prob(dists, x)
        A_ub.append(row)
        b_ub.append(0.0)
    bounds = [(0, 1)] * nb + [(0, q[y]) for y in range(V)]
    res = linprog(c, A_ub=np.array(A_ub), b_ub=np.array(b_ub), A_eq=np.array(A_eq), b_eq=np.array(b_eq),
                  bounds=bounds, method="highs")
    assert res.status == 0, res.message
    return -res.fun


def thm3_pstar(p, q):
    """Theorem 3, Eq. (opt): K = 2 i.i.d. drafts,
    min over S of sum_S q + (sum_{S^c} p)^2 + 2 (sum_S p)(sum_{S^c} p)."""
    V = len(p)
    best = np.inf
    for mask in range(1 << V):
        S = [i for i in range(V) if mask >> i & 1]
        Sc = [i for i in range(V) if not mask >> i & 1]
        qs = sum(q[i] for i in S)
        ps = sum(p[i] for i in S)
        pc = sum(p[i] for i in Sc)
        best = min(best, qs + pc * pc + 2.0 * ps * pc)
    return best


def remark2_pstar(p, q, K=2):
    """Remark 2, Eq. (opt_old): min over S of sum_S q - (sum_S p)^K + 1
    (proved for K = 2; the paper conjectures it for K > 2)."""
    V = len(p)
    best = np.inf
    for mask in range(1 << V):
        S = [i for i in range(V) if mask >> i & 1]
        best = min(best, sum(q[i] for i in S) - sum(p[i] for i in S) ** K + 1.0)
    return best


def pstar_sorted(p, q, K=2):
    """Theorem 3 / Remark 2 on any vocabulary size: the minimum over S of
    sum_S q - (sum_S p)^K + 1 (for K = 2 the optimum of Theorem 3; for K > 2
    Remark 2's conjectured form), by a scan over V + 1 sets.

    Why a scan suffices: t^K is convex, so -t^K = min_l [(K-1) l^K - K l^(K-1) t]
    (its tangent lines), and the minimum over S and l can be taken in either
    order.  For a fixed l the inner minimum of sum_{s in S} (q_s - K l^(K-1) p_s)
    takes exactly the tokens with q_s / p_s below K l^(K-1) (ties contribute
    0), so some optimal S is a prefix of the tokens sorted by the ratio
    q_s / p_s (tokens with p_s = 0 last).  This is a derivation from the
    paper's closed form, not an algorithm the paper states; it is pinned
    against the 2^V-subset minimum."""
    p = np.asarray(p, dtype=np.float64)
    q = np.asarray(q, dtype=np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        ratio = np.where(p > 0, q / np.where(p > 0, p, 1.0), np.inf)
    order = np.argsort(ratio, kind="stable")
    Q = np.concatenate([[0.0], np.cumsum(q[order])])
    P = np.concatenate([[0.0], np.cumsum(p[order])])
    return float(np.min(Q - P ** K) + 1.0)


def thm2_condition(p, q, tol=0.0):
    """Theorem 2, Eq. (conj): sum_S q >= (sum_S p)^2 for every subset S.
    S = Omega holds with equality (1 >= 1) and is skipped so that rounding of
    the sums cannot decide the answer."""
    V = len(p)
    for mask in range(1, (1 << V) - 1):
        S = [i for i in range(V) if mask >> i & 1]
        if sum(q[i] for i in S) < sum(p[i] for i in S) ** 2 - tol:
            return False
    return True


def single_draft_acceptance(p, q):
    """Appendix A: Algorithm 1 accepts with probability sum_x min(p, q) = 1 - d_TV."""
    return float(np.minimum(p, q).sum())


def stage_lp_optimum(q, a, b, omega1):
    """The s-variable LP of one WIS stage solved directly (HiGHS), built from
    its definition: for k in Omega_1,
        p_I(k) = a_k b_k + sum_{l not in Omega_1} (a_k b_l + a_l b_k)
                 + sum_{l in Omega_1, l != k} (a_k b_l + a_l b_k) w_kl,
    w_kl + w_lk = 1, 0 <= w <= 1; maximise sum_{k in Omega_1} min(q_k, p_I(k))."""
    om = list(omega1)
    s = len(om)
    out = np.ones(len(q), dtype=bool)
    out[om] = False
    ends = [(i, j) for i in range(s) for j in range(i + 1, s)]
    P = len(ends)
    n = P + s                       # variables: w_e (fraction to side i), t_k
    c = np.zeros(n)
    c[P:] = -1.0
    A_ub, b_ub = [], []
    for k in range(s):
        kk = om[k]
        fixed = a[kk] * b[kk] + float(np.sum(a[kk] * b[out] + a[out] * b[kk]))
        row = np.zeros(n)
        row[P + k] = 1.0
        rhs = fixed
        for e, (i, j) in enumerate(ends):
            m = a[om[i]] * b[om[j]] + a[om[j]] * b[om[i]]
            if i == k:
                row[e] -= m          # t_k <= fixed + m w_e
            elif j == k:
                row[e] += m          # t_k <= fixed + m (1 - w_e)
                rhs += m
        A_ub.append(row)
        b_ub.append(rhs)
    bounds = [(0, 1)] * P + [(None, q[om[k]]) for k in range(s)]
    res = linprog(c, A_ub=np.array(A_ub), b_ub=np.array(b_ub), bounds=bounds, method="highs")
    assert res.status == 0, res.message
    return -res.fun


def stage_min_cut(d, m, s):
    """Max-flow value of a stage's pair/token network by the min-cut formula:
    min over token sets N of sum_{k in N} d_k + sum of masses of pairs not
    contained in N."""
    ends = [(i, j) for i in range(s) for j in range(i + 1, s)]
    best = np.inf
    for mask in range(1 << s):
        val = sum(d[k] for k in range(s) if mask >> k & 1)
        val += sum(m[e] for e, (i, j) in enumerate(ends) if not ((mask >> i & 1) and (mask >> j & 1)))
        best = min(best, val)
    return best
