"""Oracle: classical importance sampling and the law of its selected token.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Selection (Section 3, after Definition 1): with weights
rho_i = q(X_i) / p_{d(i)}(X_i) over the valid drafts in branch order,
I = the smallest i with rho_1 + ... + rho_i > u * (rho_1 + ... + rho_K), and
Y = X_I.

Law of Y.  The paper gives no formula for p_I under this rule.  Writing
Pr(I = i, X_i = y) = p_{d(i)}(y) E[rho_i(y) / (rho_i(y) + sum_{j != i} rho_j(X_j))],
using 1/c = int_0^inf exp(-t c) dt and the independence of the drafts:

    p_I(y) = q(y) sum_i int_0^inf exp(-t rho_i(y)) prod_{j != i} M_j(t) dt,
    M_j(t) = sum_x p_{d(j)}(x) exp(-t rho_j(x)).

Grouping the valid branches by draft model d (c_d branches each):

    p_I(y) = q(y) sum_d c_d int_0^inf exp(-t rho_d(y)) M_d(t)^(c_d - 1)
                          prod_{d' != d} M_d'(t)^(c_d') dt.

Quadrature (reading): trapezoid rule in u = ln t on the grid u_m = m h,
m = floor(u_lo/h) .. ceil(u_hi/h), u_lo = -ln(K rho_max) - 40,
u_hi = ln(40 / rho_min), rho over every (model, token) with positive p and q;
at most IS_NODES_MAX nodes (the top of the range is cut if more).  The
integrand decays like exp(u) below u_lo and like exp(-40) beyond u_hi, and
the trapezoid rule converges geometrically for it, so the fp64 result is
exact to rounding for h = 1/4.
"""
import math

import numpy as np

IS_NODES_MAX = 1024
BAND_SELECT = 1e-6


def node_grid(rho_min, rho_max, K, h):
    """Integer node range (m_lo, m_hi) of the trapezoid grid u_m = m h."""
    u_lo = -math.log(K * rho_max) - 40.0
    u_hi = math.log(40.0 / rho_min)
    m_lo = math.floor(u_lo / h)
    m_hi = math.ceil(u_hi / h)
    if m_hi - m_lo + 1 > IS_NODES_MAX:
        m_hi = m_lo + IS_NODES_MAX - 1
    return m_lo, m_hi


def is_law(q, rows, counts, h):
    """p_I over the whole vocabulary.

    rows    dict model -> p_d (fp64 vectors)
    counts  dict model -> c_d (number of valid branches drawn from model d)"""
    models = sorted(rows)
    K = sum(counts[d] for d in models)
    rho = {d: np.where(rows[d] > 0, q / np.where(rows[d] > 0, rows[d], 1.0), np.inf) for d in models}
    finite = np.concatenate([r[np.isfinite(r) & (r > 0)] for r in rho.values()])
    rho_min, rho_max = float(finite.min()), float(finite.max())
    m_lo, m_hi = node_grid(rho_min, rho_max, K, h)
    acc = np.zeros_like(q)
    for mm in range(m_lo, m_hi + 1):
        t = math.exp(mm * h)
        M = {d: float(np.sum(rows[d] * np.exp(-t * rho[d]))) for d in models}
        for d in models:
            c = counts[d]
            weight = h * t * c * M[d] ** (c - 1)
            for d2 in models:
                if d2 != d:
                    weight *= M[d2] ** counts[d2]
            if weight != 0.0:
                acc += weight * np.exp(-t * rho[d])
    return q * acc


def is_select(rec, q, rows, mids, X, u, h):
    """Selection and p_I for the valid drafts X drawn from models ``mids``.

    rows  dict model -> p_d.  Returns (Y, p_I)."""
    if len(X) == 1:
        return X[0], rows[mids[0]]
    rho = np.array([q[x] / rows[d][x] if rows[d][x] > 0 else np.inf for x, d in zip(X, mids)])
    if np.isinf(rho).any():
        I = int(np.argmax(np.isinf(rho)))
    else:
        tot = float(np.sum(rho))
        c = np.cumsum(rho)
        t = u * tot
        I = int(np.searchsorted(c, t, side="right"))
        I = min(I, len(X) - 1)
        lo = c[I - 1] if I > 0 else 0.0
        if tot > 0:
            rec.note("is_select", min(c[I] - t, t - lo) / tot, BAND_SELECT)
    counts = {}
    for d in mids:
        counts[d] = counts.get(d, 0) + 1
    pI = is_law(q, {d: rows[d] for d in counts}, counts, h)
    return X[I], pI
