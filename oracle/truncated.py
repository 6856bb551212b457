"""Oracle: the truncated-alphabet scheme and top-k / top-p preprocessing.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  Plain fp64 numpy.

Truncated alphabet (Section 4, "truncated alphabet" scheme; the non-iid
appendix's closing remark on applying it to distinct drafts)
------------------------------------------------------------------------
Omega_0 is a high-probability subset of the vocabulary under the target q.
Reading of "a subset of size M": the tokens whose probability is strictly
above the (M+1)-th largest probability (counted with multiplicity), so at
most M tokens; tokens tied at the cut are all left out, which makes Omega_0
a function of the distribution alone, not of the token numbering.  With one
temperature per row this is the same as comparing target logits.  If
M >= V, Omega_0 is the whole vocabulary.  The scheme below returns target
tokens for any choice of Omega_0; the choice only moves the acceptance
rate.  With p_a = q(Omega_0) and q~ = q 1[Omega_0] / p_a:

1. The multi-draft scheme is run on the alphabet Omega_0 with target q~ and
   produces Y' ~ q~.  Reading of the two passages together: only the input
   tokens that lie in Omega_0 are kept (the non-iid remark), each with its
   draft law truncated to Omega_0, p~_d = p_d 1[Omega_0] / p_d(Omega_0).
   Conditioned on which branches land in Omega_0, the kept tokens are
   independent with exactly those laws, so the weighted importance stages
   (Remark 4) followed by Algorithm 1 against q~ give Y' ~ q~:
     - two or more kept tokens: the pairwise stages over the kept tokens in
       branch order, Omega_1 chosen inside Omega_0, selection uniform of
       stage m = draw m, then Algorithm 1 with q~ (accept draw 16, residual
       max(0, q~ - p_I) over Omega_0 with draw 32);
     - one kept token: Algorithm 1 with p_I = its truncated draft law;
     - no kept token: Y' is drawn from q~ directly (draw 32).
2. Y' is kept with probability p_a (draw 34); otherwise the output is drawn
   from Omega \\ Omega_0 in proportion to q (draw 35, inverse CDF in token-id
   order).  Then Pr(Z = x) = p_a q~(x) = q(x) on Omega_0 and
   (1 - p_a) q(x) / (1 - p_a) = q(x) outside it.
If Omega \\ Omega_0 carries no target mass (M >= V), Y' is always kept; if
Omega_0 is empty (ties at the top), the output is drawn from q (draw 35).

Top-k / top-p preprocessing (Section 5: top-p with p = 0.95 on both models;
top-k with k = 5 or 10 on both models)
---------------------------------------------------------------------------
A row's distribution is restricted to its k most probable tokens (ties:
lower id), then to the shortest prefix of those, in the same order, whose
mass reaches top_p times the mass kept by top-k (reading: the common
nucleus rule, top-k applied first), and renormalised.  The filtered rows
replace the target and draft distributions before any scheme runs; the
caller's draft tokens must have been drawn from the filtered draft rows.
"""
import numpy as np

from . import philox
from . import wis as wis_mod

DRAW_KEEP = 34       # keep Y' (drawn from q~) with probability p_a
DRAW_OUTSIDE = 35    # the replacement drawn from Omega minus Omega_0
BAND_KEEP = 1e-6     # |u - p_a|
BAND_NUCLEUS = 1e-9  # relative distance of the nucleus boundary to top_p


def top_order(dist):
    """Token ids by decreasing probability, ties to the lower id."""
    n = len(dist)
    return np.lexsort((np.arange(n), -np.asarray(dist, dtype=np.float64)))


def top_filter(dist, top_k=0, top_p=1.0, note=None):
    """Top-k then top-p restriction of one row, renormalised (Section 5).

    top_k <= 0 keeps every token; top_p >= 1 skips the nucleus step.  The
    nucleus is the shortest prefix of the top-k order whose cumulative mass
    is at least top_p times the top-k mass."""
    dist = np.asarray(dist, dtype=np.float64)
    order = top_order(dist)
    keep = order if top_k <= 0 else order[:min(int(top_k), len(dist))]
    if top_p < 1.0:
        c = np.cumsum(dist[keep])
        need = float(top_p) * c[-1]
        m = int(np.searchsorted(c, need, side="left")) + 1
        m = min(m, len(keep))
        if note is not None:
            lo = c[m - 2] if m >= 2 else 0.0
            note("nucleus", min(abs(c[m - 1] - need), abs(need - lo)) / c[-1], BAND_NUCLEUS)
        keep = keep[:m]
    out = np.zeros_like(dist)
    out[keep] = dist[keep]
    return out / out.sum()


def omega0(q, M):
    """Omega_0: the tokens with probability above the (M+1)-th largest one
    (every token if M >= V), in increasing token-id order."""
    q = np.asarray(q, dtype=np.float64)
    if int(M) >= len(q):
        return np.arange(len(q))
    cut = np.sort(q)[::-1][int(M)]
    return np.flatnonzero(q > cut)


def truncate(dist, om):
    """A row restricted to Omega_0 (given as sorted ids) and renormalised;
    None if it has no mass there."""
    sub = np.asarray(dist, dtype=np.float64)[om]
    tot = sub.sum()
    return None if tot <= 0.0 else sub / tot


def truncated_step(rec, q, dists, X, seed, sid, j, M, s):
    """One depth of the truncated-alphabet scheme (module docstring) with the
    weighted importance stages inside Omega_0.  ``dists`` are the valid
    branches' draft laws over the whole vocabulary, ``X`` their tokens.
    Returns the output token Z; ``rec`` receives the inner step's record
    (Y, q~(Y), p_I(Y), ratio in Omega_0 terms, Y as a vocabulary id)."""
    from .verify import BAND_CDF, _speculative_step, inverse_cdf
    om = omega0(q, M)
    rest = np.asarray(q, dtype=np.float64).copy()
    rest[om] = 0.0
    if len(om) == 0:
        z, m = inverse_cdf(rest, philox.uniform(seed, sid, j, DRAW_OUTSIDE))
        rec.note("cdf", m, BAND_CDF)
        return int(z)
    where = {int(t): i for i, t in enumerate(om)}
    pa = float(q[om].sum())
    qt = q[om] / pa
    kept = [(where[int(x)], truncate(p, om)) for x, p in zip(X, dists) if int(x) in where]
    # a token whose own draft law puts no mass on Omega_0 cannot have been drawn
    # there; such inconsistent input is dropped rather than kept
    kept = [(k, d) for k, d in kept if d is not None and d[k] > 0.0]
    if not kept:
        # no input token in Omega_0: Y' ~ q~ directly
        y, m = inverse_cdf(qt, philox.uniform(seed, sid, j, philox.DRAW_RESIDUAL))
        rec.note("cdf", m, BAND_CDF)
    else:
        Xk = [k for k, _ in kept]
        dk = [d for _, d in kept]
        us = [philox.uniform(seed, sid, j, philox.DRAW_SELECT + m) for m in range(len(Xk) - 1)]
        Y, pI = wis_mod.wis_select(rec, qt, dk, Xk, us, s)
        y = _speculative_step(rec, qt, pI, Y, philox.uniform(seed, sid, j, philox.DRAW_ACCEPT),
                              philox.uniform(seed, sid, j, philox.DRAW_RESIDUAL))
        rec.Y = int(om[Y])
    if rest.sum() <= 0.0:
        return int(om[y])
    u_keep = philox.uniform(seed, sid, j, DRAW_KEEP)
    rec.note("keep", abs(u_keep - pa), BAND_KEEP)
    if u_keep < pa:
        return int(om[y])
    z, m = inverse_cdf(rest, philox.uniform(seed, sid, j, DRAW_OUTSIDE))
    rec.note("cdf", m, BAND_CDF)
    return int(z)


def output_law(q, dists, M, s):
    """Law of Z for one depth of the truncated-alphabet scheme, by exhaustive
    enumeration of the draft tuple over Omega^K (tiny vocabularies): the
    membership pattern of the tuple in Omega_0 fixes the kept inputs, the
    kept inputs' WIS chain and Algorithm 1 are integrated analytically, then
    the keep / replace step.  Used to pin ``truncated_step``."""
    from . import enum
    q = np.asarray(q, dtype=np.float64)
    V = len(q)
    om = omega0(q, M)
    if len(om) == 0:
        return q.copy()
    where = {int(t): i for i, t in enumerate(om)}
    pa = float(q[om].sum())
    qt = q[om] / pa
    rest = q.copy()
    rest[om] = 0.0
    law0 = np.zeros(len(om))      # law of Y' over Omega_0
    cache = {}
    for x, pr in enum._tuples(dists):
        if pr == 0.0:
            continue
        keep_idx = tuple(i for i, xi in enumerate(x) if int(xi) in where)
        if not keep_idx:
            law0 += pr * qt
            continue
        if keep_idx not in cache:
            dk = [truncate(dists[i], om) for i in keep_idx]
            if len(dk) == 1:
                stages, pI = [], dk[0]
            else:
                stages = enum.wis_stages(qt, dk, s)
                pI = stages[-1].pI
            acc = np.minimum(1.0, np.where(pI > 0, qt / np.where(pI > 0, pI, 1.0), np.inf))
            r = np.maximum(0.0, qt - pI)
            res = r / r.sum() if r.sum() > 0 else qt
            cache[keep_idx] = (stages, acc, res)
        stages, acc, res = cache[keep_idx]
        xk = [where[int(x[i])] for i in keep_idx]
        beta = enum.wis_beta(stages, xk) if stages else {xk[0]: 1.0}
        for y, by in beta.items():
            law0[y] += pr * by * acc[y]
            law0 += pr * by * (1.0 - acc[y]) * res
    law = np.zeros(V)
    if rest.sum() <= 0.0:
        law[om] = law0
        return law
    law[om] = pa * law0
    law += (1.0 - pa) * rest / rest.sum()
    return law
