"""Oracle: token-level multi-draft verification walked along the draft tree.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  Plain fp64 numpy; one
sequence at a time, one depth at a time, in the order the paper states the
steps.  Notation follows the paper: ``q`` is the target distribution, ``p``
(``p_d`` for draft model d) a draft distribution, ``p_I`` the distribution of
the intermediate token chosen by the importance step (Section 3, Definition 1
and Theorem 1).

Per depth j of sequence b:

1. temperature softmax of the target row and of one row per distinct draft
   model among the valid branches (Section 3: q(.) = M_b(.|u^t),
   p(.) = M_s(.|u^t); temperatures as in Section 5);
2. importance step -> intermediate token Y and its law p_I (scheme below);
3. single-draft speculative step on Y (Appendix A, Algorithm 1): accept with
   probability min(1, q(Y)/p_I(Y)), else sample the normalised residual
   max(0, q - p_I);
4. walk: the output Z continues the walk iff Z is one of the valid draft
   tokens (the selection rule's acceptance event Z in S, Section 3 / Problem
   1); the valid branches become those whose token is Z.  After L accepted
   positions a bonus token is drawn from the target row at depth L.

Schemes
-------
single   Algorithm 1 on the lowest valid branch (p_I = that branch's p).
IS       classical importance sampling, Pr(I = i) proportional to
         q(X_i)/p_{d(i)}(X_i) (Section 3, after Definition 1).  p_I has no
         closed form in the paper; it is evaluated through the identity
         p_I(y) = q(y) * sum_i int_0^inf exp(-t rho_i(y)) prod_{j!=i} M_j(t) dt,
         M_j(t) = sum_x p_{d(j)}(x) exp(-t rho_j(x)), rho_i(y) = q(y)/p_{d(i)}(y),
         integrated by the trapezoid rule in u = ln t (module ``is_laplace``).
WIS      the paper's weighted importance sampling with the variant truncated
         LP (Appendix "Variant of Truncated LP", Eq. heur2 / p_Ieq3), extended
         to K > 2 drafts by pairwise stages (Remark 4) and to distinct draft
         models by the non-iid form (Appendix "non-iid", key q - p_1 p_2)
         (module ``wis``).
SpecTr   sequential-rejection baseline (reading: Algorithm 1 applied to the
         valid drafts in turn against the running residual target).
WISsort  the truncated LP with the sorted rule on Omega_2 (Section 4 Eq. heur,
         Algorithm 2; module ``sorted_lp``), pairwise stages for K > 2.
WIS0     WIS on the truncated alphabet Omega_0 = the ``omega0`` most probable
         target tokens, followed by the keep / replace step that restores the
         target (Section 4, "truncated alphabet"; module ``truncated``).

Optional top-k / top-p preprocessing (Section 5) replaces the target and
draft rows by their filtered, renormalised versions before any scheme runs.

Each depth also records the margins of its discrete decisions; a depth whose
margin is below the band thresholds is flagged ``band`` (GPU and oracle may
legitimately differ there because they round differently).
"""
import numpy as np

from . import philox
from .philox import DRAW_ACCEPT, DRAW_BONUS, DRAW_RESIDUAL, DRAW_SELECT
from . import wis as wis_mod
from . import is_laplace
from . import truncated
from . import sorted_lp

SCHEMES = {"single": 0, "IS": 1, "WIS": 2, "SpecTr": 3, "WIS0": 4, "WISsort": 5}

# Band thresholds (absolute, on quantities in [0, 1] or scaled as stated).
BAND_ACCEPT = 1e-6   # |u - min(1, q(Y)/p_I(Y))|
BAND_CDF = 1e-6      # inverse-CDF boundary distance, relative to the total mass
BAND_SELECT = 1e-6   # selection uniform vs the selection threshold


def softmax_t(logits, temperature):
    """softmax(l / T) in fp64 (Section 5 sets temperatures on both models)."""
    x = np.asarray(logits, dtype=np.float64)
    m = x.max()
    e = np.exp((x - m) / float(temperature))
    return e / e.sum()


def inverse_cdf(r, u):
    """Smallest k with sum_{k' <= k} r_k' > u * sum(r), in token-id order.

    Returns (k, margin) where margin is the distance of the threshold to the
    nearest CDF boundary that decided k, relative to sum(r)."""
    c = np.cumsum(r)
    total = c[-1]
    t = u * total
    k = int(np.searchsorted(c, t, side="right"))
    k = min(k, len(r) - 1)
    hi = c[k]
    lo = c[k - 1] if k > 0 else 0.0
    margin = min(hi - t, t - lo) / total if total > 0 else 0.0
    return k, margin


class DepthRecord:
    """Per-(sequence, depth) diagnostics."""

    __slots__ = ("j", "Y", "Z", "ratio", "u_acc", "accepted", "margins", "band", "qY", "pIY", "in_S", "R")

    def __init__(self, j):
        self.j = j
        self.Y = -1
        self.Z = -1
        self.ratio = float("nan")
        self.u_acc = float("nan")
        self.accepted = False
        self.margins = {}
        self.band = False
        self.qY = float("nan")
        self.pIY = float("nan")
        self.in_S = False
        self.R = float("nan")   # residual mass sum max(0, q - p_I); 1 - R = sum min(q, p_I)

    def note(self, name, value, threshold):
        prev = self.margins.get(name, np.inf)
        self.margins[name] = min(prev, value)
        if value < threshold:
            self.band = True


def _speculative_step(rec, q, pI, Y, u_acc, u_res):
    """Algorithm 1 applied to the intermediate token Y with law p_I."""
    ratio = q[Y] / pI[Y] if pI[Y] > 0 else np.inf
    rec.Y = int(Y)
    rec.qY = float(q[Y])
    rec.pIY = float(pI[Y])
    rec.ratio = float(ratio)
    rec.u_acc = float(u_acc)
    # Theorem 1: the step accepts with probability sum_k min(q_k, p_I(k)) = 1 - R
    rec.R = float(np.maximum(0.0, q - pI).sum())
    acc_prob = min(1.0, ratio)
    rec.note("accept", abs(u_acc - acc_prob), BAND_ACCEPT)
    if u_acc < acc_prob:
        rec.accepted = True
        return int(Y)
    r = np.maximum(0.0, q - pI)
    if r.sum() <= 0.0:
        # Only reachable by rounding: sum(q) = sum(p_I) = 1 makes the residual
        # positive whenever a rejection can happen.  Reading: sample q.
        r = q
    z, m = inverse_cdf(r, u_res)
    rec.note("cdf", m, BAND_CDF)
    return z


def _spectr_step(rec, q, dists, X, seed, b, j):
    """Sequential rejection over the valid drafts (reading of SpecTr's
    'modified sequential rejection'): round i accepts X_i with probability
    min(1, q_i(X_i)/p_{d(i)}(X_i)); on rejection the target becomes
    q_{i+1} = max(0, q_i - p_{d(i)}) / R_i.  If every round rejects, Z is drawn
    from the last residual target."""
    qi = q.copy()
    for i, (x, p) in enumerate(zip(X, dists)):
        u = philox.uniform(seed, b, j, DRAW_ACCEPT + i)
        ratio = qi[x] / p[x] if p[x] > 0 else np.inf
        acc_prob = min(1.0, ratio)
        rec.note("accept", abs(u - acc_prob), BAND_ACCEPT)
        if i == 0:
            rec.Y = int(x)
            rec.ratio = float(ratio)
            rec.u_acc = float(u)
            rec.qY = float(qi[x])
            rec.pIY = float(p[x])
        if u < acc_prob:
            rec.accepted = True
            return int(x)
        r = np.maximum(0.0, qi - p)
        tot = r.sum()
        if tot > 0.0:
            qi = r / tot
        # tot <= 0 is only reachable by rounding (then q_i == p): keep q_i.
    z, m = inverse_cdf(qi, philox.uniform(seed, b, j, DRAW_RESIDUAL))
    rec.note("cdf", m, BAND_CDF)
    return z


def verify_sequence(b, target_logits, draft_logits, draft_model_id, draft_tokens, temperatures,
                    scheme, seed, wis_s=5, is_h=0.25, draw_id=None, omega0=40, top_k=0, top_p=1.0):
    """Walk the sequence stored at index b of the arrays; its Philox draws use
    sequence id ``draw_id`` (default b).  Returns (tokens [L+1] with -1
    padding, accept_len, list of DepthRecord)."""
    filt = top_k > 0 or top_p < 1.0

    def dist(logits, temperature, rec):
        d = softmax_t(logits, temperature)
        return truncated.top_filter(d, top_k, top_p, rec.note) if filt else d

    sid = b if draw_id is None else int(draw_id)
    K = target_logits.shape[1]
    L = draft_tokens.shape[2]
    out = np.full(L + 1, -1, dtype=np.int64)
    records = []
    valid = list(range(K))
    for j in range(L):
        rec = DepthRecord(j)
        records.append(rec)
        kstar = valid[0]
        q = dist(target_logits[b, kstar, j], temperatures[b, 0], rec)
        # one row per distinct draft model, read from its lowest valid branch
        rows = {}
        for k in valid:
            d = int(draft_model_id[k])
            if d not in rows:
                rows[d] = dist(draft_logits[k][b, j], temperatures[b, 1 + k], rec)
        X = [int(draft_tokens[b, k, j]) for k in valid]
        dists = [rows[int(draft_model_id[k])] for k in valid]
        if scheme == "single":
            Y, pI = X[0], dists[0]
            Z = _speculative_step(rec, q, pI, Y, philox.uniform(seed, sid, j, DRAW_ACCEPT),
                                  philox.uniform(seed, sid, j, DRAW_RESIDUAL))
        elif scheme == "IS":
            mids = [int(draft_model_id[k]) for k in valid]
            Y, pI = is_laplace.is_select(rec, q, rows, mids, X, philox.uniform(seed, sid, j, DRAW_SELECT), is_h)
            Z = _speculative_step(rec, q, pI, Y, philox.uniform(seed, sid, j, DRAW_ACCEPT),
                                  philox.uniform(seed, sid, j, DRAW_RESIDUAL))
        elif scheme == "WIS":
            us = [philox.uniform(seed, sid, j, DRAW_SELECT + m) for m in range(max(0, len(X) - 1))]
            Y, pI = wis_mod.wis_select(rec, q, dists, X, us, wis_s)
            Z = _speculative_step(rec, q, pI, Y, philox.uniform(seed, sid, j, DRAW_ACCEPT),
                                  philox.uniform(seed, sid, j, DRAW_RESIDUAL))
        elif scheme == "SpecTr":
            Z = _spectr_step(rec, q, dists, X, seed, sid, j)
        elif scheme == "WISsort":
            us = [philox.uniform(seed, sid, j, DRAW_SELECT + m) for m in range(max(0, len(X) - 1))]
            Y, pI = sorted_lp.sorted_select(rec, q, dists, X, us, wis_s)
            Z = _speculative_step(rec, q, pI, Y, philox.uniform(seed, sid, j, DRAW_ACCEPT),
                                  philox.uniform(seed, sid, j, DRAW_RESIDUAL))
        elif scheme == "WIS0":
            Z = truncated.truncated_step(rec, q, dists, X, seed, sid, j, omega0, wis_s)
        else:
            raise ValueError(f"unknown scheme {scheme!r}")
        rec.Z = int(Z)
        out[j] = Z
        if Z in X:
            rec.in_S = True
            valid = [k for k in valid if int(draft_tokens[b, k, j]) == Z]
        else:
            return out, j, records
    # all L positions accepted: bonus token from the target row at depth L
    rec = DepthRecord(L)
    records.append(rec)
    q = dist(target_logits[b, valid[0], L], temperatures[b, 0], rec)
    z, m = inverse_cdf(q, philox.uniform(seed, sid, L, DRAW_BONUS))
    rec.note("cdf", m, BAND_CDF)
    rec.Z = int(z)
    out[L] = z
    return out, L, records


def oracle_verify(target_logits, draft_logits, draft_model_id, draft_tokens, temperatures,
                  scheme, seed, wis_s=5, is_h=0.25, seqs=None, seq_ids=None, omega0=40, top_k=0, top_p=1.0):
    """Oracle over a batch.

    target_logits  [B, K, L+1, V] (any real dtype; upcast exactly to fp64)
    draft_logits   list of K arrays [B, L, V]
    draft_model_id [K] ints (equal id: i.i.d. drafts of one model)
    draft_tokens   [B, K, L] ints
    temperatures   [B, 1+K] (target, then per branch)
    seqs           optional iterable of sequence indices to evaluate
    seq_ids        optional global sequence ids of the B stored sequences (a
                   sample of a larger batch); Philox draws use these ids and
                   the results are keyed by them
    omega0         |Omega_0| of the truncated-alphabet scheme WIS0
    top_k, top_p   preprocessing of every row (0 / 1.0: off)

    Returns (out_tokens, accept_len, records {id: [DepthRecord]}).  Without
    seq_ids the arrays are [B, L+1] and [B] and rows of sequences not in
    ``seqs`` are -1; with seq_ids they are dicts keyed by the global id."""
    target_logits = np.asarray(target_logits)
    B, K = target_logits.shape[0], target_logits.shape[1]
    L = np.asarray(draft_tokens).shape[2]
    out = np.full((B, L + 1), -1, dtype=np.int64)
    acc = np.full(B, -1, dtype=np.int64)
    recs = {}
    temps = np.asarray(temperatures, dtype=np.float64)
    if seq_ids is not None:
        out_d, acc_d = {}, {}
        for i, sid in enumerate(seq_ids):
            o, a, r = verify_sequence(i, target_logits, draft_logits, draft_model_id, draft_tokens, temps,
                                      scheme, seed, wis_s, is_h, draw_id=sid, omega0=omega0,
                                      top_k=top_k, top_p=top_p)
            out_d[int(sid)], acc_d[int(sid)], recs[int(sid)] = o, a, r
        return out_d, acc_d, recs
    for b in (range(B) if seqs is None else seqs):
        o, a, r = verify_sequence(b, target_logits, draft_logits, draft_model_id, draft_tokens,
                                  temps, scheme, seed, wis_s, is_h, omega0=omega0, top_k=top_k, top_p=top_p)
        out[b] = o
        acc[b] = a
        recs[b] = r
    return out, acc, recs
