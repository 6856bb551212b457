"""Oracle pins: exhaustive enumeration over Omega^K for tiny vocabularies.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

These functions compute the law of the intermediate token and of the output
token by summing over every draft tuple x in Omega^K with probability
prod_i p_{d(i)}(x_i) and integrating each uniform analytically.  They share no
arithmetic with the closed forms in ``wis`` and ``is_laplace`` (which they
pin): only the rule's fixed parameters (Omega_1 and the LP weights of each
stage) are taken from a stage object.
"""
import itertools

import numpy as np

from . import wis as wis_mod


def _tuples(dists):
    V = len(dists[0])
    for x in itertools.product(range(V), repeat=len(dists)):
        pr = 1.0
        for xi, p in zip(x, dists):
            pr *= p[xi]
        yield x, pr


def is_beta(q, dists, x):
    """Classical IS selection law given the tuple x: Pr(Y = y | x)."""
    V = len(q)
    rho = np.array([q[xi] / p[xi] for xi, p in zip(x, dists)])
    beta = np.zeros(V)
    tot = rho.sum()
    for xi, r in zip(x, rho):
        beta[xi] += r / tot
    return beta


def is_law_enum(q, dists):
    """p_I of classical importance sampling by enumeration (Section 3)."""
    V = len(q)
    pI = np.zeros(V)
    for x, pr in _tuples(dists):
        if pr > 0:
            pI += pr * is_beta(q, dists, x)
    return pI


def stage_beta(st, A, B):
    """Law of one WIS stage's output given ordered inputs (A, B), from the
    stage's Omega_1 and weights (selection rule of the variant truncated LP)."""
    if A == B:
        return {A: 1.0}
    ia, ib = st.in1[A], st.in1[B]
    if ia and ib:
        pa = int(np.searchsorted(st.omega1, A))
        pb = int(np.searchsorted(st.omega1, B))
        if pa < pb:
            wa = st.w[st.pair_index[(pa, pb)]]
        else:
            wa = 1.0 - st.w[st.pair_index[(pb, pa)]]
        return {A: wa, B: 1.0 - wa}
    if ia:
        return {A: 1.0}
    if ib:
        return {B: 1.0}
    return {A: 0.5, B: 0.5}


def wis_stages(q, dists, s):
    """The stage objects of the pairwise WIS chain (Remark 4) for the draft
    laws ``dists`` in branch order, built by the oracle."""
    stages = []
    a = dists[0]
    for m in range(1, len(dists)):
        st = wis_mod.stage_law(q, a, dists[m], s)
        stages.append(st)
        a = st.pI
    return stages


def wis_beta(stages, x):
    """Law of the chained WIS output given the whole tuple x."""
    cur = {x[0]: 1.0}
    for m, st in enumerate(stages):
        nxt = {}
        for a_tok, pa in cur.items():
            for y, py in stage_beta(st, a_tok, x[m + 1]).items():
                nxt[y] = nxt.get(y, 0.0) + pa * py
        cur = nxt
    return cur


def wis_law_enum(q, dists, s):
    """Law of the chained WIS output by enumeration over Omega^K."""
    V = len(q)
    stages = wis_stages(q, dists, s)
    pI = np.zeros(V)
    for x, pr in _tuples(dists):
        if pr == 0:
            continue
        for y, py in wis_beta(stages, x).items():
            pI[y] += pr * py
    return pI, stages


def output_law(q, dists, beta_fn, pI):
    """Law of Z after the speculative step (Algorithm 1) with intermediate
    law beta_fn(x) and the claimed p_I used for the accept test and the
    residual.  Also returns Pr(Z in S)."""
    V = len(q)
    acc = np.minimum(1.0, np.where(pI > 0, q / np.where(pI > 0, pI, 1.0), np.inf))
    r = np.maximum(0.0, q - pI)
    R = r.sum()
    res = r / R if R > 0 else q
    law = np.zeros(V)
    p_in_s = 0.0
    for x, pr in _tuples(dists):
        if pr == 0:
            continue
        sx = set(x)
        beta = beta_fn(x)
        items = beta.items() if isinstance(beta, dict) else [(y, by) for y, by in enumerate(beta) if by > 0]
        zx = np.zeros(V)
        for y, by in items:
            zx[y] += by * acc[y]
            zx += by * (1.0 - acc[y]) * res
        law += pr * zx
        p_in_s += pr * sum(zx[z] for z in sx)
    return law, p_in_s


def spectr_output_law(q, dists):
    """Law of Z under sequential rejection (the baseline reading) by
    enumeration: round i accepts x_i with probability min(1, q_i(x_i)/p_i(x_i))."""
    V = len(q)
    targets = [q]
    for p in dists:
        r = np.maximum(0.0, targets[-1] - p)
        targets.append(r / r.sum() if r.sum() > 0 else targets[-1])
    law = np.zeros(V)
    p_in_s = 0.0
    for x, pr in _tuples(dists):
        if pr == 0:
            continue
        zx = np.zeros(V)
        alive = 1.0
        for i, (xi, p) in enumerate(zip(x, dists)):
            a = min(1.0, targets[i][xi] / p[xi]) if p[xi] > 0 else 1.0
            zx[xi] += alive * a
            alive *= 1.0 - a
        zx += alive * targets[len(dists)]
        law += pr * zx
        p_in_s += pr * sum(zx[z] for z in set(x))
    return law, p_in_s
