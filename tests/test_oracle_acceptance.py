"""Pins for the per-depth acceptance probability the oracle records.

Theorem 1: the two-step scheme accepts the intermediate token with
probability sum_k min(q_k, p_I(k)) = 1 - R, R = sum_k max(0, q_k - p_I(k)).
Checked against the single-draft closed form 1 - TV(p, q) (App. A), against
Theorem 3's optimum for K = 2 i.i.d. drafts when the WIS LP is not truncated
(s = |Omega|), and against the empirical accept rate of the sampler.
"""
import numpy as np
import pytest

from oracle import theory
from oracle.verify import oracle_verify


def _rows(V, B, K, L, seed, sigma=1.0):
    rng = np.random.default_rng(seed)
    row = rng.normal(0.0, 1.5, size=V)
    tl = np.broadcast_to(row, (B, K, L + 1, V)).copy()
    drow = row + rng.normal(0.0, sigma, size=V)
    drafts = [np.broadcast_to(drow, (B, L, V)).copy() for _ in range(K)]
    pd = np.exp(drow - drow.max())
    pd /= pd.sum()
    q = np.exp(row - row.max())
    q /= q.sum()
    tokens = rng.choice(V, size=(B, K, L), p=pd)
    return tl, drafts, np.zeros(K, dtype=int), tokens, np.ones((B, 1 + K)), q, pd


def test_single_draft_is_one_minus_tv():
    tl, dr, mids, tok, temps, q, p = _rows(7, 4, 1, 1, seed=1)
    _, _, recs = oracle_verify(tl, dr, mids, tok, temps, "single", seed=3)
    for b in recs:
        assert 1.0 - recs[b][0].R == pytest.approx(np.minimum(p, q).sum(), abs=1e-14)


def test_untruncated_wis_attains_theorem3():
    for seed in range(4):
        V = 5
        tl, dr, mids, tok, temps, q, p = _rows(V, 3, 2, 1, seed=seed)
        _, _, recs = oracle_verify(tl, dr, mids, tok, temps, "WIS", seed=1, wis_s=V)
        for b in recs:
            if tok[b, 0, 0] == tok[b, 1, 0]:
                continue    # one valid token value: the step is Algorithm 1 on p
            assert 1.0 - recs[b][0].R == pytest.approx(theory.thm3_pstar(p, q), abs=1e-6)


@pytest.mark.parametrize("scheme", ["WIS", "IS"])
def test_accept_rate_matches(scheme):
    """Same rows for every sequence, independent draws: the fraction of
    accepted depth-0 steps estimates 1 - R (binomial 4 sigma)."""
    V, B = 6, 4000
    tl, dr, mids, tok, temps, q, p = _rows(V, B, 3, 1, seed=9)
    _, _, recs = oracle_verify(tl, dr, mids, tok, temps, scheme, seed=17)
    acc = np.array([recs[b][0].accepted for b in range(B)], dtype=float)
    pacc = np.array([1.0 - recs[b][0].R for b in range(B)])
    # p_I, hence R, depends on which draft values were drawn; the mean of the
    # per-sequence acceptance probabilities is the expected rate
    m = pacc.mean()
    assert abs(acc.mean() - m) < 4.0 * np.sqrt(m * (1 - m) / B)


def test_analytic_evaluator_matches_the_walk_and_the_ceiling():
    """oracle.acceptance: single / IS / WIS / WISsort equal 1 - R of the walk's depth 0;
    every scheme stays below Theorem 3's optimum for K = 2 i.i.d. drafts (the
    optimum over all token-level selection rules)."""
    from oracle import acceptance
    for seed in range(5):
        V, B = 6, 2
        tl, dr, mids, tok, temps, q, p = _rows(V, B, 2, 1, seed=40 + seed)
        best = theory.thm3_pstar(p, q)
        assert acceptance.optimal_acceptance(q, p, 2) == pytest.approx(best, abs=1e-12)
        for scheme in ("single", "IS", "WIS", "WISsort", "SpecTr"):
            val = acceptance.scheme_acceptance(q, [p, p], [0, 0], scheme)
            assert val <= best + 1e-9, (scheme, val, best)
            if scheme == "SpecTr":
                continue
            _, _, recs = oracle_verify(tl, dr, mids, tok, temps, scheme, seed=1)
            for b in recs:
                if scheme != "single" and tok[b, 0, 0] == tok[b, 1, 0]:
                    continue   # one distinct token: the walk's step is Algorithm 1 on p
                assert 1.0 - recs[b][0].R == pytest.approx(val, abs=1e-9), (scheme, b)


def test_spectr_evaluator_matches_its_sampler():
    from oracle import acceptance
    V, B = 5, 4000
    tl, dr, mids, tok, temps, q, p = _rows(V, B, 3, 1, seed=3)
    _, _, recs = oracle_verify(tl, dr, mids, tok, temps, "SpecTr", seed=8)
    rate = np.mean([recs[b][0].accepted for b in range(B)])
    want = acceptance.scheme_acceptance(q, [p, p, p], [0, 0, 0], "SpecTr")
    assert abs(rate - want) < 4.0 * np.sqrt(want * (1 - want) / B)


def test_truncated_evaluator_matches_enumeration():
    """WIS0's acceptance by its membership-pattern formula equals a direct
    enumeration of the draft tuple: for each tuple, the kept inputs' stage
    chain selects Y with law beta(. | tuple), Algorithm 1 against q~ accepts
    with min(1, q~(Y)/p_I(Y)), and the p_a test keeps it."""
    from oracle import acceptance, enum, truncated
    rng = np.random.default_rng(12)
    for V, K, M in ((5, 2, 3), (5, 3, 2), (6, 3, 4), (4, 2, 4)):
        q = rng.dirichlet(np.full(V, 0.7))
        rows = [rng.dirichlet(np.full(V, 0.7)) for _ in range(2)]
        dists = [rows[k % 2] for k in range(K)]
        om = truncated.omega0(q, M)
        where = {int(t): i for i, t in enumerate(om)}
        pa = q[om].sum()
        qt = q[om] / pa
        laws = [truncated.truncate(d, om) for d in dists]
        want = 0.0
        for x, pr in enum._tuples(dists):
            kept = [i for i in range(K) if int(x[i]) in where]
            if pr == 0.0 or not kept:
                continue
            xs = [where[int(x[i])] for i in kept]
            if len(kept) == 1:
                beta, pI = {xs[0]: 1.0}, laws[kept[0]]
            else:
                stages = enum.wis_stages(qt, [laws[i] for i in kept], 2)
                beta, pI = enum.wis_beta(stages, xs), stages[-1].pI
            want += pr * sum(by * min(1.0, qt[y] / pI[y]) for y, by in beta.items())
        got = acceptance.truncated_acceptance(q, dists, M, s=2)
        assert got == pytest.approx(pa * want, abs=1e-12)


def test_wis_reaches_theorem3_when_the_target_keeps_at_most_s_tokens():
    """A positive key q - p^2 needs q > 0, so with at most s target tokens
    every positive key lies in Omega_1; a target token with a negative key
    already has p_I >= p^2 > q, and tokens outside the target's support add
    nothing to sum min(q, p_I).  The truncated LP (either Omega_2 rule) then
    attains the full optimum: Theorem 3 for K = 2 i.i.d. drafts, up to the
    stage LP's saturation threshold (residuals at or below 1e-6 of the
    stage's mass count as zero, so a few such residuals may stay unserved).
    Checked on top-k restricted rows (Section 5's setting) with s = 5."""
    from oracle import acceptance, truncated
    rng = np.random.default_rng(21)
    for trial in range(40):
        V = int(rng.integers(6, 60))
        k = int(rng.integers(1, 6))
        q = truncated.top_filter(rng.dirichlet(np.full(V, 0.5)), top_k=k)
        p = rng.dirichlet(np.full(V, 0.5))
        if trial % 2:
            p = truncated.top_filter(p, top_k=int(rng.integers(1, 12)))
        best = acceptance.optimal_acceptance(q, p, 2)
        for scheme in ("WIS", "WISsort"):
            val = acceptance.scheme_acceptance(q, [p, p], [0, 0], scheme)
            assert best - 1e-5 <= val <= best + 1e-9, (trial, scheme, val, best)
