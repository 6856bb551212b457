"""Pins for the truncated LP with the sorted rule on Omega_2 (Eq. heur,
Algorithm 2, App. I).

The closed form of p_I is checked against exhaustive enumeration of the
selection rule over Omega^K, the whole step against target preservation,
the acceptance against the truncation bound printed after Eq. p_Ieq
(P~ >= P* - sum_{Omega_2} (q - p^2)^+, and its non-iid form), and with
s = |Omega| against Theorem 3.
"""
import numpy as np
import pytest

from oracle import enum, sorted_lp, theory
from oracle.verify import DepthRecord

RNG = np.random.default_rng(777)


def _dir(V, alpha=0.7):
    return RNG.dirichlet(np.full(V, alpha))


def _chain(q, dists, s):
    stages, a = [], dists[0]
    for m in range(1, len(dists)):
        st = sorted_lp.stage(q, a, dists[m], s)
        stages.append(st)
        a = st.pI
    return stages, a


def _law_enum(stages, dists, V):
    law = np.zeros(V)
    for x, pr in enum._tuples(dists):
        cur = {x[0]: 1.0}
        for m, st in enumerate(stages):
            nxt = {}
            for a_tok, pa in cur.items():
                for y, py in sorted_lp.beta(st, a_tok, x[m + 1]).items():
                    nxt[y] = nxt.get(y, 0.0) + pa * py
            cur = nxt
        for y, py in cur.items():
            law[y] += pr * py
    return law


@pytest.mark.parametrize("mids", [[0, 0], [0, 1], [0, 0, 0], [0, 1, 0], [1, 0, 1, 0]])
def test_closed_form_matches_enumeration(mids):
    for s in (1, 2, 3, 5):
        V = 5
        q = _dir(V)
        rows = {d: _dir(V) for d in set(mids)}
        dists = [rows[d] for d in mids]
        stages, pI = _chain(q, dists, s)
        np.testing.assert_allclose(_law_enum(stages, dists, V), pI, rtol=0, atol=1e-13)
        assert pI.sum() == pytest.approx(1.0, abs=1e-13)


def test_iid_omega2_formula_is_eq_p_Ieq():
    """i.i.d. inputs: p_I(k) = p_k^2 + sum_{i after k} 2 p_i p_k on Omega_2."""
    V, s = 8, 3
    p, q = _dir(V), _dir(V)
    st = sorted_lp.stage(q, p, p, s)
    for pos, k in enumerate(st.order[s:]):
        after = st.order[s + pos + 1:]
        assert st.pI[k] == pytest.approx(p[k] ** 2 + 2 * p[k] * p[after].sum(), abs=1e-15)


def test_truncation_bound_iid():
    """Section 4: P~ >= P* - sum_{Omega_2} (q - p^2)^+, P* from Theorem 3."""
    for _ in range(25):
        V = int(RNG.integers(3, 8))
        s = int(RNG.integers(1, V))
        p, q = _dir(V, 0.5), _dir(V, 0.5)
        st = sorted_lp.stage(q, p, p, s)
        pt = float(np.minimum(q, st.pI).sum())
        ps = theory.thm3_pstar(p, q)
        pen = float(np.maximum(0.0, q - p * p)[~st.in1].sum())
        assert ps - pen - 1e-6 <= pt <= ps + 1e-9


def test_truncation_bound_non_iid():
    for _ in range(10):
        V = int(RNG.integers(3, 6))
        s = int(RNG.integers(1, V))
        p1, p2, q = _dir(V, 0.6), _dir(V, 0.6), _dir(V, 0.6)
        st = sorted_lp.stage(q, p1, p2, s)
        pt = float(np.minimum(q, st.pI).sum())
        ps = theory.iws_optimum(q, [p1, p2])
        pen = float(np.maximum(0.0, q - p1 * p2)[~st.in1].sum())
        assert ps - pen - 1e-6 <= pt <= ps + 1e-7


def test_full_lp_when_s_is_v():
    for _ in range(10):
        V = int(RNG.integers(2, 6))
        p, q = _dir(V, 0.6), _dir(V, 0.6)
        st = sorted_lp.stage(q, p, p, V)
        assert float(np.minimum(q, st.pI).sum()) == pytest.approx(theory.thm3_pstar(p, q), abs=1e-5)


def test_sorted_rule_differs_from_the_variant_on_omega2():
    """The sorted rule gives Omega_2 tokens early in the key order more mass
    than the variant's 1/2 rule: the first Omega_2 token's p_I exceeds p_k P(Omega_2)."""
    from oracle import wis
    V, s = 7, 2
    p, q = _dir(V), _dir(V)
    st = sorted_lp.stage(q, p, p, s)
    var = wis.stage_law(q, p, p, s)
    k = st.order[s]
    assert st.pI[k] > var.pI[k]
    np.testing.assert_allclose(st.pI[st.omega1], var.pI[var.omega1], atol=1e-15)


def test_target_preserved_by_the_speculative_step():
    V = 5
    for mids in ([0, 0], [0, 1, 0]):
        q = _dir(V)
        rows = {d: _dir(V) for d in set(mids)}
        dists = [rows[d] for d in mids]
        stages, pI = _chain(q, dists, 2)
        law, _ = enum.output_law(q, dists, lambda x: _beta_chain(stages, x), pI)
        np.testing.assert_allclose(law, q, atol=1e-13)


def _beta_chain(stages, x):
    cur = {x[0]: 1.0}
    for m, st in enumerate(stages):
        nxt = {}
        for a_tok, pa in cur.items():
            for y, py in sorted_lp.beta(st, a_tok, x[m + 1]).items():
                nxt[y] = nxt.get(y, 0.0) + pa * py
        cur = nxt
    return cur


def test_sampler_follows_the_stage_law():
    """The sampled selection with Philox-free uniforms reproduces beta."""
    V = 6
    q, a, b = _dir(V), _dir(V), _dir(V)
    st = sorted_lp.stage(q, a, b, 3)
    N = 20000
    A = RNG.choice(V, size=N, p=a)
    B = RNG.choice(V, size=N, p=b)
    u = RNG.random(N)
    y = np.array([sorted_lp.select(st, int(x1), int(x2), float(uu)) for x1, x2, uu in zip(A, B, u)])
    emp = np.bincount(y, minlength=V) / N
    assert 0.5 * np.abs(emp - st.pI).sum() < 4.0 / np.sqrt(N)
    rec = DepthRecord(0)
    Y, pI = sorted_lp.sorted_select(rec, q, [a, b], [int(A[0]), int(B[0])], [0.3], 3)
    assert Y in (int(A[0]), int(B[0]))


def test_walk_first_token_follows_target():
    """The walk with the sorted rule: the first emitted token follows q
    (Monte Carlo over sequences, V = 4, K = 3)."""
    from oracle.verify import oracle_verify
    V, K, L, B = 4, 3, 2, 3000
    rng = np.random.default_rng(5)
    row = rng.normal(0.0, 1.0, size=V)
    tl = np.broadcast_to(row, (B, K, L + 1, V)).copy()
    drow = row + rng.normal(0.0, 1.0, size=V)
    drafts = [np.broadcast_to(drow, (B, L, V)).copy() for _ in range(K)]
    pd = np.exp(drow - drow.max())
    pd /= pd.sum()
    tokens = rng.choice(V, size=(B, K, L), p=pd)
    out, acc, _ = oracle_verify(tl, drafts, np.zeros(K, dtype=int), tokens, np.ones((B, 1 + K)), "WISsort",
                                seed=4, wis_s=2)
    q = np.exp(row - row.max())
    q /= q.sum()
    emp = np.bincount(out[:, 0], minlength=V) / B
    assert 0.5 * np.abs(emp - q).sum() < 4.0 / np.sqrt(B)
