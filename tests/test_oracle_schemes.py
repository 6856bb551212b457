"""Pins for the oracle's selection schemes.

The closed forms for p_I (module oracle.wis and oracle.is_laplace) are checked
against exhaustive enumeration of the selection rule over Omega^K, the
speculative step against exact target preservation, the WIS stage LP against
the min-cut formula and a direct HiGHS solve, and the truncated scheme
against the paper's truncation bound.
"""
import numpy as np
import pytest

from oracle import enum, is_laplace, theory, wis

RNG = np.random.default_rng(1234)


def _dir(V, alpha=1.0):
    return RNG.dirichlet(np.full(V, alpha))


# ----------------------------------------------------------------- plain IS


@pytest.mark.parametrize("K", [2, 3, 4])
def test_is_law_iid_matches_enumeration(K):
    for V in (2, 4, 6):
        for alpha in (0.4, 2.0):
            p, q = _dir(V, alpha), _dir(V, alpha)
            want = enum.is_law_enum(q, [p] * K)
            got = is_laplace.is_law(q, {0: p}, {0: K}, 0.25)
            np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-15)


def test_is_law_distinct_models_matches_enumeration():
    for mids in ([0, 1], [0, 1, 2], [0, 0, 1], [1, 0, 1, 0]):
        V = 5
        rows = {d: _dir(V, 0.8) for d in set(mids)}
        q = _dir(V, 0.8)
        want = enum.is_law_enum(q, [rows[d] for d in mids])
        counts = {d: mids.count(d) for d in set(mids)}
        got = is_laplace.is_law(q, rows, counts, 0.25)
        np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-15)
        assert got.sum() == pytest.approx(1.0, abs=1e-12)


def test_is_law_quadrature_step_converged():
    """Halving h leaves p_I unchanged to rounding (the trapezoid rule in ln t
    is geometrically convergent for this integrand)."""
    p, q = _dir(8, 0.3), _dir(8, 0.3)
    a = is_laplace.is_law(q, {0: p}, {0: 3}, 0.25)
    b = is_laplace.is_law(q, {0: p}, {0: 3}, 0.125)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-16)


def test_is_law_single_draft_is_p():
    p, q = _dir(6), _dir(6)
    np.testing.assert_allclose(is_laplace.is_law(q, {0: p}, {0: 1}, 0.25), p, rtol=1e-11)


# ----------------------------------------------------------------- WIS


@pytest.mark.parametrize("s", [1, 2, 3, 5])
def test_wis_law_iid_matches_enumeration(s):
    for K in (2, 3, 4):
        V = 5
        p, q = _dir(V, 0.7), _dir(V, 0.7)
        got, stages = enum.wis_law_enum(q, [p] * K, s)
        np.testing.assert_allclose(stages[-1].pI, got, rtol=1e-12, atol=1e-16)
        assert stages[-1].pI.sum() == pytest.approx(1.0, abs=1e-12)


@pytest.mark.parametrize("s", [1, 2, 4])
def test_wis_law_distinct_matches_enumeration(s):
    for K in (2, 3):
        V = 5
        ps = [_dir(V, 0.7) for _ in range(K)]
        q = _dir(V, 0.7)
        got, stages = enum.wis_law_enum(q, ps, s)
        np.testing.assert_allclose(stages[-1].pI, got, rtol=1e-12, atol=1e-16)


def test_wis_iid_stage1_omega2_is_p_times_mass():
    """Variant truncated LP, i.i.d. inputs: p_I(k) = p_k P(Omega_2) on Omega_2."""
    p, q = _dir(9), _dir(9)
    st = wis.stage_law(q, p, p, 3)
    om2 = ~st.in1
    np.testing.assert_allclose(st.pI[om2], p[om2] * p[om2].sum(), rtol=1e-13)


def test_printed_omega2_formula_does_not_normalise():
    """Documents the reading of the garbled Omega_2 formula of the variant
    truncated LP: summing p_i p_k over every i != k (as printed) does not give
    a distribution, the Omega_2-only reading does."""
    p, q = _dir(12), _dir(12)
    st = wis.stage_law(q, p, p, 4)
    om2 = ~st.in1
    printed = st.pI.copy()
    printed[om2] = p[om2] ** 2 + p[om2] * (1.0 - p[om2])
    assert abs(printed.sum() - 1.0) > 1e-3
    assert st.pI.sum() == pytest.approx(1.0, abs=1e-12)


def test_wis_omega1_is_topk_by_key():
    p, q = _dir(30, 0.5), _dir(30, 0.5)
    st = wis.stage_law(q, p, p, 5)
    key = q - p * p
    thr = np.sort(key)[-5]
    assert set(st.omega1) == set(np.flatnonzero(key >= thr))


def test_wis_stage_lp_is_optimal():
    """Max-flow value = min-cut formula, and sum_{Omega_1} min(q, p_I) equals
    the stage LP optimum solved directly."""
    for trial in range(30):
        V = int(RNG.integers(3, 10))
        s = int(RNG.integers(2, 6))
        a, b, q = _dir(V, 0.5), _dir(V, 0.5), _dir(V, 0.5)
        if trial % 2:
            b = a
        st = wis.stage_law(q, a, b, s)
        s_eff = len(st.omega1)
        assert st.flow_value == pytest.approx(theory.stage_min_cut(st.d, st.m, s_eff), abs=1e-12)
        got = float(np.sum(np.minimum(q[st.omega1], st.pI[st.omega1])))
        assert got == pytest.approx(theory.stage_lp_optimum(q, a, b, st.omega1), abs=1e-5)


def test_truncation_bound_iid():
    """Section 4, Eq. (p_acc_bnd): P* - sum_{Omega_2}(q - p^2)^+ <= P~ <= P*."""
    for _ in range(20):
        V = int(RNG.integers(3, 8))
        s = int(RNG.integers(1, V))
        p, q = _dir(V, 0.5), _dir(V, 0.5)
        st = wis.stage_law(q, p, p, s)
        pt = float(np.sum(np.minimum(q, st.pI)))
        ps = theory.thm3_pstar(p, q)
        pen = float(np.sum(np.maximum(0.0, q - p * p)[~st.in1]))
        assert ps - pen - 1e-6 <= pt <= ps + 1e-9


def test_truncation_bound_non_iid():
    """Non-iid appendix: P~ >= P* - sum_{Omega_2}(q - p_1 p_2)^+, P* from the
    importance-weighted LP of Theorem 1 with distinct drafts."""
    for _ in range(10):
        V = int(RNG.integers(3, 6))
        s = int(RNG.integers(1, V))
        p1, p2, q = _dir(V, 0.6), _dir(V, 0.6), _dir(V, 0.6)
        st = wis.stage_law(q, p1, p2, s)
        pt = float(np.sum(np.minimum(q, st.pI)))
        ps = theory.iws_optimum(q, [p1, p2])
        pen = float(np.sum(np.maximum(0.0, q - p1 * p2)[~st.in1]))
        assert ps - pen - 1e-6 <= pt <= ps + 1e-7


def test_wis_full_lp_matches_theorem3_when_s_is_v():
    """With s = |Omega| the truncated LP is the full K = 2 LP: its acceptance
    equals Theorem 3."""
    for _ in range(10):
        V = int(RNG.integers(2, 6))
        p, q = _dir(V, 0.6), _dir(V, 0.6)
        st = wis.stage_law(q, p, p, V)
        assert float(np.sum(np.minimum(q, st.pI))) == pytest.approx(theory.thm3_pstar(p, q), abs=1e-5)


# ----------------------------------------------------- target preservation


def _cases():
    V = 5
    p, q, p2 = _dir(V, 0.6), _dir(V, 0.6), _dir(V, 0.6)
    onehot = np.zeros(V)
    onehot[2] = 1.0
    return [
        ("iid2", q, [p, p]),
        ("iid3", q, [p, p, p]),
        ("distinct", q, [p, p2]),
        ("mixed", q, [p, p2, p]),
        ("p_eq_q", q, [q, q]),
        ("onehot_q", onehot, [p, p]),
        ("K1", q, [p]),
    ]


@pytest.mark.parametrize("case", range(7))
def test_target_preservation_all_schemes(case):
    """Theorem 1's two-step scheme (any importance step + Algorithm 1) and the
    sequential-rejection baseline emit Z ~ q exactly."""
    name, q, dists = _cases()[case]
    # single draft: p_I = p of the first draft
    law, _ = enum.output_law(q, dists, lambda x: {x[0]: 1.0}, dists[0])
    np.testing.assert_allclose(law, q, atol=1e-13)
    # plain IS
    mids = []
    rows = {}
    for p in dists:
        key = next((d for d, r in rows.items() if r is p), None)
        if key is None:
            key = len(rows)
            rows[key] = p
        mids.append(key)
    counts = {d: mids.count(d) for d in rows}
    if np.all(q > 0):
        pI = is_laplace.is_law(q, rows, counts, 0.25)
        law, pacc = enum.output_law(q, dists, lambda x: enum.is_beta(q, dists, x), pI)
        np.testing.assert_allclose(law, q, atol=1e-12)
    # WIS
    for s in (1, 2, 5):
        stages = enum.wis_stages(q, dists, s)
        pI = stages[-1].pI if stages else dists[0]
        law, pacc = enum.output_law(q, dists, (lambda x: enum.wis_beta(stages, x)) if stages else
                                    (lambda x: {x[0]: 1.0}), pI)
        np.testing.assert_allclose(law, q, atol=1e-13)
        assert pacc >= float(np.sum(np.minimum(q, pI))) - 1e-12
    # sequential rejection
    law, _ = enum.spectr_output_law(q, dists)
    np.testing.assert_allclose(law, q, atol=1e-13)


def test_k2_wis_with_full_lp_attains_theorem3():
    """The canonical decomposition with the optimal weights attains P*: with
    s = |Omega|, sum_y min(q, p_I) (the probability that Algorithm 1 accepts
    the intermediate token) equals Theorem 3's expression."""
    V = 4
    p, q = _dir(V), _dir(V)
    stages = enum.wis_stages(q, [p, p], V)
    assert float(np.sum(np.minimum(q, stages[0].pI))) == pytest.approx(theory.thm3_pstar(p, q), abs=1e-5)
