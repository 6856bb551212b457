"""Pins that tie the brute-force programs to the paper's theorems.

Each test compares two independently computed quantities the paper states
are equal (a linear program solved by HiGHS against a closed form, or two
different programs), so that a mistake in either shows up.
"""
import os

import numpy as np
import pytest

from oracle import theory

RNG = np.random.default_rng(2410_18234)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "example1.txt")


def _dirichlet(V, alpha=1.0):
    return RNG.dirichlet(np.full(V, alpha))


@pytest.mark.parametrize("V,K", [(2, 2), (3, 2), (4, 2), (3, 3)])
def test_theorem1_tlsr_equals_iws(V, K):
    """Theorem 1: the optimal token-level selection rule (Problem 1) attains
    the importance-weighted-sampling optimum of Eq. (IS-opt1a)."""
    for _ in range(4):
        p, q = _dirichlet(V, 0.7), _dirichlet(V, 0.7)
        assert theory.tlsr_optimum(q, [p] * K) == pytest.approx(theory.iws_optimum(q, [p] * K), abs=1e-9)


def test_theorem1_extends_to_distinct_drafts():
    """Remark 1 / Theorem 4: the decomposition holds for independent drafts
    from different distributions."""
    for _ in range(4):
        ps = [_dirichlet(3), _dirichlet(3)]
        q = _dirichlet(3)
        assert theory.tlsr_optimum(q, ps) == pytest.approx(theory.iws_optimum(q, ps), abs=1e-9)


def test_single_draft_acceptance_is_one_minus_tv():
    """Appendix A: for K = 1 the optimum is sum_x min(p(x), q(x))."""
    for V in (2, 3, 5):
        p, q = _dirichlet(V), _dirichlet(V)
        assert theory.tlsr_optimum(q, [p]) == pytest.approx(theory.single_draft_acceptance(p, q), abs=1e-9)
        assert theory.single_draft_acceptance(p, q) == pytest.approx(1 - 0.5 * np.abs(p - q).sum(), abs=1e-12)


@pytest.mark.parametrize("V", [2, 3, 4, 5, 6])
def test_theorem3_closed_form_equals_lp(V):
    """Theorem 3: for K = 2 i.i.d. drafts P* equals the subset minimum of Eq. (opt)."""
    for alpha in (0.3, 1.0, 3.0):
        p, q = _dirichlet(V, alpha), _dirichlet(V, alpha)
        assert theory.thm3_pstar(p, q) == pytest.approx(theory.iws_optimum(q, [p, p]), abs=1e-9)


@pytest.mark.parametrize("V", [3, 5, 8])
def test_remark2_form_equals_theorem3(V):
    """Remark 2: Eq. (opt) equals min_S {sum_S q - (sum_S p)^2 + 1}."""
    for _ in range(5):
        p, q = _dirichlet(V), _dirichlet(V)
        assert theory.remark2_pstar(p, q) == pytest.approx(theory.thm3_pstar(p, q), abs=1e-12)


def test_theorem2_condition_iff_pstar_one():
    """Theorem 2: P* = 1 iff sum_S q >= (sum_S p)^2 for all S (K = 2)."""
    seen = {True: 0, False: 0}
    for _ in range(60):
        V = int(RNG.integers(2, 5))
        p = _dirichlet(V, 2.0)
        # q near p so that both outcomes occur
        q = np.abs(p + RNG.normal(0, 0.08, V))
        q /= q.sum()
        cond = theory.thm2_condition(p, q)
        pstar = theory.iws_optimum(q, [p, p])
        margin = min(sum(q[i] for i in range(V) if m >> i & 1) - sum(p[i] for i in range(V) if m >> i & 1) ** 2
                     for m in range(1, (1 << V) - 1))
        if abs(margin) < 1e-7:
            continue
        seen[cond] += 1
        assert (pstar > 1 - 1e-9) == cond
    assert seen[True] > 3 and seen[False] > 3


def test_example1_golden():
    """Section 3, Example 1 (printed statement, tests/golden/example1.txt)."""
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert len(rows) >= 10
    p = np.array([0.5, 0.5])
    for q1, k2, k1 in rows:
        q = np.array([float(q1), 1 - float(q1)])
        assert (theory.iws_optimum(q, [p, p]) > 1 - 1e-9) == bool(int(k2))
        assert (theory.thm3_pstar(p, q) > 1 - 1e-9) == bool(int(k2))
        assert (theory.single_draft_acceptance(p, q) > 1 - 1e-9) == bool(int(k1))


def test_three_letter_conditions():
    """Appendix (proof of Theorem 2, Omega = {1,2,3}): P* = 1 iff
    q_i >= p_i^2 and q_i + q_j >= (p_i + p_j)^2 for all i, j."""
    for _ in range(30):
        p = _dirichlet(3, 3.0)
        q = np.abs(p + RNG.normal(0, 0.1, 3))
        q /= q.sum()
        cond = all(q[i] >= p[i] ** 2 for i in range(3)) and all(
            q[i] + q[j] >= (p[i] + p[j]) ** 2 for i in range(3) for j in range(i + 1, 3))
        assert cond == theory.thm2_condition(p, q)
        assert (theory.thm3_pstar(p, q) > 1 - 1e-12) == cond


def test_figure2_optimal_curves_reach_one_on_the_predicted_range():
    """Figure 2 setting: p uniform on 3 letters, q = [1/3, q2, 2/3 - q2] and
    [1/6, q2, 5/6 - q2].  By Theorem 2 the optimum is 1 exactly for q2 in
    [1/9, 5/9] (left) and [5/18, 5/9] (right); Theorem 3 and the LP agree."""
    p = np.full(3, 1 / 3)
    for first, lo, hi in ((1 / 3, 1 / 9, 5 / 9), (1 / 6, 5 / 18, 5 / 9)):
        for q2 in np.linspace(0.0, 1.0 - first, 23):
            q = np.array([first, q2, 1 - first - q2])
            pstar = theory.thm3_pstar(p, q)
            assert pstar == pytest.approx(theory.iws_optimum(q, [p, p]), abs=1e-9)
            if lo + 1e-9 < q2 < hi - 1e-9:
                assert pstar == pytest.approx(1.0, abs=1e-12)
            elif q2 < lo - 1e-9 or q2 > hi + 1e-9:
                assert pstar < 1 - 1e-9


def test_sorted_scan_equals_subset_minimum():
    """The ratio-sorted prefix scan gives Theorem 3's subset minimum (K = 2)
    and Remark 2's conjectured form (K = 3, 4) exactly, on random rows with
    zeros in p and in q."""
    rng = np.random.default_rng(31)
    for _ in range(60):
        V = int(rng.integers(1, 10))
        p = rng.dirichlet(np.full(V, 0.6))
        q = rng.dirichlet(np.full(V, 0.6))
        if V > 2:
            p[rng.integers(0, V)] = 0.0
            q[rng.integers(0, V)] = 0.0
            p /= p.sum()
            q /= q.sum()
        assert theory.pstar_sorted(p, q) == pytest.approx(theory.thm3_pstar(p, q), abs=1e-12)
        for K in (3, 4):
            assert theory.pstar_sorted(p, q, K) == pytest.approx(theory.remark2_pstar(p, q, K), abs=1e-12)


def test_sorted_scan_example1_and_large_rows():
    """Example 1's interval (P* = 1 on [0.25, 0.75]) and, on a 50000-token
    row, the sandwich 1 - TV(p, q) <= P*(K=2) <= 1 (two drafts do no worse
    than one)."""
    p = np.array([0.5, 0.5])
    for q1, want_one in ((0.2, False), (0.25, True), (0.5, True), (0.75, True), (0.8, False)):
        v = theory.pstar_sorted(p, np.array([q1, 1 - q1]))
        assert (abs(v - 1.0) < 1e-12) == want_one
    rng = np.random.default_rng(2)
    lq = 4.0 * rng.standard_normal(50000)
    lp = lq + rng.standard_normal(50000)
    q = np.exp(lq - lq.max()); q /= q.sum()
    p = np.exp(lp - lp.max()); p /= p.sum()
    v = theory.pstar_sorted(p, q)
    assert np.minimum(p, q).sum() - 1e-12 <= v <= 1.0 + 1e-12
