"""The pins catch plausible mistakes: each test plants one mistake in a copy
of an oracle step (on the CPU) and checks that the quantity the pin compares
moves well outside the pin's tolerance."""
import numpy as np

from oracle import enum, sorted_lp, theory, truncated

RNG = np.random.default_rng(2024)


def _dir(V, alpha=0.7):
    return RNG.dirichlet(np.full(V, alpha))


def test_truncated_law_pin_catches_a_missing_renormalisation(monkeypatch):
    q, p1, p2 = _dir(5), _dir(5), _dir(5)
    assert np.abs(truncated.output_law(q, [p1, p2, p1], 3, 2) - q).max() < 1e-12
    monkeypatch.setattr(truncated, "truncate", lambda d, om: np.asarray(d, dtype=np.float64)[om])
    assert np.abs(truncated.output_law(q, [p1, p2, p1], 3, 2) - q).max() > 1e-3


def test_truncated_law_pin_catches_the_untruncated_target():
    """Running the inner scheme against q instead of q~ (no renormalisation
    by p_a) breaks the law of Z."""
    q, p = _dir(5), _dir(5)
    om = truncated.omega0(q, 3)
    pa = q[om].sum()
    good = truncated.output_law(q, [p, p], 3, 2)
    # the inner step's law against q restricted (not renormalised) to Omega_0
    qt_bad = q[om]
    laws = [truncated.truncate(p, om)] * 2
    stages = enum.wis_stages(qt_bad, laws, 2)
    pI = stages[-1].pI
    acc = np.minimum(1.0, qt_bad / pI)
    r = np.maximum(0.0, qt_bad - pI)
    res = r / r.sum()
    law_y = pI * acc + (1.0 - (pI * acc).sum()) * res
    assert abs(law_y.sum() - 1.0) < 1e-12
    bad = q.copy()
    bad[om] = pa * law_y
    assert np.abs(good - q).max() < 1e-12 and np.abs(bad - q).max() > 1e-3


def test_sorted_scan_pin_catches_a_reversed_order():
    worst = 0.0
    for _ in range(30):
        V = int(RNG.integers(3, 8))
        p, q = _dir(V), _dir(V)
        ratio = q / p
        order = np.argsort(-ratio)                       # planted: largest ratio first
        Q = np.concatenate([[0.0], np.cumsum(q[order])])
        P = np.concatenate([[0.0], np.cumsum(p[order])])
        wrong = float(np.min(Q - P ** 2) + 1.0)
        worst = max(worst, abs(wrong - theory.thm3_pstar(p, q)))
    assert worst > 1e-3


def test_sorted_lp_pin_catches_prefix_instead_of_suffix_sums():
    q, a, b = _dir(6), _dir(6), _dir(6)
    st = sorted_lp.stage(q, a, b, 2)
    tail = st.order[2:]
    # planted: Omega_2 tokens collect the pairs with tokens BEFORE them in key order
    a_before = np.concatenate([[0.0], np.cumsum(a[tail])[:-1]])
    b_before = np.concatenate([[0.0], np.cumsum(b[tail])[:-1]])
    wrong = st.pI.copy()
    wrong[tail] = a[tail] * b[tail] + b[tail] * a_before + a[tail] * b_before
    law = np.zeros(6)
    for x, pr in enum._tuples([a, b]):
        for y, py in sorted_lp.beta(st, x[0], x[1]).items():
            law[y] += pr * py
    assert np.abs(law - st.pI).max() < 1e-13
    assert np.abs(law - wrong).max() > 1e-3
