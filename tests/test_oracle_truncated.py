"""Pins for the truncated-alphabet scheme and the top-k / top-p filters.

The truncated-alphabet scheme (Section 4) must return tokens distributed
exactly as the target: checked by exhaustive enumeration of the draft tuple
(law of Z equal to q to rounding) and by a Monte Carlo run of the sampler
itself.  With Omega_0 = Omega it reduces to plain WIS draw for draw.  The
filters are checked on hand-made rows with exact binary masses.
"""
import numpy as np
import pytest

from oracle import philox, truncated
from oracle.verify import DepthRecord, oracle_verify

RNG = np.random.default_rng(4321)


def _dir(V, alpha=0.7):
    return RNG.dirichlet(np.full(V, alpha))


CASES = [
    # (V, models of the K branches, M, s)
    (5, [0, 0], 3, 2),
    (5, [0, 0, 0], 2, 5),
    (6, [0, 1], 4, 2),
    (5, [0, 1, 0], 3, 3),
    (5, [0, 0], 1, 5),
    (5, [0, 0, 0], 5, 5),
    (6, [0, 1, 1], 6, 2),
    (4, [0, 0, 0, 0], 2, 2),
]


@pytest.mark.parametrize("V,mids,M,s", CASES)
def test_output_law_is_target(V, mids, M, s):
    for alpha in (0.4, 1.5):
        q = _dir(V, alpha)
        rows = {d: _dir(V, alpha) for d in set(mids)}
        law = truncated.output_law(q, [rows[d] for d in mids], M, s)
        np.testing.assert_allclose(law, q, rtol=0, atol=1e-12)


def test_output_law_with_sparse_rows():
    """A one-hot target, drafts with no mass on Omega_0, and a target with
    zero mass outside Omega_0 (the keep step then always keeps)."""
    V = 5
    onehot = np.zeros(V)
    onehot[3] = 1.0
    p = _dir(V)
    np.testing.assert_allclose(truncated.output_law(onehot, [p, p], 2, 2), onehot, atol=1e-12)
    q = _dir(V)
    off = np.array([0.0, 0.0, 0.5, 0.5, 0.0])
    law = truncated.output_law(q, [off, p], 2, 2)
    np.testing.assert_allclose(law, q, atol=1e-12)
    q3 = np.array([0.5, 0.0, 0.25, 0.25, 0.0])
    np.testing.assert_allclose(truncated.output_law(q3, [p, p, off], 3, 2), q3, atol=1e-12)


def test_omega0_cut_and_ties():
    """At most M tokens, all strictly above the (M+1)-th largest probability;
    tokens tied at the cut are left out together."""
    q = np.array([0.1, 0.3, 0.1, 0.3, 0.2])
    assert truncated.omega0(q, 1).tolist() == []          # 0.3 twice: tied at the cut
    assert truncated.omega0(q, 2).tolist() == [1, 3]
    assert truncated.omega0(q, 3).tolist() == [1, 3, 4]
    assert truncated.omega0(q, 4).tolist() == [1, 3, 4]   # 0.1 twice: tied at the cut
    assert truncated.omega0(q, 5).tolist() == [0, 1, 2, 3, 4]
    assert truncated.omega0(q, 9).tolist() == [0, 1, 2, 3, 4]
    for _ in range(30):
        d = np.round(_dir(12, 0.5), 2)
        M = int(RNG.integers(0, 13))
        om = truncated.omega0(d, M)
        assert len(om) <= M
        inside = np.zeros(12, dtype=bool)
        inside[om] = True
        if inside.any() and (~inside).any():
            assert d[inside].min() > d[~inside].max()
        # the cut is the (M+1)-th largest value: one more token would need a tie break
        if M < 12:
            assert np.sum(d >= np.sort(d)[::-1][M]) >= M + 1


def test_empty_omega0_samples_the_target():
    """All tokens tied: Omega_0 is empty and the output is drawn from q."""
    q = np.full(4, 0.25)
    p = _dir(4)
    np.testing.assert_allclose(truncated.output_law(q, [p, p], 2, 2), q, atol=1e-15)
    rec = DepthRecord(0)
    z = truncated.truncated_step(rec, q, [p, p], [0, 1], 3, 0, 0, 2, 2)
    assert 0 <= z < 4


def _sample_z(q, dists, X, M, s, n, seed):
    """Z from the sampler for n independent depths (sequence ids 0..n-1)."""
    out = np.empty(n, dtype=np.int64)
    for i in range(n):
        rec = DepthRecord(0)
        out[i] = truncated.truncated_step(rec, q, dists, X[i], seed, i, 0, M, s)
    return out


def test_sampler_matches_target_monte_carlo():
    """Empirical law of the sampler's output, draft tuples drawn from the
    draft laws: total variation to q below 4/sqrt(N)."""
    V, M, s, N = 6, 3, 2, 12000
    q = _dir(V, 0.8)
    p1, p2 = _dir(V, 0.8), _dir(V, 0.8)
    dists = [p1, p2, p1]
    X = np.stack([RNG.choice(V, size=N, p=d) for d in dists], axis=1)
    z = _sample_z(q, dists, X, M, s, N, seed=99)
    emp = np.bincount(z, minlength=V) / N
    tv = 0.5 * np.abs(emp - q).sum()
    assert tv < 4.0 / np.sqrt(N), tv


def test_sampler_keep_rate_is_target_mass():
    """The output lands outside Omega_0 with probability 1 - p_a."""
    V, M, N = 8, 2, 6000
    q = _dir(V, 1.5)
    p = _dir(V, 1.5)
    X = RNG.choice(V, size=(N, 2), p=p)
    z = _sample_z(q, [p, p], X, M, 5, N, seed=7)
    om = truncated.omega0(q, M)
    outside = float(np.mean(~np.isin(z, om)))
    pr = 1.0 - q[om].sum()
    assert abs(outside - pr) < 4.0 * np.sqrt(pr * (1 - pr) / N)


def _workload(V, K, L, B, mids, seed):
    rng = np.random.default_rng(seed)
    tl = rng.normal(0.0, 2.0, size=(B, K, L + 1, V))
    tl[:, :, :] = tl[:, :1, :]         # one tree node per depth (equal prefixes share rows)
    drafts = [tl[:, k, :L] + rng.normal(0.0, 0.7, size=(B, L, V)) for k in range(K)]
    for k in range(K):
        drafts[k] = drafts[mids.index(mids[k])]
    tokens = np.zeros((B, K, L), dtype=np.int64)
    for b in range(B):
        for k in range(K):
            for j in range(L):
                lg = drafts[k][b, j]
                pk = np.exp(lg - lg.max())
                tokens[b, k, j] = rng.choice(V, p=pk / pk.sum())
    temps = np.ones((B, 1 + K))
    return tl, drafts, np.array(mids), tokens, temps


def test_full_alphabet_reduces_to_wis():
    """Omega_0 = Omega: p_a = 1 and every input is kept, so the scheme is
    plain WIS with the same draws."""
    V, K, L, B = 7, 3, 3, 40
    w = _workload(V, K, L, B, [0, 0, 1], seed=3)
    a_out, a_acc, _ = oracle_verify(*w, "WIS", seed=5, wis_s=3)
    b_out, b_acc, _ = oracle_verify(*w, "WIS0", seed=5, wis_s=3, omega0=V)
    np.testing.assert_array_equal(a_out, b_out)
    np.testing.assert_array_equal(a_acc, b_acc)


def test_walk_emits_target_tokens():
    """Walk with the truncated scheme on V = 3, K = 2, L = 2: the first emitted
    token follows q exactly in law (Monte Carlo over sequences)."""
    V, K, L, B = 3, 2, 2, 3000
    rng = np.random.default_rng(11)
    row = rng.normal(0.0, 1.0, size=V)
    tl = np.broadcast_to(row, (B, K, L + 1, V)).copy()
    drow = row + rng.normal(0.0, 1.0, size=V)
    drafts = [np.broadcast_to(drow, (B, L, V)).copy() for _ in range(K)]
    pd = np.exp(drow - drow.max())
    pd /= pd.sum()
    tokens = rng.choice(V, size=(B, K, L), p=pd)
    temps = np.ones((B, 1 + K))
    out, acc, _ = oracle_verify(tl, drafts, np.array([0, 0]), tokens, temps, "WIS0", seed=1, wis_s=2, omega0=2)
    q = np.exp(row - row.max())
    q /= q.sum()
    emp = np.bincount(out[:, 0], minlength=V) / B
    assert 0.5 * np.abs(emp - q).sum() < 4.0 / np.sqrt(B)


# ------------------------------------------------------------------- filters


def test_top_k_keeps_the_k_largest_with_lower_id_ties():
    d = np.array([0.25, 0.125, 0.25, 0.25, 0.125])
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=2), [0.5, 0.0, 0.5, 0.0, 0.0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=4),
                                  [0.25 / 0.875, 0.125 / 0.875, 0.25 / 0.875, 0.25 / 0.875, 0.0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=0), d)
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=9), d)


def test_top_p_shortest_prefix_reaching_the_mass():
    d = np.array([0.125, 0.5, 0.25, 0.0625, 0.0625])
    # prefix masses in order 1, 2, 0, 3, 4: 0.5, 0.75, 0.875, 0.9375, 1.0
    np.testing.assert_array_equal(truncated.top_filter(d, top_p=0.5), [0, 1, 0, 0, 0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_p=0.75), [0, 2 / 3, 1 / 3, 0, 0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_p=0.76),
                                  [0.125 / 0.875, 0.5 / 0.875, 0.25 / 0.875, 0, 0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_p=0.9), [0.125 / 0.9375, 0.5 / 0.9375,
                                                                      0.25 / 0.9375, 0.0625 / 0.9375, 0])
    # top-k first, then the nucleus of the renormalised top-k row
    # (top-2 renormalised: 2/3, 1/3)
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=2, top_p=0.6), [0, 1, 0, 0, 0])
    np.testing.assert_array_equal(truncated.top_filter(d, top_k=2, top_p=0.7), [0, 2 / 3, 1 / 3, 0, 0])


def test_top_p_prefix_is_minimal_on_random_rows():
    for _ in range(50):
        V = int(RNG.integers(2, 30))
        d = _dir(V, 0.3)
        tp = float(RNG.uniform(0.05, 0.99))
        f = truncated.top_filter(d, top_p=tp)
        kept = f > 0
        assert d[kept].sum() >= tp - 1e-12
        # dropping the smallest kept token falls short of the mass
        smallest = d[kept].min()
        assert d[kept].sum() - smallest < tp + 1e-12
        # nothing outside is more probable than anything inside
        if (~kept).any():
            assert d[~kept].max() <= smallest


def test_filtered_walk_uses_filtered_rows():
    """With top-k = 1 on every row the target is one-hot at its argmax: every
    emitted token is the target's argmax at its depth."""
    V, K, L, B = 9, 2, 2, 30
    tl, drafts, mids, tokens, temps = _workload(V, K, L, B, [0, 0], seed=8)
    tokens[:] = np.argmax(drafts[0], axis=-1)[:, None, :]    # drawn from the top-1 draft rows
    out, acc, _ = oracle_verify(tl, drafts, mids, tokens, temps, "WIS0", seed=2, wis_s=2, omega0=3, top_k=1)
    for b in range(B):
        for j in range(int(acc[b]) + 1):
            assert out[b, j] == int(np.argmax(tl[b, 0, j]))


def test_draw_ids_are_distinct_from_the_other_steps():
    ids = {philox.DRAW_ACCEPT, philox.DRAW_RESIDUAL, philox.DRAW_BONUS, truncated.DRAW_KEEP,
           truncated.DRAW_OUTSIDE}
    assert len(ids) == 5 and min(truncated.DRAW_KEEP, truncated.DRAW_OUTSIDE) > philox.DRAW_BONUS
