"""Pins for the oracle's sampling path and tree walk (oracle.verify).

The enumeration tests pin the selection laws; these tests pin the code that
actually draws: the inverse CDF, the accept test, the walk along the tree
and the bonus token, by Monte Carlo over many sequences (every sequence has
its own Philox draws) against the exact target laws of a three-letter,
two-level draft tree.
"""
import numpy as np
import pytest

from oracle import verify
from oracle.verify import inverse_cdf, oracle_verify

RNG = np.random.default_rng(77)


def test_inverse_cdf_brute_force():
    for _ in range(50):
        n = int(RNG.integers(1, 9))
        r = RNG.random(n) * (RNG.random(n) < 0.7)
        if r.sum() == 0:
            r[0] = 1.0
        for k24 in (0, 1, 1 << 22, (1 << 23) + 5, (1 << 24) - 1):
            u = k24 * 2.0 ** -24
            z, _ = inverse_cdf(r, u)
            t = u * r.sum()
            # brute force: first index whose running sum exceeds t
            run = 0.0
            want = None
            for k in range(n):
                run += r[k]
                if run > t:
                    want = k
                    break
            assert z == want
            assert r[z] > 0


def _tree_inputs(N, V, K, L, rng, mids=None, temps=(1.0, 1.0)):
    """Inputs for a draft tree whose rows depend only on the node (token
    prefix): tables T[prefix] and D[model][prefix] of logits."""
    mids = mids or [0] * K
    tables_t = {}
    tables_d = {}

    def row_t(prefix):
        if prefix not in tables_t:
            tables_t[prefix] = rng.normal(0, 1.5, V)
        return tables_t[prefix]

    def row_d(m, prefix):
        if (m, prefix) not in tables_d:
            tables_d[(m, prefix)] = row_t(prefix) + rng.normal(0, 1.0, V)
        return tables_d[(m, prefix)]

    target = np.zeros((N, K, L + 1, V))
    drafts = [np.zeros((N, L, V)) for _ in range(K)]
    tokens = np.zeros((N, K, L), dtype=np.int64)
    tq, td = temps
    for b in range(N):
        for k in range(K):
            prefix = ()
            for j in range(L + 1):
                target[b, k, j] = row_t(prefix)
                if j == L:
                    break
                d = row_d(mids[k], prefix)
                drafts[k][b, j] = d
                p = np.exp((d - d.max()) / td)
                p /= p.sum()
                x = int(rng.choice(V, p=p))
                tokens[b, k, j] = x
                prefix = prefix + (x,)
    temps_arr = np.zeros((N, 1 + K))
    temps_arr[:, 0] = tq
    temps_arr[:, 1:] = td
    return target, drafts, mids, tokens, temps_arr, row_t


def _tv(counts, q):
    n = counts.sum()
    return 0.5 * np.abs(counts / n - q).sum(), n


@pytest.mark.parametrize("scheme,N", [("single", 12000), ("WIS", 12000), ("SpecTr", 12000), ("IS", 2500),
                                      ("WIS0", 12000), ("WISsort", 12000)])
def test_walk_emits_target_model_samples(scheme, N):
    """Z_0 ~ q(root); given a continued walk through z, Z_1 ~ q(z); after two
    accepted positions the bonus ~ q(z0, z1).  TV below 4/sqrt(n) per law."""
    V, K, L = 3, 2, 2
    rng = np.random.default_rng(5 + len(scheme))
    target, drafts, mids, tokens, temps, row_t = _tree_inputs(N, V, K, L, rng)
    # WIS0 with |Omega_0| = 2 < V: a two-token inner stage and the keep / replace step at every depth
    out, acc, _ = oracle_verify(target, drafts, mids, tokens, temps, scheme, seed=99, wis_s=2, omega0=2)

    def q_of(prefix):
        x = row_t(prefix)
        e = np.exp(x - x.max())
        return e / e.sum()

    assert np.all((acc >= 0) & (acc <= L))
    for b in range(N):
        assert np.all(out[b, acc[b] + 1:] == -1) and np.all(out[b, :acc[b] + 1] >= 0)
    c0 = np.bincount(out[:, 0], minlength=V)
    tv, n = _tv(c0, q_of(()))
    assert tv < 4 / np.sqrt(n)
    for z in range(V):
        sel = (out[:, 0] == z) & (acc >= 1)
        if sel.sum() > 400:
            tv, n = _tv(np.bincount(out[sel, 1], minlength=V), q_of((z,)))
            assert tv < 4 / np.sqrt(n)
        for z1 in range(V):
            sel2 = sel & (out[:, 1] == z1) & (acc == 2)
            if sel2.sum() > 400:
                tv, n = _tv(np.bincount(out[sel2, 2], minlength=V), q_of((z, z1)))
                assert tv < 4 / np.sqrt(n)


def test_accept_rate_matches_analytic_single():
    """Algorithm 1: Pr(accept the draft) = sum min(p, q); with the walk rule a
    rejected draft can still land in S, so Pr(acc_len >= 1) >= that value."""
    N, V = 20000, 4
    rng = np.random.default_rng(3)
    target, drafts, mids, tokens, temps, row_t = _tree_inputs(N, V, 1, 1, rng)
    _, acc, recs = oracle_verify(target, drafts, mids, tokens, temps, "single", seed=5)
    x = row_t(())
    q = np.exp(x - x.max())
    q /= q.sum()
    d = drafts[0][0, 0]
    p = np.exp(d - d.max())
    p /= p.sum()
    rate = np.mean([recs[b][0].accepted for b in range(N)])
    want = np.minimum(p, q).sum()
    assert abs(rate - want) < 4 * np.sqrt(want * (1 - want) / N)
    assert np.mean(acc >= 1) == pytest.approx(rate, abs=1e-12)   # K = 1: S = {X}


def test_degenerate_vocab_of_one():
    N, V, K, L = 3, 1, 3, 2
    target = np.zeros((N, K, L + 1, V))
    drafts = [np.zeros((N, L, V)) for _ in range(K)]
    tokens = np.zeros((N, K, L), dtype=np.int64)
    temps = np.ones((N, 1 + K))
    for scheme in ("single", "IS", "WIS", "SpecTr"):
        out, acc, _ = oracle_verify(target, drafts, [0] * K, tokens, temps, scheme, seed=1)
        assert np.all(acc == L) and np.all(out == 0)


def test_identical_target_and_draft_always_accepts():
    N, V, K, L = 50, 16, 2, 3
    rng = np.random.default_rng(11)
    target = rng.normal(0, 2, (N, K, L + 1, V))
    target[:, 1] = target[:, 0]
    drafts = [target[:, 0, :L].copy(), target[:, 0, :L].copy()]
    tokens = rng.integers(0, V, (N, K, L))
    tokens[:, 1] = tokens[:, 0]
    temps = np.ones((N, 1 + K))
    # single draft and sequential rejection accept every draft when p = q (the
    # truncated WIS does not: it moves mass from Omega_2 to Omega_1)
    for scheme in ("single", "SpecTr"):
        out, acc, recs = oracle_verify(target, drafts, [0, 0], tokens, temps, scheme, seed=4)
        assert np.all(acc == L), scheme
        assert np.array_equal(out[:, :L], tokens[:, 0])


def test_band_flag_set_on_near_ties():
    rec = verify.DepthRecord(0)
    rec.note("accept", 5e-7, verify.BAND_ACCEPT)
    assert rec.band
    rec2 = verify.DepthRecord(0)
    rec2.note("accept", 5e-6, verify.BAND_ACCEPT)
    assert not rec2.band
