"""Comparison of the CUDA path with the oracle (shared by the GPU tests).

Outputs must be identical for every sequence, except that a sequence may
diverge from the first depth whose oracle record carries the band flag (a
discrete decision within rounding of its boundary).  Such sequences are
counted and returned.  Where both sides chose the same intermediate token the
probabilities q(Y) and p_I(Y) must agree within the stated relative tolerance.
"""
import numpy as np

PROB_RTOL = 1e-5        # softmax probabilities, fp32 kernel vs fp64 oracle
PROB_RTOL_IS = 2e-5     # p_I of plain IS adds a ~300-node quadrature sum in fp32
PI_ATOL = 1e-6          # p_I of WIS: the stage LP moves unit-scale masses in fp32 over <= 28
                        # pairs, so its absolute rounding is ~28 * 2^-24 ~ 1.7e-6 at worst


def compare(g_out, g_acc, o_out, o_acc, recs, seqs=None, g_diag=None, scheme=None, strict_prob=True):
    """Returns dict(n, band, mismatches, max_rel_q, max_rel_pI)."""
    g_out = np.asarray(g_out)
    g_acc = np.asarray(g_acc)
    seqs = list(recs.keys()) if seqs is None else list(seqs)
    band = 0
    bad = []
    max_q = 0.0
    max_p = 0.0
    worst = None
    for b in seqs:
        o_out_b, o_acc_b = np.asarray(o_out[b]), int(o_acc[b])
        same = np.array_equal(g_out[b], o_out_b) and int(g_acc[b]) == o_acc_b
        rr = recs[b]
        if not same:
            # first differing position
            diff = np.flatnonzero(g_out[b] != o_out_b)
            j = int(diff[0]) if len(diff) else min(int(g_acc[b]), o_acc_b)
            if any(r.band for r in rr[: j + 1]):
                band += 1
            else:
                bad.append((b, j, g_out[b].tolist(), int(g_acc[b]), o_out_b.tolist(), o_acc_b))
            limit = j
        else:
            limit = len(rr)
        if g_diag is not None:
            for r in rr[:limit]:
                # a band depth may legitimately take a different LP structure
                if r.Y < 0 or int(g_diag[b, r.j, 3]) != r.Y or r.band:
                    continue
                qg, pg = float(g_diag[b, r.j, 0]), float(g_diag[b, r.j, 1])
                if r.qY > 1e-30:
                    max_q = max(max_q, abs(qg - r.qY) / r.qY)
                if r.pIY > 1e-30:
                    rel = max(0.0, abs(pg - r.pIY) - PI_ATOL) / r.pIY
                    if rel > max_p:
                        max_p = rel
                        worst = (b, r.j, r.Y, pg, r.pIY, {k: float(v) for k, v in r.margins.items()})
    return dict(n=len(seqs), band=band, mismatches=bad, max_rel_q=max_q, max_rel_pI=max_p, worst_pI=worst)


def check(res, scheme, max_band_frac=0.05):
    assert not res["mismatches"], f"{scheme}: {len(res['mismatches'])} mismatches outside the band, " \
                                  f"first: {res['mismatches'][:2]}"
    tol = PROB_RTOL_IS if scheme == "IS" else PROB_RTOL
    assert res["max_rel_q"] <= PROB_RTOL, f"{scheme}: q(Y) rel err {res['max_rel_q']}"
    assert res["max_rel_pI"] <= tol, f"{scheme}: p_I(Y) rel err {res['max_rel_pI']} at {res['worst_pI']}"
    assert res["band"] <= max(1, max_band_frac * res["n"]), f"{scheme}: {res['band']} band sequences"
