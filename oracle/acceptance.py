"""Oracle: acceptance probability of each scheme on one row (analytic).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).  Plain fp64 numpy.

For a target law q and the valid branches' draft laws, the probability that
a depth accepts one of the draft tokens:

single, IS, WIS,  Theorem 1: sum_k min(q_k, p_I(k)) with p_I the law of the
WISsort           intermediate token (the draft law itself; the Laplace
                  identity of ``is_laplace``; the pairwise stage chain of
                  ``wis``, or of ``sorted_lp`` for the sorted rule).
SpecTr            the sequential-rejection reading: 1 - prod_i R_i, R_i the
                  residual mass left after round i.
WIS0              the truncated alphabet (Section 4): p_a = q(Omega_0) times
                  the expectation, over which branches land in Omega_0, of
                  the inner WIS acceptance sum_{Omega_0} min(q~, p_I) of the
                  kept inputs (their draft laws truncated to Omega_0).
optimal           Theorem 3 for K = 2 i.i.d. drafts and Remark 2's
                  conjectured form for K > 2 (``theory.pstar_sorted``), the
                  ceiling of any token-level selection rule.

Running the module prints these for depth 0 of a few sequences of every
named synthetic workload (the counterpart of the paper's Table 2 on the
stand-in rows):  python -m oracle.acceptance [--top-p=0.95] [--top-k=5] [workload ...]
"""
import itertools

import numpy as np

from . import enum, is_laplace, sorted_lp, theory, truncated


def scheme_acceptance(q, dists, mids, scheme, s=5, is_h=0.25):
    """Acceptance probability of ``scheme`` for target q and the valid
    branches' draft laws ``dists`` (model ids ``mids``)."""
    q = np.asarray(q, dtype=np.float64)
    if scheme == "single" or len(dists) == 1:
        return float(np.minimum(q, dists[0]).sum())
    if scheme == "WIS":
        pI = enum.wis_stages(q, dists, s)[-1].pI
        return float(np.minimum(q, pI).sum())
    if scheme == "WISsort":
        pI = np.asarray(dists[0], dtype=np.float64)
        for d in dists[1:]:
            pI = sorted_lp.stage(q, pI, d, s).pI
        return float(np.minimum(q, pI).sum())
    if scheme == "IS":
        rows, counts = {}, {}
        for d, m in zip(dists, mids):
            rows[m] = d
            counts[m] = counts.get(m, 0) + 1
        return float(np.minimum(q, is_laplace.is_law(q, rows, counts, is_h)).sum())
    if scheme == "SpecTr":
        qi, reject = q.copy(), 1.0
        for p in dists:
            r = np.maximum(0.0, qi - p)
            R = float(r.sum())
            reject *= R
            if R > 0:
                qi = r / R
        return 1.0 - reject
    raise ValueError(scheme)


def truncated_acceptance(q, dists, M, s=5):
    """Probability that a truncated-alphabet depth outputs an accepted draft
    token (kept by the p_a test), for target q and the valid branches' draft
    laws ``dists`` in branch order."""
    q = np.asarray(q, dtype=np.float64)
    om = truncated.omega0(q, M)
    if len(om) == 0:
        return 0.0
    pa = float(q[om].sum())
    qt = q[om] / pa
    inside = [float(np.asarray(d, dtype=np.float64)[om].sum()) for d in dists]
    laws = [truncated.truncate(d, om) for d in dists]
    total = 0.0
    for pattern in itertools.product((0, 1), repeat=len(dists)):
        pr = 1.0
        for hit, pin in zip(pattern, inside):
            pr *= pin if hit else 1.0 - pin
        kept = [i for i, hit in enumerate(pattern) if hit and laws[i] is not None]
        if pr == 0.0 or not kept:
            continue
        if len(kept) == 1:
            pI = laws[kept[0]]
        else:
            pI = enum.wis_stages(qt, [laws[i] for i in kept], s)[-1].pI
        total += pr * float(np.minimum(qt, pI).sum())
    return pa * total


def optimal_acceptance(q, p, K):
    """Theorem 3 (K = 2) / Remark 2's conjecture (K > 2) for i.i.d. drafts."""
    return theory.pstar_sorted(p, q, K)


def _softmax(x, t):
    z = np.asarray(x, dtype=np.float64) / t
    e = np.exp(z - z.max())
    return e / e.sum()


def table(names=None, seqs=(0, 1, 2, 3), top_p=1.0, top_k=0):
    """Rows of (workload, sequence, K, single, IS, WIS, WISsort, WIS0,
    SpecTr, optimal) at depth 0, every row top-k / top-p filtered first when
    set (Section 5); IS is skipped above 60000 tokens (its quadrature costs
    V x T)."""
    from synth import WORKLOADS, make_workload
    out = []
    for name in names or list(WORKLOADS):
        spec = WORKLOADS[name].with_(B=max(seqs) + 1)
        w = make_workload(spec, device="cpu")
        for b in seqs:
            temps = w.temps[b].double().numpy()
            q = _softmax(w.target[b, 0, 0].float().numpy(), temps[0])
            dists = [_softmax(w.drafts[k, b, 0].float().numpy(), temps[1 + k]) for k in range(spec.K)]
            if top_p < 1.0 or top_k > 0:
                q = truncated.top_filter(q, top_k=top_k, top_p=top_p)
                dists = [truncated.top_filter(d, top_k=top_k, top_p=top_p) for d in dists]
            mids = list(spec.model_ids)
            row = {"workload": name, "b": b, "K": spec.K}
            for sch in ("single", "IS", "WIS", "WISsort", "SpecTr"):
                if sch == "IS" and spec.V > 60000:
                    row[sch] = None
                    continue
                row[sch] = scheme_acceptance(q, dists, mids, sch)
            row["WIS0"] = truncated_acceptance(q, dists, 20)
            iid = len(set(mids)) == 1
            row["optimal"] = optimal_acceptance(q, dists[0], spec.K) if iid else None
            out.append(row)
    return out


if __name__ == "__main__":
    import sys
    args = sys.argv[1:]
    tp, tk = 1.0, 0
    while args and args[0].startswith("--"):
        opt, val = args.pop(0).split("=", 1)
        if opt == "--top-p":
            tp = float(val)
        elif opt == "--top-k":
            tk = int(val)
        else:
            raise SystemExit(f"unknown option {opt}")
    rows = table(args or None, top_p=tp, top_k=tk)
    print("| workload | b | K | single | IS | WIS (s = 5) | WISsort (s = 5) | WIS0 (M = 20) | SpecTr reading | "
          "optimal (Thm 3 / Remark 2) |")
    print("|---|---|---|---|---|---|---|---|---|---|")
    f = lambda v: "—" if v is None else f"{v:.4f}"   # noqa: E731
    for r in rows:
        print(f"| {r['workload']} | {r['b']} | {r['K']} | {f(r['single'])} | {f(r['IS'])} | {f(r['WIS'])} | "
              f"{f(r['WISsort'])} | {f(r['WIS0'])} | {f(r['SpecTr'])} | {f(r['optimal'])} |")
