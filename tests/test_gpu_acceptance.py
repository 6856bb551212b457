"""CUDA path vs the oracle for the per-depth acceptance probability
(acc_prob = 1): out_diag[b][j][2] must hold R = sum max(0, q - p_I) at every
visited depth below L, accepted or not, within the tolerance of a
vocabulary-long fp32 sum; the emitted tokens must not change.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, make_workload, host_copy  # noqa: E402
from oracle.verify import oracle_verify  # noqa: E402

DEV = "cuda:0"
R_ATOL = {"single": 2e-5, "WIS": 2e-5, "IS": 1e-4}   # IS: p_I from a ~300-node fp32 quadrature


def run(spec, scheme, seed, acc_prob, cluster=0, seqs=None):
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, cluster=cluster, acc_prob=acc_prob)
    out, acc, diag = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, seed, diag=True)
    torch.cuda.synchronize()
    assert v.status()[0] == 0
    v.close()
    return w, out.cpu().numpy(), acc.cpu().numpy(), diag.cpu().numpy()


@pytest.mark.parametrize("name,kw,scheme", [
    ("tiny", dict(), "IS"),
    ("tiny", dict(), "single"),
    ("llama2-32k", dict(B=10, V=5003), "WIS"),
    ("two-models-50k", dict(B=10, V=7001), "WIS"),
    ("llama3-128k", dict(B=8, V=9000), "WIS"),
    ("serving-152k", dict(B=8, V=6007, L=5), "IS"),
], ids=lambda x: x if isinstance(x, str) else "")
def test_residual_mass_at_every_depth(name, kw, scheme):
    spec = WORKLOADS[name].with_(**kw)
    w, out, acc, diag = run(spec, scheme, 7, acc_prob=1)
    _, out0, acc0, _ = run(spec, scheme, 7, acc_prob=0)
    np.testing.assert_array_equal(out, out0)
    np.testing.assert_array_equal(acc, acc0)
    o_out, o_acc, recs = oracle_verify(*host_copy(w), scheme, 7)
    checked = 0
    for b in range(spec.B):
        for r in recs[b]:
            if r.j >= spec.L or r.band:
                break
            if not np.array_equal(out[b, :r.j + 1], o_out[b][:r.j + 1]):
                break
            assert abs(diag[b, r.j, 2] - r.R) <= R_ATOL[scheme], (b, r.j, diag[b, r.j, 2], r.R)
            checked += 1
    assert checked >= spec.B // 2


@pytest.mark.parametrize("cluster", [2, 8])
def test_clusters(cluster):
    spec = WORKLOADS["llama2-32k"].with_(B=6, V=4099)
    w, out, acc, diag = run(spec, "WIS", 3, acc_prob=1, cluster=cluster)
    o_out, o_acc, recs = oracle_verify(*host_copy(w), "WIS", 3)
    for b in range(spec.B):
        for r in recs[b]:
            if r.j >= spec.L or r.band or not np.array_equal(out[b, :r.j + 1], o_out[b][:r.j + 1]):
                break
            assert abs(diag[b, r.j, 2] - r.R) <= R_ATOL["WIS"]


def test_full_size_sampled():
    spec = WORKLOADS["llama3-128k"]
    seqs = [0, 1, 100, 255]
    w, out, acc, diag = run(spec, "WIS", spec.verify_seed, acc_prob=1)
    o_out, o_acc, recs = oracle_verify(*host_copy(w, seqs), "WIS", spec.verify_seed, seq_ids=seqs)
    for b in seqs:
        assert np.array_equal(out[b], o_out[b])
        for r in recs[b]:
            if r.j >= spec.L or r.band:
                break
            assert abs(diag[b, r.j, 2] - r.R) <= R_ATOL["WIS"]



@pytest.mark.parametrize("name,kw,cluster", [
    ("two-models-50k", dict(B=8, V=7001), 0),
    ("llama2-32k", dict(B=8, V=5003), 0),
    ("serving-152k", dict(B=6, V=6007, L=4), 2),
], ids=lambda x: x if isinstance(x, str) else "")
def test_spectr_rejection_probability(name, kw, cluster):
    # The sequential-rejection reading: out_diag[b][j][2] = prod_i R_i, the
    # probability that every round rejects, at every visited depth below L
    # (the rounds after an acceptance computed too), against the oracle's
    # analytic 1 - acceptance on the same rows; tokens unchanged.
    from oracle.acceptance import scheme_acceptance
    from oracle.verify import softmax_t
    spec = WORKLOADS[name].with_(**kw)
    w, out, acc, diag = run(spec, "SpecTr", 5, acc_prob=1, cluster=cluster)
    _, out0, acc0, _ = run(spec, "SpecTr", 5, acc_prob=0, cluster=cluster)
    np.testing.assert_array_equal(out, out0)
    np.testing.assert_array_equal(acc, acc0)
    target, drafts, mids, tokens, temps = host_copy(w)
    checked = 0
    for b in range(spec.B):
        valid = list(range(spec.K))
        for j in range(min(int(acc[b]) + 1, spec.L)):
            k0 = valid[0]
            q = softmax_t(target[b, k0, j], temps[b, 0])
            dists = [softmax_t(drafts[k][b, j], temps[b, 1 + k]) for k in valid]
            R = 1.0 - scheme_acceptance(q, dists, [mids[k] for k in valid], "SpecTr")
            assert abs(diag[b, j, 2] - R) <= 2e-5 * len(valid), (b, j, float(diag[b, j, 2]), R)
            checked += 1
            valid = [k for k in valid if tokens[b, k, j] == out[b, j]]
            if not valid:
                break
    assert checked >= spec.B
