"""CUDA path vs the oracle with top-k restriction of every row (Section 5's
top-k runs, Tables 2 and 3: k = 5 and 10).

The oracle restricts each softmax row to its k most probable tokens (ties to
the lower id) and renormalises (oracle/truncated.py:top_filter) before the
scheme runs; the top-k kernel selects each visited row's top k and runs the
scheme on the union of the kept tokens.  Cases: k from 1 to the largest, f32
and bf16 rows, rows fetched by 16-byte units and by element loads (ragged V),
one and two draft models, the variant (WIS) and the sorted rule (WISsort) on
Omega_2, s = 8 (the shared-memory LP), V below k and below s (zero-key tokens
outside the union fill Omega_1), draft tokens drawn
without the restriction (p_I(Y) = 0), acc_prob, the allocation-free entry
point, and sampled sequences of the full-size workload.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from oracle.verify import oracle_verify  # noqa: E402
from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, host_copy, make_workload  # noqa: E402
from parity import check, compare  # noqa: E402

DEV = "cuda:0"


def run_topk(spec, scheme, seed, top_k, wis_s=5, acc_prob=0, seqs=None):
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, wis_s=wis_s, acc_prob=acc_prob, top_k=top_k)
    out, acc, diag = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, seed, diag=True)
    torch.cuda.synchronize()
    bits, _ = v.status()
    v.close()
    if seqs is None:
        o_out, o_acc, recs = oracle_verify(*host_copy(w), scheme, seed, wis_s=wis_s, top_k=top_k)
    else:
        # keyed by the global sequence ids, as the GPU arrays are indexed
        o_out, o_acc, recs = oracle_verify(*host_copy(w, seqs), scheme, seed, wis_s=wis_s, seq_ids=seqs,
                                           top_k=top_k)
    res = compare(out.cpu().numpy(), acc.cpu().numpy(), o_out, o_acc, recs, g_diag=diag.cpu().numpy(),
                  scheme=scheme)
    res["status"] = bits
    res["diag"] = diag.cpu().numpy()
    res["recs"] = recs
    res["acc"] = acc.cpu().numpy()
    return res


def ok(res, scheme):
    check(res, scheme)
    assert res["status"] == 0, res["status"]


CASES = [
    ("tiny", dict(B=8)),                                      # f32, 16-byte units
    ("llama2-32k", dict(B=12, V=5003)),                       # bf16, ragged: element loads
    ("two-models-50k", dict(B=16, V=7001)),                   # two draft models
    ("llama3-128k", dict(B=8, V=9000)),                       # K = 8, bf16 units
    ("serving-152k", dict(B=12, V=6007, L=5)),                # per-sequence temperatures
]


@pytest.mark.parametrize("name,kw", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("top_k", [5, 10])
def test_paper_top_k_matches_oracle(name, kw, top_k):
    spec = WORKLOADS[name].with_(top_k=top_k, **kw)
    for scheme in ("WIS", "WISsort", "single", "SpecTr"):
        ok(run_topk(spec, scheme, seed=7 + top_k, top_k=top_k), scheme)


@pytest.mark.parametrize("top_k", [1, 2, 16])
def test_extreme_k(top_k):
    spec = WORKLOADS["llama2-32k"].with_(B=10, V=4099, K=3, model_ids=[0, 0, 0], top_k=top_k)
    for scheme in ("WIS", "WISsort", "single", "SpecTr"):
        ok(run_topk(spec, scheme, seed=3, top_k=top_k), scheme)


def test_largest_s_uses_the_shared_memory_lp():
    spec = WORKLOADS["llama3-128k"].with_(B=8, V=6000, top_k=10)
    for scheme in ("WIS", "WISsort"):
        ok(run_topk(spec, scheme, seed=5, top_k=10, wis_s=8), scheme)
        ok(run_topk(spec, scheme, seed=6, top_k=10, wis_s=1), scheme)


def test_vocabulary_smaller_than_k_and_s():
    # V = 3: every row keeps the whole vocabulary; s = min(5, V)
    spec = WORKLOADS["tiny"].with_(B=16, V=3, K=4, model_ids=[0, 1, 0, 1], draft_sigma=[0.7, 1.5],
                                   t_draft=[1.0, 0.8], top_k=5)
    for scheme in ("WIS", "WISsort", "single", "SpecTr"):
        ok(run_topk(spec, scheme, seed=2, top_k=5), scheme)


def test_draft_tokens_outside_the_restriction():
    # tokens drawn from the unrestricted draft rows: p_I(Y) = 0 accepts Y
    spec = WORKLOADS["llama2-32k"].with_(B=12, V=3001)
    for scheme in ("WIS", "WISsort", "single", "SpecTr"):
        ok(run_topk(spec, scheme, seed=9, top_k=5), scheme)


def test_acceptance_probability_reported():
    spec = WORKLOADS["two-models-50k"].with_(B=12, V=5000, top_k=5)
    for scheme in ("WIS", "single", "SpecTr"):
        res = run_topk(spec, scheme, seed=4, top_k=5, acc_prob=1)
        ok(res, scheme)
        diag, recs, acc = res["diag"], res["recs"], res["acc"]
        for b, rr in recs.items():
            for r in rr[: int(acc[b]) + 1]:
                if r.j >= diag.shape[1] - 1 or r.band or np.isnan(r.R) or scheme == "SpecTr":
                    continue
                assert abs(float(diag[b, r.j, 2]) - r.R) <= 1e-5 + 1e-4 * r.R, (b, r.j, diag[b, r.j], r.R)


def test_sampled_sequences_of_full_size_workload():
    spec = WORKLOADS["llama3-128k"].with_(top_k=10)
    seqs = [0, 1, 37, 101, 128, 200, 254, 255]
    ok(run_topk(spec, "WIS", seed=1, top_k=10, seqs=seqs), "WIS")


def test_unserved_schemes_refused():
    spec = WORKLOADS["tiny"].with_(B=4, V=1000, top_k=5)
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, top_k=5)
    for scheme in ("IS", "WIS0"):
        with pytest.raises(mds.MdsError) as e:
            v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, 1)
        assert e.value.code == mds.MDS_EUNSUP
    torch.cuda.synchronize()
    v.close()
    # the sorted rule is served on restricted rows only
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype)
    with pytest.raises(mds.MdsError) as e:
        v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WISsort", 1)
    assert e.value.code == mds.MDS_EUNSUP
    torch.cuda.synchronize()
    v.close()


def test_allocation_free_entry_point_agrees():
    spec = WORKLOADS["two-models-50k"].with_(B=8, V=4096, top_k=10)
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, top_k=10)
    out, acc, _ = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WIS", 5)
    torch.cuda.synchronize()
    v.close()
    o2 = torch.empty_like(out)
    a2 = torch.empty_like(acc)
    mds.mds_verify_noalloc(spec.B, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, w.tokens, w.temps,
                           "WIS", 5, o2, a2, dtype=spec.dtype, top_k=10)
    torch.cuda.synchronize()
    assert torch.equal(out, o2) and torch.equal(acc, a2)
    assert mds.mds_noalloc_status(0) == (0, "ok")
