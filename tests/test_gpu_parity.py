"""CUDA path vs the oracle, through the C ABI.

Small cases span several tiles and a ragged tail (oracle finishes in
seconds); full-size workloads run in the launch configuration the bench
uses and are compared on sampled sequences.  Edge cases: vocabularies of
1..9 tokens, K = 1, L = 1, duplicated draft tokens, one-hot targets,
non-unit temperatures, rows whose byte length is not a multiple of 16 (plain
loads instead of bulk copies), every cluster size.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, WorkloadSpec, make_workload, host_copy  # noqa: E402
from oracle.verify import oracle_verify  # noqa: E402
from parity import compare, check  # noqa: E402

DEV = "cuda:0"


def run_both(spec, scheme, seed, cluster=0, seqs=None, wis_s=5, omega0=20):
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, wis_s=wis_s, cluster=cluster, omega0=omega0)
    out, acc, diag = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, seed, diag=True)
    torch.cuda.synchronize()
    bits, msg = v.status()
    cn = v.cluster_size
    v.close()
    if seqs is None:
        o_out, o_acc, recs = oracle_verify(*host_copy(w), scheme, seed, wis_s=wis_s, omega0=omega0)
    else:
        o_out, o_acc, recs = oracle_verify(*host_copy(w, seqs), scheme, seed, wis_s=wis_s, seq_ids=seqs,
                                           omega0=omega0)
    res = compare(out.cpu().numpy(), acc.cpu().numpy(), o_out, o_acc, recs, g_diag=diag.cpu().numpy(),
                  scheme=scheme)
    res["status"] = bits
    res["cn"] = cn
    return res


def small(name, **kw):
    return WORKLOADS[name].with_(**kw)


SMALL_CASES = [
    ("tiny", dict(), ["IS", "single", "WIS", "SpecTr"]),
    ("llama2-32k", dict(B=12, V=5003), ["IS", "WIS", "single", "SpecTr"]),
    ("two-models-50k", dict(B=16, V=7001), ["WIS", "SpecTr", "single", "IS"]),
    ("llama3-128k", dict(B=12, V=9000), ["WIS", "single", "SpecTr"]),
    ("serving-152k", dict(B=12, V=6007, L=5), ["single", "IS", "WIS", "SpecTr"]),
]


@pytest.mark.parametrize("name,kw,schemes", SMALL_CASES, ids=[c[0] for c in SMALL_CASES])
def test_small_workloads_match_oracle(name, kw, schemes):
    spec = small(name, **kw)
    for scheme in schemes:
        res = run_both(spec, scheme, seed=11)
        check(res, scheme)
        assert res["status"] == 0


@pytest.mark.parametrize("cluster", [1, 2, 4, 8, 16])
def test_every_cluster_size(cluster):
    spec = small("llama2-32k", B=6, V=4099, K=3, model_ids=[0, 0, 0])
    for scheme in ("WIS", "single", "SpecTr"):
        res = run_both(spec, scheme, seed=5, cluster=cluster)
        assert res["cn"] == cluster
        check(res, scheme)


@pytest.mark.parametrize("V", [1, 2, 3, 5, 7, 8, 9, 17, 100])
def test_tiny_vocabularies(V):
    for dtype in ("f32", "bf16"):
        spec = WorkloadSpec(f"v{V}", B=24, K=3, L=3, V=V, dtype=dtype, model_ids=[0, 0, 1], target_scale=2.0,
                            draft_sigma=[0.5, 1.0], t_target=1.0, t_draft=[1.0, 1.3], data_seed=V)
        for scheme in ("single", "IS", "WIS", "SpecTr"):
            res = run_both(spec, scheme, seed=V + 1, wis_s=min(5, max(1, V)))
            check(res, scheme)


def test_k1_l1_and_s_values():
    spec = WorkloadSpec("k1", B=16, K=1, L=1, V=3001, dtype="bf16", model_ids=[0], target_scale=3.0,
                        draft_sigma=[1.0], t_target=0.8, t_draft=[1.1], data_seed=9)
    for scheme in ("single", "IS", "WIS", "SpecTr"):
        check(run_both(spec, scheme, seed=2), scheme)
    spec = small("llama3-128k", B=8, V=3000)
    for s in (1, 2, 3, 8):
        check(run_both(spec, "WIS", seed=4, wis_s=s), "WIS")


def test_duplicated_tokens_and_peaked_target():
    # very peaked distributions make most draft tokens coincide
    spec = WorkloadSpec("peaked", B=16, K=6, L=4, V=2048, dtype="bf16", model_ids=[0] * 6, target_scale=12.0,
                        draft_sigma=[0.2], t_target=0.5, t_draft=[0.5], data_seed=3)
    for scheme in ("WIS", "IS", "SpecTr", "single"):
        check(run_both(spec, scheme, seed=8), scheme)


def test_ragged_rows_without_bulk_copies():
    # V * 2 bytes is not a multiple of 16: every row is fetched with plain loads
    spec = small("two-models-50k", B=8, V=4097)
    for scheme in ("WIS", "SpecTr"):
        check(run_both(spec, scheme, seed=6), scheme)
    spec = small("tiny", V=1001)        # f32, 4004-byte rows
    for scheme in ("IS", "WIS"):
        check(run_both(spec, scheme, seed=6), scheme)


def test_mixed_models_and_temperatures():
    spec = WorkloadSpec("mixed", B=16, K=4, L=4, V=3000, dtype="bf16", model_ids=[0, 1, 0, 2], target_scale=4.0,
                        draft_sigma=[0.5, 1.5, 1.0], t_target=0.9, t_draft=[1.0, 2.0, 0.7], data_seed=17)
    for scheme in ("WIS", "IS", "SpecTr", "single"):
        check(run_both(spec, scheme, seed=13), scheme)


def test_more_draft_models_than_a_candidate_list_holds():
    # five distinct draft models: six rows per depth, more than the candidate
    # list carries, so every WIS stage is a full-vocabulary pass; also the
    # stage LP with s = 8 (pair state outside the five-token fast path)
    spec = WorkloadSpec("five", B=12, K=5, L=3, V=3000, dtype="bf16", model_ids=[0, 1, 2, 3, 4], target_scale=3.0,
                        draft_sigma=[0.4, 0.8, 1.2, 1.6, 2.0], t_target=1.0, t_draft=[1.0, 1.3, 0.8, 1.1, 0.9],
                        data_seed=29)
    for wis_s in (5, 8):
        check(run_both(spec, "WIS", seed=21, wis_s=wis_s), "WIS")
    check(run_both(spec, "single", seed=21), "single")


def test_small_slices_and_flat_rows():
    # small batches cut each row into many small slices (threads without a
    # unit), and nearly flat target rows put many tokens at the top: the
    # candidate threshold and its overflow path
    spec = WorkloadSpec("flat", B=4, K=4, L=3, V=1283, dtype="bf16", model_ids=[0] * 4, target_scale=0.02,
                        draft_sigma=[0.01], t_target=1.0, t_draft=[1.0], data_seed=31)
    for scheme in ("WIS", "single"):
        check(run_both(spec, scheme, seed=2), scheme)
    spec = WorkloadSpec("ramp", B=3, K=3, L=2, V=4096, dtype="f32", model_ids=[0] * 3, target_scale=0.0,
                        draft_sigma=[0.5], t_target=1.0, t_draft=[1.0], data_seed=33)
    for scheme in ("WIS", "single"):
        check(run_both(spec, scheme, seed=4), scheme)


def spread(B, n):
    """n sequence ids spread over the batch (the first, the last and evenly between)."""
    return sorted(set(np.linspace(0, B - 1, min(n, B)).round().astype(int).tolist()))


# every workload at full size, in the bench's launch configuration, on
# sampled sequences: 32 per scheme (8 for plain IS, whose oracle integrates
# a ~300-node quadrature over every token)
FULL = [
    ("tiny", ["IS", "WIS", "single", "SpecTr"]),
    ("llama2-32k", ["WIS", "single", "SpecTr", "IS"]),
    ("two-models-50k", ["WIS", "SpecTr", "single", "IS"]),
    ("llama3-128k", ["WIS", "single", "SpecTr"]),
    ("serving-152k", ["single", "WIS", "SpecTr", "IS"]),
    ("serving-152k-k2", ["single", "WIS", "SpecTr", "IS"]),
]


@pytest.mark.parametrize("name,schemes", FULL, ids=[f[0] for f in FULL])
def test_full_size_workloads_sampled(name, schemes):
    spec = WORKLOADS[name]
    for scheme in schemes:
        seqs = spread(spec.B, 8 if scheme == "IS" else 32)
        res = run_both(spec, scheme, seed=spec.verify_seed, seqs=seqs)
        check(res, scheme)
        assert res["status"] == 0


def test_dataflow_launches_are_reproducible():
    # The slice-dataflow engine: a sequence's result may not depend on which
    # CTA takes which slice, on the batch of the call (the slice geometry is
    # fixed by the context's max_B) or on what ran before.  Bit-identical
    # tokens, accept lengths and diagnostics across repeated and interleaved
    # launches and across a prefix batch.
    spec = small("llama2-32k", B=24, V=12007, K=4, model_ids=[0, 0, 1, 1], draft_sigma=[1.0, 0.6],
                 t_draft=[1.2, 0.9])
    w = make_workload(spec, device=DEV)
    other = make_workload(small("tiny", B=8), device=DEV)
    v = mds.Verifier(64, spec.K, spec.L, spec.V, dtype=spec.dtype)

    def run(scheme, B):
        out, acc, diag = v.verify(w.target[:B], [d[:B] for d in w.draft_list()], w.model_ids, w.tokens[:B],
                                  w.temps[:B], scheme, 21, diag=True)
        torch.cuda.synchronize()
        acc_h = acc.cpu().numpy().copy()
        dg = diag.cpu().numpy().copy()
        for b in range(B):             # depths past the walk's end are not written
            dg[b, acc_h[b] + 1:] = 0.0
        return out.cpu().numpy().copy(), acc_h, dg

    for scheme in ("WIS", "single", "WIS0"):
        ref = run(scheme, spec.B)
        assert v.cluster_size == 0, "the dataflow engine serves this call"
        for rep in range(3):
            t = mds.Verifier(8, other.spec.K, other.spec.L, other.spec.V, dtype=other.spec.dtype)
            t.verify(other.target, other.draft_list(), other.model_ids, other.tokens, other.temps, "WIS", rep)
            torch.cuda.synchronize()
            t.close()
            for B in (spec.B, 13):
                got = run(scheme, B)
                for nm, a, b in zip(("tokens", "accept", "diag"), ref, got):
                    a = a[:B]
                    same = (a == b) | (np.isnan(a) & np.isnan(b)) if a.dtype.kind == "f" else a == b
                    bad = np.argwhere(~same)
                    assert bad.size == 0, f"{scheme} rep {rep} B {B}: {nm} differs at {bad[:4].tolist()}"
    assert v.status()[0] == 0
    v.close()


@pytest.mark.parametrize("cluster", [2, 4])
def test_repeated_launches_are_identical(cluster):
    # The result of a sequence may not depend on which cluster takes it, on
    # the launch's cluster count or on what ran before: repeat the same
    # verification with different batch capacities (so different grids) and
    # interleaved launches of another configuration.
    spec = small("llama2-32k", B=24, V=12007, K=4, model_ids=[0, 0, 1, 1], draft_sigma=[1.0, 0.6],
                 t_draft=[1.2, 0.9])
    w = make_workload(spec, device=DEV)
    other = make_workload(small("tiny", B=8), device=DEV)
    ref = {}
    for rep, max_B in enumerate((24, 24, 64, 200, 24)):
        v = mds.Verifier(max_B, spec.K, spec.L, spec.V, dtype=spec.dtype, cluster=cluster)
        for scheme in ("WIS", "SpecTr", "IS"):
            out, acc, diag = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, 21,
                                      diag=True)
            torch.cuda.synchronize()
            acc_h = acc.cpu().numpy().copy()
            dg = diag.cpu().numpy().copy()
            for b in range(spec.B):         # depths past the walk's end are not written
                dg[b, acc_h[b] + 1:] = 0.0
            got = (out.cpu().numpy().copy(), acc_h, dg)
            if scheme not in ref:
                ref[scheme] = got
            else:
                for name, a, b in zip(("tokens", "accept", "diag"), ref[scheme], got):
                    bad = np.argwhere(~((a == b) | (np.isnan(a) & np.isnan(b)) if a.dtype.kind == "f" else a == b))
                    assert bad.size == 0, (f"{scheme} launch {rep}: {name} differs at {bad[:4].tolist()}: "
                                           f"{a[tuple(bad[0])]} vs {b[tuple(bad[0])]}")
        assert v.status()[0] == 0
        v.close()
        t = mds.Verifier(8, other.spec.K, other.spec.L, other.spec.V, dtype=other.spec.dtype)
        t.verify(other.target, other.draft_list(), other.model_ids, other.tokens, other.temps, "WIS", rep)
        torch.cuda.synchronize()
        t.close()


def test_host_entry_point_reads_pinned_logits_in_place():
    # mds_verify_host: pinned logits are read in place (plain loads over the
    # host link), pageable ones are copied first; both must give exactly the
    # device entry point's result
    spec = small("two-models-50k", B=8, V=6000)
    w = make_workload(spec, device=DEV)
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype)
    out, acc, diag = v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WIS", 3, diag=True)
    torch.cuda.synchronize()
    ref = (out.cpu().numpy(), acc.cpu().numpy())
    for pinned in (True, False):
        def host(t):
            t = t.cpu()
            return t.pin_memory() if pinned else t
        h_out = torch.empty(spec.B, spec.L + 1, dtype=torch.int32)
        h_acc = torch.empty(spec.B, dtype=torch.int32)
        h_out, h_acc = (h_out.pin_memory(), h_acc.pin_memory()) if pinned else (h_out, h_acc)
        mds.mds_verify_host(v.ctx, host(w.target), [host(d) for d in w.draft_list()], w.model_ids, host(w.tokens),
                            host(w.temps), "WIS", 3, h_out, h_acc)
        assert np.array_equal(h_out.numpy(), ref[0]), f"pinned={pinned}"
        assert np.array_equal(h_acc.numpy(), ref[1]), f"pinned={pinned}"
    assert v.status()[0] == 0
    v.close()
