"""CUDA path vs the oracle for the truncated-alphabet scheme (WIS0).

Omega_0 sizes from 1 to the largest supported one, vocabularies smaller
than Omega_0 (Omega_0 = the whole vocabulary), more draft models than one
statistics pass holds, every cluster size, rows fetched with plain loads,
peaked targets, and sampled sequences of the full-size workloads.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, WorkloadSpec  # noqa: E402
from parity import check  # noqa: E402
from test_gpu_parity import run_both, small  # noqa: E402


def ok(res, allow_uncertified=False):
    check(res, "WIS0")
    bits = res["status"] & ~(mds.MDS_ST_OMEGA0 if allow_uncertified else 0)
    assert bits == 0, res["status"]


@pytest.mark.parametrize("name,kw", [
    ("tiny", dict()),
    ("llama2-32k", dict(B=12, V=5003)),
    ("two-models-50k", dict(B=16, V=7001)),
    ("llama3-128k", dict(B=12, V=9000)),
    ("serving-152k", dict(B=12, V=6007, L=5)),
], ids=lambda x: x if isinstance(x, str) else "")
def test_small_workloads(name, kw):
    spec = small(name, **kw)
    for M in (1, 5, 20):
        ok(run_both(spec, "WIS0", seed=11 + M, omega0=M))


def test_largest_omega0_on_f32_rows():
    # f32 logits have no ties, so the cut of the largest Omega_0 is certified
    spec = small("tiny", B=8, V=5000)
    ok(run_both(spec, "WIS0", seed=3, omega0=mds.MDS_MAX_OMEGA0))
    ok(run_both(spec, "WIS0", seed=4, omega0=mds.MDS_MAX_OMEGA0_CLUSTER, cluster=2))


@pytest.mark.parametrize("name,kw", [
    ("llama3-128k", dict(B=12, V=9000)),
    ("two-models-50k", dict(B=12, V=7001, dtype="f32")),
    ("serving-152k", dict(B=10, V=6007, L=4)),
], ids=lambda x: x if isinstance(x, str) else "")
def test_paper_omega0_sizes(name, kw):
    # |Omega_0| = 40 and 50 (Section 5's runs) and the largest size: a
    # 64-entry list, two entries per lane of the decision warp (bf16 ties at
    # the cut may leave it uncertified)
    spec = small(name, **kw)
    for M in (31, 40, 50, mds.MDS_MAX_OMEGA0):
        ok(run_both(spec, "WIS0", seed=M, omega0=M), allow_uncertified=(spec.dtype == "bf16"))


def test_large_omega0_needs_the_dataflow_engine():
    # the per-sequence engine's list holds 32 entries: a cluster size with
    # |Omega_0| above 30 is refused before any launch
    spec = small("tiny", B=4, V=3000)
    from synth import make_workload
    w = make_workload(spec, device="cuda:0")
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, cluster=2, omega0=40)
    with pytest.raises(mds.MdsError) as e:
        v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WIS0", 1)
    assert e.value.code == mds.MDS_EUNSUP
    v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WIS", 1)   # other schemes run
    torch.cuda.synchronize()
    v.close()


@pytest.mark.parametrize("cluster", [1, 2, 4, 8, 16])
def test_every_cluster_size(cluster):
    spec = small("llama2-32k", B=6, V=4099, K=3, model_ids=[0, 0, 0])
    res = run_both(spec, "WIS0", seed=5, cluster=cluster, omega0=10)
    assert res["cn"] == cluster
    ok(res)


@pytest.mark.parametrize("V", [1, 2, 3, 5, 9, 17, 31, 40, 100])
def test_tiny_vocabularies(V):
    for dtype in ("f32", "bf16"):
        spec = WorkloadSpec(f"v{V}", B=24, K=3, L=3, V=V, dtype=dtype, model_ids=[0, 0, 1], target_scale=2.0,
                            draft_sigma=[0.5, 1.0], t_target=1.0, t_draft=[1.0, 1.3], data_seed=V)
        for M in (1, 5, 30, 45):
            # bf16 ties at the cut can leave the larger Omega_0 uncertified
            ok(run_both(spec, "WIS0", seed=V + M, omega0=M, wis_s=min(5, max(1, V))),
               allow_uncertified=(dtype == "bf16" and M >= 30))


def test_more_draft_models_than_one_pass_holds():
    spec = WorkloadSpec("five", B=12, K=5, L=3, V=3000, dtype="bf16", model_ids=[0, 1, 2, 3, 4], target_scale=3.0,
                        draft_sigma=[0.5, 1.0, 1.5, 0.7, 0.3], t_target=1.0, t_draft=[1.0, 1.2, 0.8, 1.0, 1.5],
                        data_seed=23)
    for M in (3, 20):
        ok(run_both(spec, "WIS0", seed=M, omega0=M))


def test_peaked_targets_and_plain_loads():
    spec = WorkloadSpec("peaked", B=16, K=6, L=4, V=2048, dtype="bf16", model_ids=[0] * 6, target_scale=12.0,
                        draft_sigma=[0.2], t_target=0.5, t_draft=[0.5], data_seed=3)
    ok(run_both(spec, "WIS0", seed=8, omega0=10))
    spec = small("two-models-50k", B=8, V=4097)     # 8194-byte rows: plain loads
    ok(run_both(spec, "WIS0", seed=6, omega0=20))
    spec = small("tiny", V=1001)                     # f32, 4004-byte rows
    ok(run_both(spec, "WIS0", seed=6, omega0=20))


def test_s_values():
    spec = small("llama3-128k", B=8, V=3000)
    for s in (1, 2, 3, 8):
        ok(run_both(spec, "WIS0", seed=4, wis_s=s, omega0=12))


@pytest.mark.parametrize("name,n", [("llama3-128k", 24), ("serving-152k", 16), ("two-models-50k", 16)],
                         ids=lambda x: x if isinstance(x, str) else "")
def test_full_size_sampled(name, n):
    # the bench's launch configuration; |Omega_0| = 20 and the paper's 40
    spec = WORKLOADS[name]
    seqs = sorted(set(np.linspace(0, spec.B - 1, n).round().astype(int).tolist()))
    for M in (20, 40):
        ok(run_both(spec, "WIS0", seed=spec.verify_seed, seqs=seqs, omega0=M),
           allow_uncertified=(M == 40 and spec.dtype == "bf16"))


def test_config_rejects_out_of_range_omega0():
    spec = small("tiny", B=4)
    for bad in (-1, mds.MDS_MAX_OMEGA0 + 1):
        with pytest.raises(mds.MdsError):
            mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, omega0=bad)
