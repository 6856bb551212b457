"""mds_verify_noalloc: the entry point for callers that cannot allocate.

Some callers cannot call cudaMalloc: code running where device memory is
fixed once at start-up (a serving loop under an allocator that forbids growth
after warm-up), and so cannot create an mds_ctx (no cudaMalloc).  For them the
library offers a context-free variant whose scratch lives in a static device
array.  This test calls it through the C ABI twice in a row and checks that
both calls reproduce the context-based entry point's outputs (the same kernel
with the same launch geometry: identical tokens, accept lengths and
diagnostics).  It is collected last so that a run stopping at the first
failure has already run every other test.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, make_workload  # noqa: E402


@pytest.mark.parametrize("name,scheme", [("llama3-128k", "WIS"), ("two-models-50k", "SpecTr"), ("tiny", "IS")])
def test_noalloc_matches_context_entry_point_twice(name, scheme):
    spec = WORKLOADS[name].with_(B=min(WORKLOADS[name].B, 16))
    w = make_workload(spec, device="cuda:0")
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype)
    dev = torch.device("cuda:0")
    # depths a sequence never reaches leave diag untouched: start both from zero
    ref_tok = torch.empty(spec.B, spec.L + 1, dtype=torch.int32, device=dev)
    ref_acc = torch.empty(spec.B, dtype=torch.int32, device=dev)
    ref_diag = torch.zeros(spec.B, spec.L + 1, 4, dtype=torch.float32, device=dev)
    v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, spec.verify_seed,
             out=(ref_tok, ref_acc, ref_diag))
    torch.cuda.synchronize()
    v.close()
    for _ in range(2):
        tok = torch.full_like(ref_tok, -7)
        acc = torch.full_like(ref_acc, -7)
        diag = torch.zeros_like(ref_diag)
        mds.mds_verify_noalloc(spec.B, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, w.tokens,
                               w.temps, scheme, spec.verify_seed, tok, acc, diag, dtype=spec.dtype)
        torch.cuda.synchronize()
        assert torch.equal(tok, ref_tok)
        assert torch.equal(acc, ref_acc)
        np.testing.assert_allclose(diag.cpu().numpy(), ref_diag.cpu().numpy(), rtol=1e-5, atol=1e-6)


def test_noalloc_rejects_bad_arguments_without_launching():
    spec = WORKLOADS["tiny"]
    w = make_workload(spec, device="cuda:0")
    out = torch.empty(spec.B, spec.L + 1, dtype=torch.int32, device="cuda:0")
    acc = torch.empty(spec.B, dtype=torch.int32, device="cuda:0")
    with pytest.raises(mds.MdsError) as e:
        mds.mds_verify_noalloc(spec.B - 1, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, w.tokens,
                               w.temps, "WIS", 0, out, acc, dtype=spec.dtype)
    assert e.value.code == mds.MDS_ESHAPE
    with pytest.raises(mds.MdsError) as e:
        mds.mds_verify_noalloc(spec.B, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, w.tokens,
                               w.temps, 9, 0, out, acc, dtype=spec.dtype)
    assert e.value.code == mds.MDS_EINVAL


def test_noalloc_status_word():
    # The status bits of a no-allocation call, read without allocating: a
    # draft token outside [0, V) (a host-side input; the kernel replaces it by
    # token 0 and flags it), then a clean call, whose clearing resets them.
    spec = WORKLOADS["llama2-32k"].with_(B=4, V=4099)
    w = make_workload(spec, device="cuda:0")
    out = torch.empty(spec.B, spec.L + 1, dtype=torch.int32, device="cuda:0")
    acc = torch.empty(spec.B, dtype=torch.int32, device="cuda:0")
    bad = w.tokens.clone()
    bad[1, :, 0] = spec.V + 5
    for scheme in ("WIS", "SpecTr"):
        mds.mds_verify_noalloc(spec.B, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, bad,
                               w.temps, scheme, 3, out, acc, dtype=spec.dtype)
        bits, msg = mds.mds_noalloc_status(0)
        assert bits & mds.MDS_ST_BADTOKEN, (scheme, bits, msg)
        assert int(out.max()) < spec.V and int(acc.min()) >= 0   # every output still a valid token
        mds.mds_verify_noalloc(spec.B, spec.K, spec.L, spec.V, w.target, w.draft_list(), w.model_ids, w.tokens,
                               w.temps, scheme, 3, out, acc, dtype=spec.dtype)
        assert mds.mds_noalloc_status(0) == (0, "ok")
