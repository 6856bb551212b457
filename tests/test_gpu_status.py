"""Data anomalies reach the status word; argument errors return codes.

A temperature <= 0 is replaced by 1 and flagged (MDS_ST_BADTEMP); a draft
token outside [0, V) is replaced by token 0 and flagged (MDS_ST_BADTOKEN);
the outputs stay valid tokens.  B above the context's max_B and an unknown
scheme id are rejected before any launch.  None of these faults the GPU:
each anomaly is checked by the kernel before the value is used.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, make_workload  # noqa: E402

DEV = "cuda:0"


def _run(w, scheme, **mut):
    spec = w.spec
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype)
    temps, tokens = w.temps.clone(), w.tokens.clone()
    if "temp" in mut:
        temps[1, 0] = mut["temp"]
    if "token" in mut:
        tokens[2, 0, 0] = mut["token"]
    out, acc, _ = v.verify(w.target, w.draft_list(), w.model_ids, tokens, temps, scheme, 5)
    torch.cuda.synchronize()
    bits, msg = v.status()
    v.close()
    return out.cpu().numpy(), acc.cpu().numpy(), bits, msg


@pytest.mark.parametrize("scheme", ["single", "WIS", "SpecTr", "WIS0"])
def test_bad_temperature_and_token_are_flagged(scheme):
    w = make_workload(WORKLOADS["llama2-32k"].with_(B=6, V=3001), device=DEV)
    V = w.spec.V
    for mut, bit in ((dict(temp=0.0), mds.MDS_ST_BADTEMP), (dict(temp=-1.0), mds.MDS_ST_BADTEMP),
                     (dict(token=V), mds.MDS_ST_BADTOKEN), (dict(token=-3), mds.MDS_ST_BADTOKEN)):
        out, acc, bits, msg = _run(w, scheme, **mut)
        assert bits & bit, (scheme, mut, bits, msg)
        for b in range(w.spec.B):
            n = int(acc[b]) + 1
            assert ((out[b, :n] >= 0) & (out[b, :n] < V)).all()
            assert (out[b, n:] == -1).all()
    out, acc, bits, msg = _run(w, scheme)
    assert bits == 0, msg


def test_argument_errors_return_codes():
    w = make_workload(WORKLOADS["tiny"].with_(B=4, V=500), device=DEV)
    spec = w.spec
    v = mds.Verifier(2, spec.K, spec.L, spec.V, dtype=spec.dtype)
    with pytest.raises(mds.MdsError) as e:
        v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, "WIS", 1)    # B = 4 > max_B = 2
    assert e.value.code == mds.MDS_ESHAPE
    with pytest.raises(mds.MdsError) as e:
        v.verify(w.target[:2], [d[:2] for d in w.draft_list()], w.model_ids, w.tokens[:2], w.temps[:2], 9, 1)
    assert e.value.code == mds.MDS_EINVAL
    assert v.status()[0] == 0
    v.close()
