"""Whole softmax rows of the CUDA path against the oracle (Sec. 3: q and p
are the softmaxes of the target and draft rows at their temperatures, Sec. 5).

The dataflow engine exports, for every (sequence, depth) its walk visits,
the statistics it derived for each streamed row (the row maximum M and 1/Z,
combined from every slice of the pass); `mds_debug_probs` then evaluates, for
every token of that row, the probability the kernel uses at any point of the
verification (the same device function).  Each element must match
`oracle.verify.softmax_t` in fp64 within 1e-5 relative (values in fp32's
normal range; below it the exponent flushes to zero, an absolute 1e-30).
Cases: a 152k bf16 vocabulary at T = 0.5, several draft models and mixed
temperatures in f32 with ragged slices, and the bench workload's rows.
"""
import math

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402
from synth import WORKLOADS, make_workload  # noqa: E402
from oracle.verify import softmax_t  # noqa: E402

RTOL = 1e-5          # the fp32 kernel against the fp64 oracle
FLOOR = 1e-30        # below fp32's normal range the kernel's exponent is 0


CASES = [
    ("serving-152k", dict(B=6, K=2, L=2, model_ids=[0, 0], temp_per_seq=None, t_target=0.5, t_draft=[0.5]),
     ["WIS", "single"]),
    ("two-models-50k", dict(B=5, K=3, L=2, V=10007, dtype="f32", model_ids=[0, 1, 2],
                            draft_sigma=[0.5, 1.0, 1.5], t_target=0.5, t_draft=[2.0, 1.0, 0.7]),
     ["WIS", "WIS0", "single"]),
    ("llama3-128k", dict(B=4), ["WIS"]),
]


def _rows(w, b, j, src):
    """The logit row a statistics entry refers to (src: the target row of
    branch src, or 100 + k for the draft row of branch k), and its temperature."""
    if src < 100:
        return w.target[b, src, j], float(w.temps[b, 0])
    k = src - 100
    return w.drafts[k][b, j], float(w.temps[b, 1 + k])


@pytest.mark.parametrize("name,kw,schemes", CASES, ids=[c[0] for c in CASES])
def test_softmax_rows_match_oracle(name, kw, schemes):
    spec = WORKLOADS[name].with_(**kw)
    w = make_workload(spec, device="cuda:0")
    v = mds.Verifier(spec.B, spec.K, spec.L, spec.V, dtype=spec.dtype, omega0=20)
    stats = torch.full((spec.B, spec.L + 1, mds.DEBUG_ROWS, 4), float("nan"), dtype=torch.float32, device="cuda:0")
    mds.mds_debug_row_stats(v.ctx, stats)
    out = torch.empty(spec.V, dtype=torch.float32, device="cuda:0")
    checked = 0
    for scheme in schemes:
        stats.fill_(float("nan"))
        v.verify(w.target, w.draft_list(), w.model_ids, w.tokens, w.temps, scheme, spec.verify_seed)
        torch.cuda.synchronize()
        assert v.cluster_size == 0, "the dataflow engine serves this call"
        st = stats.cpu().numpy()
        for b in range(spec.B):
            for j in range(spec.L + 1):
                for r in range(mds.DEBUG_ROWS):
                    M, iz, c, src = (float(x) for x in st[b, j, r])
                    if math.isnan(src):
                        continue
                    row, T = _rows(w, b, j, int(src))
                    assert c == pytest.approx(math.log2(math.e) / T, rel=1e-6)
                    assert M == float(row.float().max())
                    mds.mds_debug_probs(row.contiguous(), M, iz, c, out)
                    torch.cuda.synchronize()
                    g = out.cpu().numpy().astype(np.float64)
                    o = softmax_t(row.float().cpu().numpy(), T)
                    big = o >= FLOOR
                    rel = np.abs(g[big] - o[big]) / o[big]
                    assert rel.max() <= RTOL, (scheme, b, j, r, float(rel.max()), int(np.argmax(rel)))
                    assert np.all(np.abs(g[~big] - o[~big]) <= FLOOR)
                    checked += 1
    assert checked >= 2 * spec.B
    mds.mds_debug_row_stats(v.ctx, None)
    assert v.status()[0] == 0
    v.close()
