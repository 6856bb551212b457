"""Law of the CUDA path's output token, without the oracle.

Every scheme must emit target tokens (Theorem 1 with Algorithm 1; Section 4
for the truncated alphabet).  Here 65536 sequences share one target row and
one row per draft model, draw their own draft tokens from the draft laws and
their own Philox streams (sequence id = b), so the first emitted tokens are
65536 independent draws of the depth-0 output.  Their empirical law, with
the 15 most probable tokens kept apart and the rest pooled (so the test's
power does not fade with V), must be within total variation 4/sqrt(N) of q
computed in fp64 from the stored logits.  Both row layouts are covered:
V = 2048 (bulk copies) and V = 257 (plain loads).
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2410_18234_gb300 import mds  # noqa: E402

DEV = "cuda:0"
N = 65536


def _softmax64(logits, t):
    x = logits.astype(np.float64) / t
    e = np.exp(x - x.max())
    return e / e.sum()


def _case(V, model_ids, seed, n=N):
    K, L = len(model_ids), 1
    g = torch.Generator(device="cpu").manual_seed(seed)
    row = (3.0 * torch.randn(V, generator=g)).to(torch.bfloat16)
    n_models = max(model_ids) + 1
    sig = [0.6, 1.2, 0.9][:n_models]
    drows = [(row.float() + s * torch.randn(V, generator=g)).to(torch.bfloat16) for s in sig]
    t_target, t_draft = 1.0, [1.1, 0.8, 1.3][:n_models]
    temps = torch.tensor([t_target] + [t_draft[m] for m in model_ids], dtype=torch.float32)
    # each branch draws its token from its own model's law, independently per sequence
    tokens = torch.empty(n, K, L, dtype=torch.int32)
    for k, m in enumerate(model_ids):
        p = torch.from_numpy(_softmax64(drows[m].float().numpy(), t_draft[m]))
        tokens[:, k, 0] = torch.multinomial(p, n, replacement=True, generator=g).to(torch.int32)
    target = row.to(DEV).view(1, 1, 1, V).expand(n, K, L + 1, V).contiguous()
    drafts = [drows[m].to(DEV).view(1, 1, V).expand(n, L, V).contiguous() for m in model_ids]
    q = _softmax64(row.float().numpy(), t_target)
    return target, drafts, tokens.to(DEV), temps.to(DEV).view(1, -1).expand(n, -1).contiguous(), q


def _coarse_tv(z, q):
    top = np.argsort(-q, kind="stable")[:15]
    emp = np.bincount(z, minlength=len(q)) / len(z)
    rest_q = 1.0 - q[top].sum()
    rest_e = 1.0 - emp[top].sum()
    return 0.5 * (np.abs(emp[top] - q[top]).sum() + abs(rest_e - rest_q))


@pytest.mark.parametrize("V", [2048, 257])
def test_first_token_follows_the_target(V):
    model_ids = [0, 0, 1, 1]
    target, drafts, tokens, temps, q = _case(V, model_ids, seed=V)
    v = mds.Verifier(N, len(model_ids), 1, V, dtype="bf16", omega0=5)
    for scheme in ("single", "IS", "WIS", "SpecTr", "WIS0"):
        out, acc, _ = v.verify(target, drafts, model_ids, tokens, temps, scheme, seed=123)
        torch.cuda.synchronize()
        z = out[:, 0].cpu().numpy().astype(np.int64)
        assert z.min() >= 0 and z.max() < V
        tv = _coarse_tv(z, q)
        assert tv < 4.0 / np.sqrt(N), (scheme, tv)
    assert v.status()[0] == 0
    v.close()


def test_first_token_follows_the_target_at_a_million_draws():
    """N = 2^20 draws (threshold 4/sqrt(N) = 0.0039) for the two weighted
    schemes on V = 257."""
    n = 1 << 20
    model_ids = [0, 0, 1, 1]
    target, drafts, tokens, temps, q = _case(257, model_ids, seed=11, n=n)
    v = mds.Verifier(n, len(model_ids), 1, 257, dtype="bf16", omega0=5)
    for scheme in ("WIS", "WIS0"):
        out, acc, _ = v.verify(target, drafts, model_ids, tokens, temps, scheme, seed=99)
        torch.cuda.synchronize()
        tv = _coarse_tv(out[:, 0].cpu().numpy().astype(np.int64), q)
        assert tv < 4.0 / np.sqrt(n), (scheme, tv)
    assert v.status()[0] == 0
    v.close()
