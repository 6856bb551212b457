"""Seeded synthetic multi-draft workloads.

This module only makes inputs: target logits per draft-tree node, draft
logits per (node, draft model), the draft tokens of every branch and the
temperatures.  It holds none of the verification arithmetic and serves both
the CUDA path and the oracle, which always read the same tensors (the oracle
a host copy).

Tree.  Sequence b has K branches of L draft tokens.  A node is a token prefix;
every branch starts at the shared root.  Each node carries one target row and
one draft row per draft model; rows are generated per (branch, depth) and
then made equal across branches that share a prefix (and, for draft rows, a
model), so the dense per-branch buffers are consistent with one tree.  Branch
k's token at depth j is sampled independently from its own draft
distribution softmax(l_d / T_k) at its node, by the Gumbel-max rule applied
to the stored (rounded) logits; with top_k set, only the row's top_k logits
(and any tied with the k-th) take part.

Logits.  target = scale * N(0,1) (plus an optional boost of the largest
entries), draft = target + sigma * N(0,1), both drawn in fp32 and then
rounded to the storage dtype; the draft is derived from the unrounded target.
Normals come from torch's seeded generator on the requested device.

The five named workloads follow the shapes of the paper's setting (draft and
target models with vocabularies of 4k to 152k tokens, K = 2..8 drafts,
L = 4..8 draft positions, temperatures 0.5..2.0) and stand in for the
paper's OPT/XSum/Dolly/WMT18 runs, whose weights and data are not used.
"""
from dataclasses import dataclass, field, replace
from typing import List, Optional, Sequence

import torch


@dataclass
class WorkloadSpec:
    name: str
    B: int
    K: int
    L: int
    V: int
    dtype: str                      # "f32" | "bf16"
    model_ids: List[int]
    target_scale: float
    draft_sigma: Sequence[float]    # per draft model, or per-sequence cycle when sigma_per_seq
    t_target: float
    t_draft: Sequence[float]        # per draft model
    top_boost: int = 0              # number of largest target entries boosted
    boost: float = 0.0
    sigma_per_seq: bool = False     # sigma_b = draft_sigma[b % len]
    temp_per_seq: Optional[tuple] = None   # (lo, hi): T_b ~ U[lo, hi] shared by target and drafts
    schemes: List[str] = field(default_factory=list)
    data_seed: int = 0
    verify_seed: int = 1
    top_k: int = 0                  # > 0: each branch samples from its draft row's top_k logits only

    def with_(self, **kw):
        return replace(self, **kw)


WORKLOADS = {
    "tiny": WorkloadSpec("tiny", B=4, K=2, L=4, V=4096, dtype="f32", model_ids=[0, 0], target_scale=3.0,
                         draft_sigma=[0.7], t_target=1.0, t_draft=[1.0], schemes=["IS"], data_seed=1000,
                         verify_seed=0),
    "llama2-32k": WorkloadSpec("llama2-32k", B=64, K=4, L=5, V=32000, dtype="bf16", model_ids=[0, 0, 0, 0],
                               target_scale=4.0, draft_sigma=[1.0], t_target=1.0, t_draft=[1.2], top_boost=50,
                               boost=6.0, schemes=["IS", "WIS"], data_seed=1001),
    "two-models-50k": WorkloadSpec("two-models-50k", B=128, K=2, L=4, V=50272, dtype="bf16", model_ids=[0, 1],
                                   target_scale=4.0, draft_sigma=[0.5, 1.5], t_target=1.0, t_draft=[1.0, 2.0],
                                   schemes=["WIS", "SpecTr"], data_seed=1002),
    "llama3-128k": WorkloadSpec("llama3-128k", B=256, K=8, L=4, V=128256, dtype="bf16", model_ids=[0] * 8,
                                target_scale=5.0, draft_sigma=[0.8], t_target=0.7, t_draft=[0.7],
                                schemes=["WIS"], data_seed=1003),
    "serving-152k": WorkloadSpec("serving-152k", B=1024, K=4, L=8, V=151936, dtype="bf16", model_ids=[0] * 4,
                                 target_scale=4.0, draft_sigma=[0.3, 1.0, 2.0], t_target=1.0, t_draft=[1.0],
                                 sigma_per_seq=True, temp_per_seq=(0.5, 1.5),
                                 schemes=["single", "IS", "WIS", "SpecTr"], data_seed=1004),
    # the same serving sweep with K = 2 draft branches (its other arm)
    "serving-152k-k2": WorkloadSpec("serving-152k-k2", B=1024, K=2, L=8, V=151936, dtype="bf16", model_ids=[0] * 2,
                                    target_scale=4.0, draft_sigma=[0.3, 1.0, 2.0], t_target=1.0, t_draft=[1.0],
                                    sigma_per_seq=True, temp_per_seq=(0.5, 1.5),
                                    schemes=["single", "IS", "WIS", "SpecTr"], data_seed=1005),
}


@dataclass
class Workload:
    spec: WorkloadSpec
    target: torch.Tensor          # [B, K, L+1, V] storage dtype
    drafts: torch.Tensor          # [K, B, L, V] storage dtype (branch k's rows: drafts[k])
    tokens: torch.Tensor          # [B, K, L] int32
    temps: torch.Tensor           # [B, 1+K] float32
    model_ids: List[int]

    def draft_list(self):
        return [self.drafts[k] for k in range(self.spec.K)]


def _storage(dtype):
    return {"f32": torch.float32, "bf16": torch.bfloat16}[dtype]


def make_workload(spec: WorkloadSpec, device="cpu", seed=None) -> Workload:
    """Generate the workload described by ``spec`` on ``device``."""
    B, K, L, V = spec.B, spec.K, spec.L, spec.V
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(spec.data_seed if seed is None else int(seed))
    st = _storage(spec.dtype)
    mids = torch.tensor(spec.model_ids, device=dev)
    n_models = int(max(spec.model_ids)) + 1

    # temperatures [B, 1+K]
    temps = torch.empty(B, 1 + K, dtype=torch.float32, device=dev)
    if spec.temp_per_seq is not None:
        lo, hi = spec.temp_per_seq
        tb = lo + (hi - lo) * torch.rand(B, generator=g, device=dev)
        temps[:] = tb[:, None]
    else:
        temps[:, 0] = spec.t_target
        for k in range(K):
            temps[:, 1 + k] = float(spec.t_draft[spec.model_ids[k]])

    # draft noise scale per (b, k)
    if spec.sigma_per_seq:
        cyc = torch.tensor(spec.draft_sigma, dtype=torch.float32, device=dev)
        sig = cyc[torch.arange(B, device=dev) % len(spec.draft_sigma)][:, None].expand(B, K)
    else:
        per_model = torch.tensor([float(spec.draft_sigma[m]) for m in spec.model_ids], dtype=torch.float32,
                                 device=dev)
        sig = per_model[None, :].expand(B, K)

    target = torch.empty(B, K, L + 1, V, dtype=st, device=dev)
    drafts = torch.empty(K, B, L, V, dtype=st, device=dev)
    tokens = torch.empty(B, K, L, dtype=torch.int32, device=dev)

    # same_prefix[b, k, k'] : branches k and k' share the prefix so far
    same = torch.ones(B, K, K, dtype=torch.bool, device=dev)
    same_model = (mids[:, None] == mids[None, :])[None]
    ar = torch.arange(K, device=dev)
    for j in range(L + 1):
        # lowest branch with the same prefix (target rows) / same prefix and model (draft rows)
        rep_t = torch.where(same, ar[None, None, :], K).min(dim=2).values
        rep_d = torch.where(same & same_model, ar[None, None, :], K).min(dim=2).values
        t32 = spec.target_scale * torch.randn(B, K, V, generator=g, device=dev)
        if spec.top_boost > 0:
            idx = torch.topk(t32, spec.top_boost, dim=2).indices
            t32.scatter_add_(2, idx, torch.full(idx.shape, spec.boost, device=dev))
        t32 = torch.gather(t32, 1, rep_t[:, :, None].expand(B, K, V))
        target[:, :, j] = t32.to(st)
        if j == L:
            break
        d32 = t32 + sig[:, :, None] * torch.randn(B, K, V, generator=g, device=dev)
        d32 = torch.gather(d32, 1, rep_d[:, :, None].expand(B, K, V))
        d_st = d32.to(st)
        drafts[:, :, j] = d_st.permute(1, 0, 2)
        # each branch samples its own token at its node (Gumbel-max on the stored logits)
        u = torch.rand(B, K, V, generator=g, device=dev).clamp_(min=1e-12)
        gum = -torch.log(-torch.log(u))
        score = d_st.float() / temps[:, 1:, None] + gum
        if spec.top_k > 0:
            # sample from the row's top_k logits (every logit tied with the k-th is kept)
            kth = torch.topk(d_st.float(), min(spec.top_k, V), dim=2).values[:, :, -1:]
            score = torch.where(d_st.float() >= kth, score, torch.full_like(score, float("-inf")))
        tk = score.argmax(dim=2)
        tokens[:, :, j] = tk.to(torch.int32)
        same = same & (tk[:, :, None] == tk[:, None, :])
    return Workload(spec, target, drafts, tokens, temps, list(spec.model_ids))


def host_copy(w: Workload, seqs=None):
    """numpy arrays for the oracle: fp32 logits (exact upcast of the stored
    values), int64 tokens, float32 temperatures.  With ``seqs`` only those
    sequences are copied (in that order)."""
    if seqs is None:
        sel = slice(None)
    else:
        sel = torch.as_tensor(list(seqs), dtype=torch.long, device=w.target.device)
    target = w.target[sel].float().cpu().numpy()
    drafts = [w.drafts[k][sel].float().cpu().numpy() for k in range(w.spec.K)]
    return (target, drafts, list(w.model_ids), w.tokens[sel].cpu().numpy().astype("int64"),
            w.temps[sel].cpu().numpy())
