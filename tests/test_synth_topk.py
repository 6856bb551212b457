"""The seeded workloads with top_k set: each branch's draft token lies among
its draft row's k largest logits (ties with the k-th included), as Section 5
samples the drafts of its top-k runs; without top_k the tokens are not so
restricted.  Input generation only (no verification arithmetic)."""
import numpy as np

from synth import WORKLOADS, make_workload


def _in_top_k(w, k):
    drafts = w.drafts.float().numpy()          # [K, B, L, V]
    tokens = w.tokens.numpy()                   # [B, K, L]
    K, B, L, V = drafts.shape
    inside = np.zeros((B, K, L), dtype=bool)
    for b in range(B):
        for kb in range(K):
            for j in range(L):
                row = drafts[kb, b, j]
                kth = np.sort(row)[::-1][min(k, V) - 1]
                inside[b, kb, j] = row[tokens[b, kb, j]] >= kth
    return inside


def test_top_k_drafts_come_from_the_restricted_rows():
    for k in (1, 5):
        spec = WORKLOADS["llama2-32k"].with_(B=6, V=3001, top_k=k)
        assert _in_top_k(make_workload(spec), k).all()


def test_unrestricted_drafts_reach_outside_the_top_k():
    spec = WORKLOADS["llama2-32k"].with_(B=6, V=3001)
    assert not _in_top_k(make_workload(spec), 1).all()
