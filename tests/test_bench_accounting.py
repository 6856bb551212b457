"""Host logic of bench.py: the vocab-row and algorithmic-byte accounting
replayed from a walk's outputs, for WIS (every visited row streamed) and the
truncated alphabet (target rows streamed, draft rows read at Omega_0); the
kernel a call runs and the recorded DRAM traffic of its current source."""
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def _walk():
    # B = 2, K = 3, L = 2; branches 0, 1 share model 0, branch 2 is model 1
    tokens = np.array([[[5, 7], [5, 8], [6, 9]],
                       [[1, 2], [1, 2], [1, 2]]], dtype=np.int64)
    mids = [0, 0, 1]
    out = np.array([[5, 8, -1],      # depth 0 keeps branches 0, 1 (model 0); depth 1: Z = 8 keeps branch 1
                    [3, -1, -1]], dtype=np.int64)   # depth 0 rejects every branch
    acc = np.array([2, 0])
    return tokens, mids, out, acc


def test_wis_counts_every_visited_row():
    tokens, mids, out, acc = _walk()
    V, es = 1000, 2
    rows, abytes = bench.walk_accounting(tokens, mids, out, acc, V, es)
    # seq 0: depth 0 target + 2 models, depth 1 target + 1 model, bonus target = 6 rows; seq 1: 3 rows
    assert rows == 9
    io = 2 * 4 * (3 * 2 + (1 + 3) + (2 + 1) + 1)
    assert abytes == rows * V * es + io


def test_truncated_alphabet_counts_target_rows_and_point_loads():
    tokens, mids, out, acc = _walk()
    V, es, M = 1000, 2, 20
    rows, abytes = bench.walk_accounting(tokens, mids, out, acc, V, es, "WIS0", M)
    assert rows == 9
    draft_rows = 2 + 1 + 2          # per visited depth, one per distinct draft model
    io = 2 * 4 * (3 * 2 + (1 + 3) + (2 + 1) + 1)
    assert abytes == (rows - draft_rows) * V * es + draft_rows * M * es + io
    # Omega_0 larger than the vocabulary reads each draft row in full at most
    _, small = bench.walk_accounting(tokens, mids, out, acc, 8, es, "WIS0", M)
    assert small == (rows - draft_rows) * 8 * es + draft_rows * 8 * es + io


def test_kernel_names_and_recorded_traffic():
    assert bench.kernel_name("WIS", 0) == "flow_kernel"
    assert bench.kernel_name("WIS", 2) == "verify_kernel"
    assert bench.kernel_name("SpecTr", 0) == "verify_kernel"
    assert bench.kernel_name("WIS", 0, top_k=10) == "topk_kernel"
    # every committed record names its kernel and matches that kernel's
    # current source, so the bench line reports it; another kernel's record
    # or a stale hash reads as unknown
    import json
    d = json.load(open(os.path.join(bench.ROOT, "profiles", "traffic.json")))
    for key, e in d.items():
        parts = key.split("/")
        top_k = int(parts[2][3:]) if len(parts) > 2 else 0
        assert bench.recorded_traffic(parts[0], parts[1], e["kernel"], top_k) == e["dram_bytes_per_launch"]
        other = "verify_kernel" if e["kernel"] != "verify_kernel" else "flow_kernel"
        assert bench.recorded_traffic(parts[0], parts[1], other, top_k) is None
    assert bench.recorded_traffic("llama3-128k", "WIS", "flow_kernel", 5) is None
