"""Host logic of bench.py: the vocab-row and algorithmic-byte accounting
replayed from a walk's outputs, for WIS (every visited row streamed) and the
truncated alphabet (target rows streamed, draft rows read at Omega_0)."""
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
