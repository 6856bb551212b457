"""Host-side logic of the N-GPU bench path, as world-size-2 gloo ranks on CPU.

Sequences are independent, so ranks shard the work with no collective on
the data path; the only collectives combine the whole-job figures (rows and
bytes summed, the slowest rank's time).  Each rank here verifies its own
batch with the oracle (no GPU) and combines through `bench.combine_ranks`;
the parent recomputes both shards alone and compares.
"""
import json
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _shard(spec, rank):
    import bench
    from synth import make_workload, host_copy
    from oracle.verify import oracle_verify
    w = make_workload(spec, device="cpu", seed=bench.rank_seed(spec, rank))
    tgt, drs, mids, toks, temps = host_copy(w)
    out, acc, _ = oracle_verify(tgt, drs, mids, toks, temps, "WIS", spec.verify_seed)
    es = 4 if spec.dtype == "f32" else 2
    rows, abytes = bench.walk_accounting(toks, w.model_ids, out, acc, spec.V, es)
    return rows, abytes, out


def _worker(rank, world, port, outdir):
    import torch.distributed as dist
    import bench
    from synth import WORKLOADS
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    spec = WORKLOADS["tiny"].with_(B=3, V=512)
    rows, abytes, out = _shard(spec, rank)
    ms = 10.0 + 5.0 * rank                     # stand-in per-rank times
    r_all, b_all, ms_all = bench.combine_ranks(rows, abytes, ms, world, "cpu")
    with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
        json.dump({"rows": rows, "abytes": abytes, "rows_all": r_all, "abytes_all": b_all, "ms": ms_all,
                   "out": out.tolist()}, f)
    dist.destroy_process_group()


def test_two_ranks_shard_and_combine(tmp_path):
    import torch.multiprocessing as mp
    from synth import WORKLOADS
    world = 2
    mp.spawn(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    spec = WORKLOADS["tiny"].with_(B=3, V=512)
    alone = [_shard(spec, r) for r in range(world)]
    for r in range(world):
        # each rank verified its own batch, exactly as a single process would
        assert res[r]["rows"] == alone[r][0] and res[r]["abytes"] == alone[r][1]
        assert np.array_equal(np.array(res[r]["out"]), alone[r][2])
        # whole-job figures: sums over ranks, the slowest rank's time, on every rank
        assert res[r]["rows_all"] == alone[0][0] + alone[1][0]
        assert res[r]["abytes_all"] == alone[0][1] + alone[1][1]
        assert res[r]["ms"] == 15.0
    # the shards are different batches (distinct seeds)
    assert not np.array_equal(np.array(res[0]["out"]), np.array(res[1]["out"]))
