"""The binding's buffer checks (no device needed): every call pattern the
GPU tests, the bench and smoke() use passes; wrong shapes, element types,
layouts, model-id counts and placements are rejected before the C call."""
import os

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2410_18234_gb300", "_lib", "libmds.so")


@pytest.fixture(scope="module")
def mds():
    if not os.path.exists(LIB):
        from paper_2410_18234_gb300 import build
        build.build()
    from paper_2410_18234_gb300 import mds as m
    return m


def _outs(B, L, diag=True):
    return (torch.empty(B, L + 1, dtype=torch.int32), torch.empty(B, dtype=torch.int32),
            torch.empty(B, L + 1, 4, dtype=torch.float32) if diag else None)


def _args(w):
    return (w.target, w.draft_list(), w.model_ids, w.tokens, w.temps)


@pytest.mark.parametrize("name,kw", [("tiny", dict()), ("llama2-32k", dict(B=3, V=500)),
                                     ("two-models-50k", dict(B=3, V=700)), ("llama3-128k", dict(B=2, V=300)),
                                     ("serving-152k", dict(B=2, V=301, L=5))])
def test_workload_calls_pass(mds, name, kw):
    from synth import WORKLOADS, make_workload
    spec = WORKLOADS[name].with_(**kw)
    w = make_workload(spec, device="cpu")
    mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, *_args(w), *_outs(spec.B, spec.L), placement="cpu")
    mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, *_args(w), *_outs(spec.B, spec.L, diag=False))
    # sliced batches (contiguous leading slices), as the status test passes them
    mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, w.target[:1], [d[:1] for d in w.draft_list()],
                      w.model_ids, w.tokens[:1], w.temps[:1], *_outs(1, spec.L))


def test_statistics_pattern_passes(mds):
    N, K, V = 64, 4, 257
    target = torch.zeros(V, dtype=torch.bfloat16).view(1, 1, 1, V).expand(N, K, 2, V).contiguous()
    drafts = [torch.zeros(V, dtype=torch.bfloat16).view(1, 1, V).expand(N, 1, V).contiguous() for _ in range(K)]
    tokens = torch.zeros(N, K, 1, dtype=torch.int32)
    temps = torch.ones(1, 1 + K).expand(N, -1).contiguous()
    mds.check_buffers(K, 1, V, "bf16", target, drafts, [0, 0, 1, 1], tokens, temps, *_outs(N, 1, diag=False))


def test_bad_buffers_are_rejected(mds):
    from synth import WORKLOADS, make_workload
    spec = WORKLOADS["llama2-32k"].with_(B=3, V=500)
    w = make_workload(spec, device="cpu")
    K, L, V = spec.K, spec.L, spec.V
    good = list(_args(w)) + list(_outs(spec.B, L))

    def expect(code, args, **kw):
        with pytest.raises(mds.MdsError) as e:
            mds.check_buffers(kw.get("K", K), L, kw.get("V", V), kw.get("dtype", spec.dtype), *args,
                              placement=kw.get("placement"))
        assert e.value.code == code

    expect(mds.MDS_ESHAPE, good, V=V + 1)                                   # vocabulary mismatch
    bad = list(good)
    bad[3] = w.tokens[:, :, :-1].contiguous()                               # tokens [B][K][L-1]
    expect(mds.MDS_ESHAPE, bad)
    expect(mds.MDS_EINVAL, good, dtype="f32")                               # bf16 logits, f32 declared
    bad = list(good)
    bad[0] = w.target.transpose(0, 1)                                       # non-contiguous (and reshaped)
    expect(mds.MDS_ESHAPE, bad)
    bad = list(good)
    bad[0] = torch.empty_strided(tuple(w.target.shape), (1,) * 4, dtype=w.target.dtype)  # right shape, wrong layout
    expect(mds.MDS_EINVAL, bad)
    bad = list(good)
    bad[2] = w.model_ids[:-1]                                               # K - 1 model ids
    expect(mds.MDS_EINVAL, bad)
    bad = list(good)
    bad[4] = w.temps.double()                                               # float64 temperatures
    expect(mds.MDS_EINVAL, bad)
    expect(mds.MDS_EINVAL, good, placement="cuda")                          # host tensors to the device entry


class _OnDevice:
    """A host tensor that reports a CUDA placement (shape, type and layout are
    the tensor's): stands in for a tensor on another GPU without needing one."""

    def __init__(self, t, index):
        self._t = t
        self.device = torch.device("cuda", index)

    shape = property(lambda self: self._t.shape)
    dtype = property(lambda self: self._t.dtype)

    def dim(self):
        return self._t.dim()

    def is_contiguous(self):
        return self._t.is_contiguous()


def test_tensors_on_another_device_are_rejected(mds):
    from synth import WORKLOADS, make_workload
    spec = WORKLOADS["tiny"].with_(B=2, V=64)
    w = make_workload(spec, device="cpu")
    on = lambda t, i: _OnDevice(t, i)  # noqa: E731
    outs = _outs(spec.B, spec.L)
    args = [on(w.target, 0), [on(d, 0) for d in w.draft_list()], w.model_ids, on(w.tokens, 0), on(w.temps, 0)]
    good_outs = [on(outs[0], 0), on(outs[1], 0), on(outs[2], 0)]
    mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, *args, *good_outs, placement="cuda", device=0)
    for i in range(len(good_outs)):
        bad = list(good_outs)
        bad[i] = on(outs[i], 1)
        with pytest.raises(mds.MdsError) as e:
            mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, *args, *bad, placement="cuda", device=0)
        assert e.value.code == mds.MDS_EINVAL
    bad_args = list(args)
    bad_args[0] = on(w.target, 1)
    with pytest.raises(mds.MdsError) as e:
        mds.check_buffers(spec.K, spec.L, spec.V, spec.dtype, *bad_args, *good_outs, placement="cuda", device=0)
    assert e.value.code == mds.MDS_EINVAL
