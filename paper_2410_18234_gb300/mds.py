"""ctypes binding of the verification library (C ABI in include/mds.h).

Argument marshalling only: every step of the verification runs in the CUDA
kernels of libmds.so.  PyTorch tensors serve as owners of device memory and
streams.  If the library is missing the import of this module fails loudly;
there is no fallback.

The module mirrors the C entry points under the same names (``mds_create``,
``mds_verify``, ``mds_verify_host``, ``mds_status``, ``mds_destroy``) and adds
a small ``Verifier`` convenience wrapper.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
# MDS_LIBRARY may name another build of the same library (the instrumented
# libmds_timers.so); the default is the in-tree libmds.so.
LIB_PATH = os.environ.get("MDS_LIBRARY") or os.path.join(_HERE, "_lib", "libmds.so")

MDS_SINGLE, MDS_IS, MDS_WIS, MDS_SPECTR, MDS_WIS0, MDS_WISSORT = 0, 1, 2, 3, 4, 5
SCHEMES = {"single": MDS_SINGLE, "IS": MDS_IS, "WIS": MDS_WIS, "SpecTr": MDS_SPECTR, "WIS0": MDS_WIS0,
           "WISsort": MDS_WISSORT}
MDS_F32, MDS_BF16 = 0, 1
DTYPES = {"f32": MDS_F32, "bf16": MDS_BF16}
TORCH_DTYPES = {MDS_F32: torch.float32, MDS_BF16: torch.bfloat16}

MDS_OK, MDS_EINVAL, MDS_ESHAPE, MDS_EVOCAB, MDS_ECUDA, MDS_EUNSUP = 0, -1, -2, -3, -4, -5
MDS_ST_NONFINITE, MDS_ST_BADTEMP, MDS_ST_ZERO_RESID, MDS_ST_TIMEOUT, MDS_ST_LP_CAP, MDS_ST_BADTOKEN = \
    1, 2, 4, 8, 16, 32
MDS_ST_OMEGA0 = 64
MDS_MAX_TOPK = 16
MDS_MAX_K = 16
MDS_MAX_OMEGA0 = 62
MDS_MAX_OMEGA0_CLUSTER = 30   # with a cluster size set (the per-sequence engine)

# every symbol include/mds.h declares
EXPORTS = ("mds_create", "mds_verify", "mds_verify_host", "mds_verify_noalloc", "mds_noalloc_status", "mds_status",
           "mds_cluster_size", "mds_phase_timers", "mds_debug_row_stats", "mds_debug_exp_count", "mds_debug_probs",
           "mds_error_string", "mds_destroy")


class MdsConfig(ctypes.Structure):
    _fields_ = [("max_B", ctypes.c_int), ("K", ctypes.c_int), ("L", ctypes.c_int), ("V", ctypes.c_int),
                ("dtype", ctypes.c_int), ("wis_s", ctypes.c_int), ("is_h", ctypes.c_float),
                ("cluster", ctypes.c_int), ("omega0", ctypes.c_int), ("acc_prob", ctypes.c_int),
                ("top_k", ctypes.c_int)]


class MdsError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        super().__init__(f"{where}: {error_string(code)} ({code})")


def load_library(path=LIB_PATH):
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with __graft_entry__.build() "
                          "(python -m paper_2410_18234_gb300.build)")
    lib = ctypes.CDLL(path)
    vp, i32p, f32p = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32), ctypes.c_void_p
    lib.mds_create.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(MdsConfig), ctypes.c_int]
    lib.mds_create.restype = ctypes.c_int
    verify_args = [vp, vp, ctypes.POINTER(vp), i32p, vp, vp, ctypes.c_int, ctypes.c_uint64, vp, vp, f32p,
                   ctypes.c_int, vp]
    lib.mds_verify.argtypes = verify_args
    lib.mds_verify.restype = ctypes.c_int
    lib.mds_verify_host.argtypes = verify_args
    lib.mds_verify_host.restype = ctypes.c_int
    lib.mds_verify_noalloc.argtypes = [ctypes.POINTER(MdsConfig), ctypes.c_int, vp, ctypes.POINTER(vp), i32p, vp, vp,
                                       ctypes.c_int, ctypes.c_uint64, vp, vp, f32p, ctypes.c_int, vp]
    lib.mds_verify_noalloc.restype = ctypes.c_int
    lib.mds_noalloc_status.argtypes = [ctypes.c_int, vp, ctypes.POINTER(ctypes.c_char_p)]
    lib.mds_noalloc_status.restype = ctypes.c_int
    lib.mds_status.argtypes = [vp, ctypes.POINTER(ctypes.c_char_p)]
    lib.mds_status.restype = ctypes.c_int
    lib.mds_cluster_size.argtypes = [vp]
    lib.mds_cluster_size.restype = ctypes.c_int
    lib.mds_phase_timers.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_uint64), ctypes.c_int]
    lib.mds_phase_timers.restype = ctypes.c_int
    lib.mds_debug_row_stats.argtypes = [vp, vp]
    lib.mds_debug_row_stats.restype = ctypes.c_int
    lib.mds_debug_exp_count.argtypes = [vp, vp]
    lib.mds_debug_exp_count.restype = ctypes.c_int
    lib.mds_debug_probs.argtypes = [vp, ctypes.c_int, ctypes.c_int, ctypes.c_float, ctypes.c_float, ctypes.c_float,
                                    vp, vp]
    lib.mds_debug_probs.restype = ctypes.c_int
    lib.mds_error_string.argtypes = [ctypes.c_int]
    lib.mds_error_string.restype = ctypes.c_char_p
    lib.mds_destroy.argtypes = [vp]
    lib.mds_destroy.restype = None
    return lib


_lib = load_library()


def error_string(code):
    return _lib.mds_error_string(int(code)).decode()


# ----------------------------------------------------------- C entry points


def mds_create(max_B, K, L, V, dtype="bf16", wis_s=5, is_h=0.25, cluster=0, device=0, omega0=0, acc_prob=0,
               top_k=0):
    cfg = MdsConfig(int(max_B), int(K), int(L), int(V), DTYPES[dtype] if isinstance(dtype, str) else int(dtype),
                    int(wis_s), float(is_h), int(cluster), int(omega0), int(acc_prob), int(top_k))
    h = ctypes.c_void_p()
    rc = _lib.mds_create(ctypes.byref(h), ctypes.byref(cfg), int(device))
    if rc != MDS_OK:
        raise MdsError(rc, "mds_create")
    return h


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else ctypes.c_void_p(0)


def _draft_ptrs(drafts, K):
    arr = (ctypes.c_void_p * K)()
    for k in range(K):
        arr[k] = drafts[k].data_ptr()
    return arr


def _ids(model_ids, K):
    arr = (ctypes.c_int32 * K)()
    for k in range(K):
        arr[k] = int(model_ids[k])
    return arr


def check_buffers(K, L, V, dtype, target, drafts, model_ids, tokens, temps, out_tokens, out_accept,
                  out_diag=None, placement=None, device=None):
    """Shapes, element types, contiguity and placement ("cuda", "cpu" or None
    to skip; with ``device``, the CUDA device index every tensor must be on)
    of one call's tensors.  The C ABI takes bare pointers and the sizes from
    its configuration, so a tensor of the wrong shape would be read or written
    out of bounds, and a tensor on another GPU would be dereferenced by a
    kernel running elsewhere: the binding rejects both first (MdsError with
    MDS_ESHAPE or MDS_EINVAL)."""
    st = TORCH_DTYPES[DTYPES[dtype] if isinstance(dtype, str) else int(dtype)]
    if len(model_ids) != K or len(drafts) < K:
        raise MdsError(MDS_EINVAL, f"{len(model_ids)} model ids and {len(drafts)} draft buffers for K = {K}")
    B = int(tokens.shape[0]) if tokens.dim() >= 1 else -1
    want = [("target", target, (B, K, L + 1, V), st), ("tokens", tokens, (B, K, L), torch.int32),
            ("temperatures", temps, (B, 1 + K), torch.float32),
            ("out_tokens", out_tokens, (B, L + 1), torch.int32), ("out_accept_len", out_accept, (B,), torch.int32)]
    want += [(f"draft_logits[{k}]", drafts[k], (B, L, V), st) for k in range(K)]
    if out_diag is not None:
        want.append(("out_diag", out_diag, (B, L + 1, 4), torch.float32))
    for name, t, shape, dt in want:
        if tuple(t.shape) != shape:
            raise MdsError(MDS_ESHAPE, f"{name} has shape {tuple(t.shape)}, expected {shape}")
        if t.dtype != dt:
            raise MdsError(MDS_EINVAL, f"{name} has type {t.dtype}, expected {dt}")
        if not t.is_contiguous():
            raise MdsError(MDS_EINVAL, f"{name} is not contiguous")
        if placement is not None and (t.device.type == "cuda") != (placement == "cuda"):
            raise MdsError(MDS_EINVAL, f"{name} is on {t.device}, expected {placement} memory")
        if device is not None and t.device.type == "cuda" and t.device.index != int(device):
            raise MdsError(MDS_EINVAL, f"{name} is on {t.device}, expected cuda:{int(device)}")


def mds_verify(ctx, target, drafts, model_ids, tokens, temps, scheme, seed, out_tokens, out_accept,
               out_diag=None, stream=None):
    """Device-buffer entry point.  ``drafts`` is a sequence of K device
    tensors (or a [K, B, L, V] tensor); ``stream`` a torch.cuda.Stream, a raw
    handle, or None for torch's current stream."""
    K = len(model_ids)
    B = int(tokens.shape[0])
    if stream is None:
        stream = torch.cuda.current_stream().cuda_stream
    elif isinstance(stream, torch.cuda.Stream):
        stream = stream.cuda_stream
    keep = _draft_ptrs(drafts, K)
    rc = _lib.mds_verify(ctx, _ptr(target), keep, _ids(model_ids, K), _ptr(tokens), _ptr(temps),
                         SCHEMES[scheme] if isinstance(scheme, str) else int(scheme), ctypes.c_uint64(int(seed)),
                         _ptr(out_tokens), _ptr(out_accept), _ptr(out_diag), B, ctypes.c_void_p(int(stream)))
    if rc != MDS_OK:
        raise MdsError(rc, "mds_verify")


def mds_verify_host(ctx, target, drafts, model_ids, tokens, temps, scheme, seed, out_tokens, out_accept,
                    out_diag=None, stream=None):
    """Host-buffer entry point: CPU tensors (pinned for speed); copies in and
    out happen inside the call, which returns after the stream synchronised."""
    K = len(model_ids)
    B = int(tokens.shape[0])
    if stream is None:
        stream = torch.cuda.current_stream().cuda_stream
    elif isinstance(stream, torch.cuda.Stream):
        stream = stream.cuda_stream
    keep = _draft_ptrs(drafts, K)
    rc = _lib.mds_verify_host(ctx, _ptr(target), keep, _ids(model_ids, K), _ptr(tokens), _ptr(temps),
                              SCHEMES[scheme] if isinstance(scheme, str) else int(scheme),
                              ctypes.c_uint64(int(seed)), _ptr(out_tokens), _ptr(out_accept), _ptr(out_diag), B,
                              ctypes.c_void_p(int(stream)))
    if rc != MDS_OK:
        raise MdsError(rc, "mds_verify_host")


def mds_verify_noalloc(max_B, K, L, V, target, drafts, model_ids, tokens, temps, scheme, seed, out_tokens,
                       out_accept, out_diag=None, stream=None, dtype="bf16", wis_s=5, is_h=0.25, cluster=0,
                       device=0, omega0=0, acc_prob=0, top_k=0):
    """Context-free entry point for callers that cannot allocate device
    memory (see include/mds.h): the configuration is passed directly and the
    kernel's scratch is a static device array inside the library."""
    check_buffers(int(K), int(L), int(V), dtype, target, drafts, model_ids, tokens, temps, out_tokens, out_accept,
                  out_diag, "cuda", device=int(device))
    cfg = MdsConfig(int(max_B), int(K), int(L), int(V), DTYPES[dtype] if isinstance(dtype, str) else int(dtype),
                    int(wis_s), float(is_h), int(cluster), int(omega0), int(acc_prob), int(top_k))
    Kn = len(model_ids)
    B = int(tokens.shape[0])
    if stream is None:
        stream = torch.cuda.current_stream(int(device)).cuda_stream
    elif isinstance(stream, torch.cuda.Stream):
        stream = stream.cuda_stream
    rc = _lib.mds_verify_noalloc(ctypes.byref(cfg), int(device), _ptr(target), _draft_ptrs(drafts, Kn),
                                 _ids(model_ids, Kn), _ptr(tokens), _ptr(temps),
                                 SCHEMES[scheme] if isinstance(scheme, str) else int(scheme),
                                 ctypes.c_uint64(int(seed)), _ptr(out_tokens), _ptr(out_accept), _ptr(out_diag), B,
                                 ctypes.c_void_p(int(stream)))
    if rc != MDS_OK:
        raise MdsError(rc, "mds_verify_noalloc")


def mds_noalloc_status(device=0, stream=None):
    """(bits, message) of the last mds_verify_noalloc call on `device`, read
    without allocating (see include/mds.h)."""
    if stream is None:
        stream = torch.cuda.current_stream(int(device)).cuda_stream
    elif isinstance(stream, torch.cuda.Stream):
        stream = stream.cuda_stream
    msg = ctypes.c_char_p()
    rc = _lib.mds_noalloc_status(int(device), ctypes.c_void_p(int(stream)), ctypes.byref(msg))
    if rc < 0:
        raise MdsError(rc, "mds_noalloc_status")
    return rc, (msg.value or b"").decode()


def mds_status(ctx):
    msg = ctypes.c_char_p()
    rc = _lib.mds_status(ctx, ctypes.byref(msg))
    if rc < 0:
        raise MdsError(rc, "mds_status")
    return rc, (msg.value or b"").decode()


def mds_cluster_size(ctx):
    return _lib.mds_cluster_size(ctx)


PHASES = ("kernel", "wait_full", "task_list", "task_stats", "task_resid", "task_full", "dec_stats",
          "dec_combine", "dec_stages", "dec_resid", "dec_full", "dec_bonus", "push", "sched_poll",
          "sched_empty", "dec_poll", "dec_plan", "dec_load", "dec_select", "dec_accept",
          "dec_walk", "list_a", "list_b", "list_c", "publish", "combine", "lp", "lp_calls", "tasks",
          "decisions")


def mds_phase_timers(device=0):
    """Phase counters of an instrumented build (None for the default build):
    a dict of SM cycles summed over CTAs per phase, and the task and decision
    counts; reading clears them."""
    buf = (ctypes.c_uint64 * 64)()
    rc = _lib.mds_phase_timers(int(device), buf, 64)
    if rc == MDS_EUNSUP:
        return None
    if rc < 0:
        raise MdsError(rc, "mds_phase_timers")
    return {name: int(buf[i]) for i, name in enumerate(PHASES[:rc])}


DEBUG_ROWS = 4   # MDS_DEBUG_ROWS


def mds_debug_row_stats(ctx, row_stats):
    """Have the context's later dataflow-engine calls write every visited
    row's statistics into row_stats (float32 CUDA tensor [max_B][L+1][4][4]:
    M, 1/Z, c, source), or stop with None.  Test export."""
    ptr = None if row_stats is None else ctypes.c_void_p(row_stats.data_ptr())
    rc = _lib.mds_debug_row_stats(ctx, ptr)
    if rc != MDS_OK:
        raise MdsError(rc, "mds_debug_row_stats")


def mds_debug_exp_count(ctx, counter):
    """Have the context's later IS calls add their quadrature exponentials to
    counter (int64 CUDA tensor of one element), or stop with None."""
    ptr = None if counter is None else ctypes.c_void_p(counter.data_ptr())
    rc = _lib.mds_debug_exp_count(ctx, ptr)
    if rc != MDS_OK:
        raise MdsError(rc, "mds_debug_exp_count")


def mds_debug_probs(row, M, invZ, c, out, stream=None):
    """The kernel's probability of every token of one logit row (CUDA tensor
    of V logits) under row statistics (M, 1/Z, c), into out (float32, V)."""
    if not (row.is_cuda and out.is_cuda and row.is_contiguous() and out.is_contiguous()):
        raise MdsError(MDS_EINVAL, "mds_debug_probs: contiguous CUDA tensors")
    if out.dtype != torch.float32 or out.numel() != row.numel():
        raise MdsError(MDS_EINVAL, "mds_debug_probs: out must be float32 of the row's length")
    dt = {torch.float32: MDS_F32, torch.bfloat16: MDS_BF16}.get(row.dtype)
    if dt is None:
        raise MdsError(MDS_EINVAL, "mds_debug_probs: logits must be float32 or bfloat16")
    if stream is None:
        stream = torch.cuda.current_stream(row.device)
    rc = _lib.mds_debug_probs(ctypes.c_void_p(row.data_ptr()), dt, int(row.numel()), float(M), float(invZ),
                              float(c), ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(stream.cuda_stream))
    if rc != MDS_OK:
        raise MdsError(rc, "mds_debug_probs")


def mds_destroy(ctx):
    if ctx:
        _lib.mds_destroy(ctx)


# ----------------------------------------------------------- convenience


class Verifier:
    """Owns one context; allocates outputs with torch on the context's device."""

    def __init__(self, max_B, K, L, V, dtype="bf16", wis_s=5, is_h=0.25, cluster=0, device=0, omega0=0,
                 acc_prob=0, top_k=0):
        self.max_B, self.K, self.L, self.V = int(max_B), int(K), int(L), int(V)
        self.dtype = dtype
        self.device = torch.device("cuda", device)
        self.ctx = mds_create(max_B, K, L, V, dtype, wis_s, is_h, cluster, device, omega0, acc_prob, top_k)

    def verify(self, target, drafts, model_ids, tokens, temps, scheme, seed, diag=False, out=None, stream=None):
        B = int(tokens.shape[0])
        if out is None:
            out_tokens = torch.empty(B, self.L + 1, dtype=torch.int32, device=self.device)
            out_accept = torch.empty(B, dtype=torch.int32, device=self.device)
            out_diag = torch.empty(B, self.L + 1, 4, dtype=torch.float32, device=self.device) if diag else None
        else:
            out_tokens, out_accept, out_diag = out
        check_buffers(self.K, self.L, self.V, self.dtype, target, drafts, model_ids, tokens, temps, out_tokens,
                      out_accept, out_diag, "cuda", device=self.device.index)
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        mds_verify(self.ctx, target, drafts, model_ids, tokens, temps, scheme, seed, out_tokens, out_accept,
                   out_diag, stream)
        return out_tokens, out_accept, out_diag

    def verify_host(self, target, drafts, model_ids, tokens, temps, scheme, seed, out=None, stream=None):
        B = int(tokens.shape[0])
        if out is None:
            out_tokens = torch.empty(B, self.L + 1, dtype=torch.int32).pin_memory()
            out_accept = torch.empty(B, dtype=torch.int32).pin_memory()
            out_diag = None
        else:
            out_tokens, out_accept, out_diag = out
        check_buffers(self.K, self.L, self.V, self.dtype, target, drafts, model_ids, tokens, temps, out_tokens,
                      out_accept, out_diag, "cpu")
        mds_verify_host(self.ctx, target, drafts, model_ids, tokens, temps, scheme, seed, out_tokens, out_accept,
                        out_diag, stream)
        return out_tokens, out_accept, out_diag

    def status(self):
        return mds_status(self.ctx)

    @property
    def cluster_size(self):
        return mds_cluster_size(self.ctx)

    def close(self):
        if self.ctx:
            mds_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
