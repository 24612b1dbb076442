"""Thin ctypes binding of libemtk.so (include/emtk.h), same names as the C ABI.

Only argument marshalling lives here: torch tensors are passed as device
pointers and the current torch stream as the CUDA stream.  Every step of the
hot path runs in the library's kernels.  If the library is not built, loading
fails loudly; there is no other implementation to fall back to.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libemtk.so")

EMTK_OK, EMTK_ERR_ARG, EMTK_ERR_ALIGN, EMTK_ERR_OOM, EMTK_ERR_CUDA, EMTK_ERR_TIMEOUT, EMTK_ERR_UNSUPPORTED = range(7)
EMTK_FP32, EMTK_TF32, EMTK_BF16, EMTK_FP16, EMTK_FP8 = 0, 1, 2, 3, 4
EMTK_PATCH_F32, EMTK_PATCH_BF16, EMTK_PATCH_F16 = 0, 1, 2
PRECISIONS = {"fp32": EMTK_FP32, "tf32": EMTK_TF32, "bf16": EMTK_BF16, "fp16": EMTK_FP16, "fp8": EMTK_FP8}
PATCH_FORMATS = {"f32": EMTK_PATCH_F32, "bf16": EMTK_PATCH_BF16, "fp16": EMTK_PATCH_F16}
KERNELS = ("intervals", "gather", "network", "head", "convert", "hitfind")

EXPORTED = ("emtk_default_options", "emtk_create", "emtk_destroy", "emtk_infer", "emtk_infer_batch",
            "emtk_extract_patches", "emtk_infer_patches", "emtk_check", "emtk_get_stats",
            "emtk_status_string", "emtk_extract_patches_static", "emtk_batcher_create", "emtk_batcher_submit",
            "emtk_batcher_wait", "emtk_batcher_stats", "emtk_batcher_destroy", "emtk_get_fp8_scales",
            "emtk_find_hits", "emtk_infer_batch_host", "emtk_debug_fail_alloc", "emtk_debug_alloc_counts",
            "emtk_debug_batcher_stall")
EMTK_STATIC_SCRATCH_BYTES = 4 << 20

_vp = ctypes.c_void_p
_fp = ctypes.POINTER(ctypes.c_float)


class emtk_weights(ctypes.Structure):
    _fields_ = [(k, _fp) for k in ("conv_w", "conv_b", "fc1_w", "fc1_b", "fc2_w", "fc2_b", "cls_w", "cls_b",
                                   "mic_w", "mic_b")]


class emtk_options(ctypes.Structure):
    _fields_ = [("precision", ctypes.c_int), ("max_hits", ctypes.c_int32), ("debug_logits", ctypes.c_int32),
                ("wait_timeout_ns", ctypes.c_int64), ("debug_stall", ctypes.c_int32), ("profile", ctypes.c_int32)]


class emtk_request(ctypes.Structure):
    _fields_ = [("d_adc", _vp), ("nwires", ctypes.c_int32), ("nticks", ctypes.c_int32), ("ld", ctypes.c_int64),
                ("d_hits", _vp), ("nhits", ctypes.c_int32), ("d_scores", _vp)]


class emtk_stats(ctypes.Structure):
    _fields_ = [("calls", ctypes.c_uint64), ("hits", ctypes.c_uint64), ("launches", ctypes.c_uint64),
                ("chunks", ctypes.c_uint64), ("batch_hist", ctypes.c_uint64 * 8),
                ("kernel_launches", ctypes.c_uint64 * 6), ("kernel_ms", ctypes.c_double * 6)]


class emtk_hitfind_request(ctypes.Structure):
    _fields_ = [("d_adc", _vp), ("nwires", ctypes.c_int32), ("nticks", ctypes.c_int32), ("ld", ctypes.c_int64),
                ("threshold", ctypes.c_float), ("capacity", ctypes.c_int32), ("d_hits", _vp), ("d_info", _vp),
                ("n_found", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class EmtkError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


_lib = None


def load_library(path: str | None = None):
    """The ctypes handle of libemtk.so; raises if it was not built."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is missing: build it with __graft_entry__.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(p)
    lib.emtk_default_options.argtypes = [ctypes.POINTER(emtk_options)]
    lib.emtk_default_options.restype = None
    lib.emtk_create.argtypes = [ctypes.POINTER(emtk_weights), ctypes.POINTER(emtk_options), ctypes.c_int,
                                ctypes.POINTER(_vp)]
    lib.emtk_destroy.argtypes = [_vp]
    lib.emtk_infer.argtypes = [_vp, _vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, _vp, ctypes.c_int32,
                               _vp, _vp]
    lib.emtk_infer_batch.argtypes = [_vp, ctypes.POINTER(emtk_request), ctypes.c_int32, _vp]
    lib.emtk_extract_patches.argtypes = [_vp, _vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, _vp,
                                         ctypes.c_int32, _vp, ctypes.c_int, _vp]
    lib.emtk_infer_patches.argtypes = [_vp, _vp, ctypes.c_int32, _vp, _vp]
    lib.emtk_check.argtypes = [_vp, _vp]
    lib.emtk_get_stats.argtypes = [_vp, ctypes.POINTER(emtk_stats)]
    lib.emtk_extract_patches_static.argtypes = [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, _vp,
                                                ctypes.c_int32, _vp, ctypes.c_int, _vp]
    lib.emtk_extract_patches_static.restype = ctypes.c_int
    lib.emtk_batcher_create.argtypes = [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, ctypes.POINTER(_vp)]
    lib.emtk_batcher_submit.argtypes = [_vp, ctypes.POINTER(emtk_request), ctypes.POINTER(ctypes.c_uint64)]
    lib.emtk_batcher_wait.argtypes = [_vp, ctypes.c_uint64, ctypes.c_int64]
    lib.emtk_batcher_stats.argtypes = [_vp, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64),
                                       ctypes.POINTER(ctypes.c_int64)]
    lib.emtk_batcher_destroy.argtypes = [_vp]
    lib.emtk_get_fp8_scales.argtypes = [_vp, _fp, _fp]
    lib.emtk_get_fp8_scales.restype = ctypes.c_int
    lib.emtk_find_hits.argtypes = [_vp, ctypes.POINTER(emtk_hitfind_request), ctypes.c_int32, _vp]
    lib.emtk_infer_batch_host.argtypes = [_vp, ctypes.POINTER(emtk_request), ctypes.c_int32, _vp]
    lib.emtk_infer_batch_host.restype = ctypes.c_int
    lib.emtk_find_hits.restype = ctypes.c_int
    lib.emtk_debug_fail_alloc.argtypes = [ctypes.c_int64]
    lib.emtk_debug_fail_alloc.restype = None
    lib.emtk_debug_alloc_counts.argtypes = [ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    lib.emtk_debug_alloc_counts.restype = None
    lib.emtk_debug_batcher_stall.argtypes = [_vp, ctypes.c_int32]
    lib.emtk_debug_batcher_stall.restype = ctypes.c_int
    for name in ("emtk_batcher_create", "emtk_batcher_submit", "emtk_batcher_wait", "emtk_batcher_stats",
                 "emtk_batcher_destroy"):
        getattr(lib, name).restype = ctypes.c_int
    lib.emtk_status_string.argtypes = [ctypes.c_int]
    lib.emtk_status_string.restype = ctypes.c_char_p
    for name in ("emtk_create", "emtk_destroy", "emtk_infer", "emtk_infer_batch", "emtk_extract_patches",
                 "emtk_infer_patches", "emtk_check", "emtk_get_stats"):
        getattr(lib, name).restype = ctypes.c_int
    if path is None:
        _lib = lib
    return lib


def status_string(status: int) -> str:
    return load_library().emtk_status_string(int(status)).decode()


def emtk_status_string(status: int) -> str:
    return status_string(status)


def _check(rc: int, what: str) -> int:
    if rc != EMTK_OK:
        raise EmtkError(rc, what)
    return rc


def _ptr(t) -> int:
    """Device pointer of a torch tensor (or a raw int)."""
    if t is None:
        return 0
    if isinstance(t, int):
        return t
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return t.data_ptr()


def _stream(stream) -> int:
    import torch
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def emtk_default_options() -> emtk_options:
    o = emtk_options()
    load_library().emtk_default_options(ctypes.byref(o))
    return o


def emtk_create(weights: dict, precision: str = "bf16", device: int = 0, max_hits: int | None = None,
                debug_logits: bool = False, wait_timeout_ns: int | None = None, debug_stall: bool = False,
                profile: bool = False):
    """Creates a context from host fp32 weights (a dict of numpy arrays in the
    layouts of include/emtk.h).  Returns an opaque handle (int)."""
    lib = load_library()
    keep = {k: np.ascontiguousarray(weights[k], dtype=np.float32) for k, _ in emtk_weights._fields_}
    w = emtk_weights(**{k: v.ctypes.data_as(_fp) for k, v in keep.items()})
    o = emtk_default_options()
    o.precision = PRECISIONS[precision] if isinstance(precision, str) else int(precision)
    if max_hits is not None:
        o.max_hits = int(max_hits)
    o.debug_logits = int(bool(debug_logits))
    if wait_timeout_ns is not None:
        o.wait_timeout_ns = int(wait_timeout_ns)
    o.debug_stall = int(bool(debug_stall))
    o.profile = int(bool(profile))
    h = _vp()
    _check(lib.emtk_create(ctypes.byref(w), ctypes.byref(o), int(device), ctypes.byref(h)), "emtk_create")
    return h.value


def emtk_destroy(ctx) -> None:
    _check(load_library().emtk_destroy(ctx), "emtk_destroy")


def emtk_infer(ctx, adc, nticks: int, hits, scores, stream=None) -> None:
    """adc: float32 [nwires][ld] CUDA tensor; hits: int32 [n][2]; scores:
    float32 [n][4] (or [n][8] with debug logits)."""
    nwires, ld = adc.shape
    _check(load_library().emtk_infer(ctx, _ptr(adc), int(nwires), int(nticks), int(ld), _ptr(hits),
                                     int(hits.shape[0]), _ptr(scores), _stream(stream)), "emtk_infer")


def make_requests(items) -> ctypes.Array:
    """items: iterable of (adc, nticks, hits, scores) tensors."""
    items = list(items)
    arr = (emtk_request * max(1, len(items)))()
    for i, (adc, nticks, hits, scores) in enumerate(items):
        arr[i] = emtk_request(_ptr(adc), int(adc.shape[0]), int(nticks), int(adc.shape[1]), _ptr(hits),
                              int(hits.shape[0]), _ptr(scores))
    return arr


def emtk_infer_batch(ctx, items, stream=None) -> None:
    items = list(items)
    reqs = make_requests(items)
    _check(load_library().emtk_infer_batch(ctx, reqs, len(items), _stream(stream)), "emtk_infer_batch")


def emtk_infer_batch_host(ctx, items, stream=None) -> None:
    """emtk_infer_batch with host (CPU) tensors: (adc, nticks, hits, scores) per
    request.  Returns once the work is enqueued; the scores are final when the
    stream has completed, and the tensors must stay alive until then."""
    items = list(items)
    reqs = make_requests(items)
    _check(load_library().emtk_infer_batch_host(ctx, reqs, len(items), _stream(stream)), "emtk_infer_batch_host")


def emtk_extract_patches(ctx, adc, nticks: int, hits, patches, fmt: str = "f32", stream=None) -> None:
    nwires, ld = adc.shape
    _check(load_library().emtk_extract_patches(ctx, _ptr(adc), int(nwires), int(nticks), int(ld), _ptr(hits),
                                               int(hits.shape[0]), _ptr(patches), PATCH_FORMATS[fmt],
                                               _stream(stream)), "emtk_extract_patches")


def emtk_extract_patches_static(adc, nticks: int, hits, patches, fmt: str = "f32", stream=None) -> None:
    """The patch cut without a context and without any device allocation, for
    callers that cannot allocate; its scratch is a fixed 4 MiB array in the
    library (see include/emtk.h for the size limit and the sharing rules)."""
    nwires, ld = adc.shape
    _check(load_library().emtk_extract_patches_static(_ptr(adc), int(nwires), int(nticks), int(ld), _ptr(hits),
                                                      int(hits.shape[0]), _ptr(patches), PATCH_FORMATS[fmt],
                                                      _stream(stream)), "emtk_extract_patches_static")


def emtk_infer_patches(ctx, patches, scores, stream=None) -> None:
    _check(load_library().emtk_infer_patches(ctx, _ptr(patches), int(patches.shape[0]), _ptr(scores),
                                             _stream(stream)), "emtk_infer_patches")


def emtk_check(ctx, stream=None) -> int:
    """Returns the status code (does not raise on EMTK_ERR_TIMEOUT)."""
    return int(load_library().emtk_check(ctx, _stream(stream)))


def emtk_get_stats(ctx) -> dict:
    s = emtk_stats()
    _check(load_library().emtk_get_stats(ctx, ctypes.byref(s)), "emtk_get_stats")
    return dict(calls=s.calls, hits=s.hits, launches=s.launches, chunks=s.chunks, batch_hist=list(s.batch_hist),
                kernel_launches=dict(zip(KERNELS, s.kernel_launches)), kernel_ms=dict(zip(KERNELS, s.kernel_ms)))


def emtk_find_hits(ctx, planes, stream=None) -> list:
    """Hit finding (see include/emtk.h) on several planes in one call.
    ``planes``: list of (adc [nwires][ld] float32 device tensor, nticks, threshold,
    hits [capacity][2] int32 device tensor, info [capacity][4] int32 device tensor
    or None).  info columns: start, end, then peak and charge as float32 bits
    (``info[:, 2:].view(torch.float32)``).  Returns the number of hits found per
    plane (which may exceed a plane's capacity); the call synchronises the stream."""
    reqs = (emtk_hitfind_request * max(1, len(planes)))()
    for i, (adc, nticks, thr, hits, info) in enumerate(planes):
        q = reqs[i]
        q.d_adc = _ptr(adc)
        q.nwires, q.ld = adc.shape
        q.nticks = int(nticks)
        q.threshold = float(thr)
        q.capacity = hits.shape[0]
        q.d_hits = _ptr(hits)
        q.d_info = _ptr(info) if info is not None else None
    _check(load_library().emtk_find_hits(ctx, reqs, len(planes), _stream(stream)), "emtk_find_hits")
    return [int(reqs[i].n_found) for i in range(len(planes))]


def emtk_get_fp8_scales(ctx) -> tuple:
    """(s_a, s_w): the dense-1 operand scales of an "fp8" context, (1, 1) otherwise."""
    a, w = ctypes.c_float(), ctypes.c_float()
    _check(load_library().emtk_get_fp8_scales(ctx, ctypes.byref(a), ctypes.byref(w)), "emtk_get_fp8_scales")
    return float(a.value), float(w.value)


# ------------------------------------------------------------------ batcher
def emtk_batcher_create(ctx, nstreams: int = 4, max_hits: int = 65536, max_delay_us: int = 200):
    """Request batcher over `ctx` (see include/emtk.h).  Returns a handle (int)."""
    out = _vp()
    _check(load_library().emtk_batcher_create(ctx, int(nstreams), int(max_hits), int(max_delay_us),
                                              ctypes.byref(out)), "emtk_batcher_create")
    return out.value


# (batcher, ticket) -> the request's tensors.  The batcher reads and writes them on its
# own streams after submit returns; holding them here until the ticket is waited for (or
# the batcher destroyed) keeps torch from freeing and reusing their memory meanwhile.
_batcher_refs = {}


def emtk_batcher_submit(b, adc, nticks: int, hits, scores) -> int:
    """Queues one request (a plane, its hits and its output); returns its ticket.  The tensors
    must stay unchanged until emtk_batcher_wait has returned for the ticket; this binding
    keeps them alive until then."""
    req = make_requests([(adc, nticks, hits, scores)])
    t = ctypes.c_uint64()
    _check(load_library().emtk_batcher_submit(b, req, ctypes.byref(t)), "emtk_batcher_submit")
    _batcher_refs[(b, t.value)] = (adc, hits, scores)
    return t.value


def emtk_batcher_wait(b, ticket: int, timeout_ms: int = -1) -> int:
    """Blocks until the ticket's scores are complete; returns the status (EMTK_ERR_TIMEOUT when
    timeout_ms ran out first, without consuming the ticket)."""
    rc = load_library().emtk_batcher_wait(b, int(ticket), int(timeout_ms))
    if rc != EMTK_ERR_TIMEOUT:  # the ticket is done with (or was never issued)
        _batcher_refs.pop((b, int(ticket)), None)
    return rc


def emtk_batcher_stats(b) -> dict:
    n = [ctypes.c_int64() for _ in range(3)]
    _check(load_library().emtk_batcher_stats(b, *[ctypes.byref(x) for x in n]), "emtk_batcher_stats")
    return dict(batches=n[0].value, requests=n[1].value, hits=n[2].value)


def emtk_batcher_destroy(b) -> None:
    _check(load_library().emtk_batcher_destroy(b), "emtk_batcher_destroy")
    for key in [k for k in _batcher_refs if k[0] == b]:
        del _batcher_refs[key]


# ------------------------------------------------------------- test hooks
def emtk_debug_fail_alloc(after: int) -> None:
    """The allocation after ``after`` more successful ones fails, once (< 0 disarms)."""
    load_library().emtk_debug_fail_alloc(int(after))


def emtk_debug_alloc_counts() -> tuple:
    """(device, pinned host) allocations of the library alive now."""
    d, h = ctypes.c_int64(), ctypes.c_int64()
    load_library().emtk_debug_alloc_counts(ctypes.byref(d), ctypes.byref(h))
    return d.value, h.value


def emtk_debug_batcher_stall(b, stall: bool) -> None:
    _check(load_library().emtk_debug_batcher_stall(b, int(bool(stall))), "emtk_debug_batcher_stall")
