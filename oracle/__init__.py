"""CPU oracle for EmTrackMichelId hit identification (arXiv:2009.04509, Sec. 2.1-2.2).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline leg may import this package; the library never does.  It wraps
``oracle.c`` (plain C, fp32 patch cut, double-precision network) through
ctypes.  It shares no code with the CUDA library; the only thing both sides
share is the seeded input generator, which contains none of the method's
arithmetic.

``build()`` compiles ``liboracle.so`` next to this file with gcc; the other
functions build it on first use.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

PATCH, DOWNSAMPLE = 48, 6
EMTK_DIMS = dict(P=48, R=5, F=48, N1=128, N2=32, NC=3)


def build(force: bool = False, extra_flags: tuple = (), out: str | None = None) -> str:
    """Compile the oracle to a shared library; returns its path.  ``extra_flags``
    and ``out`` let a test build a variant (e.g. with a planted mistake) under
    another name without touching the real one."""
    target = out or _LIB
    if not force and not extra_flags and os.path.exists(target) and \
            os.path.getmtime(target) >= os.path.getmtime(_SRC):
        return target
    cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           *extra_flags, _SRC, "-o", target + ".tmp", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(target + ".tmp", target)
    return target


class _Dims(ctypes.Structure):
    _fields_ = [(k, ctypes.c_int) for k in ("P", "R", "F", "N1", "N2", "NC")]


def _bind(path: str):
    lib = ctypes.CDLL(path)
    f32p = ctypes.POINTER(ctypes.c_float)
    f64p = ctypes.POINTER(ctypes.c_double)
    i32p = ctypes.POINTER(ctypes.c_int32)
    lib.or_extract_patches.argtypes = [f32p, ctypes.c_int, ctypes.c_int, ctypes.c_long, i32p,
                                       ctypes.c_long, ctypes.c_int, ctypes.c_int, f32p]
    lib.or_extract_patches.restype = ctypes.c_int
    lib.or_forward.argtypes = [ctypes.POINTER(_Dims), f32p, ctypes.c_long] + [f32p] * 10 + \
        [ctypes.c_int, f64p, f64p]
    lib.or_forward.restype = ctypes.c_int
    lib.or_conv_relu.argtypes = [f64p, ctypes.c_int, f64p, f64p, ctypes.c_int, ctypes.c_int, f64p]
    lib.or_dense.argtypes = [f64p, ctypes.c_long, f32p, f32p, ctypes.c_int, ctypes.c_int, f64p]
    lib.or_heads.argtypes = [f64p, ctypes.c_int, ctypes.c_double, f64p]
    lib.or_round_bf16.argtypes = [f32p, ctypes.POINTER(ctypes.c_uint16), ctypes.c_long]
    lib.or_round_fp16.argtypes = [f32p, f32p, ctypes.c_long]
    lib.or_round_e4m3.argtypes = [f32p, f32p, ctypes.c_long]
    lib.or_set_fp8_scales.argtypes = [ctypes.c_double, ctypes.c_double]
    lib.or_find_hits.argtypes = [f32p, ctypes.c_int, ctypes.c_int, ctypes.c_long, ctypes.c_float, ctypes.c_long,
                                 i32p, i32p, i32p, i32p, f32p, f64p]
    lib.or_find_hits.restype = ctypes.c_long
    lib.or_set_threads.argtypes = [ctypes.c_int]
    lib.or_max_threads.restype = ctypes.c_int
    return lib


def load(path: str | None = None):
    """The ctypes handle of the oracle (a variant when ``path`` is given)."""
    global _lib
    if path is not None:
        return _bind(path)
    with _lock:
        if _lib is None:
            _lib = _bind(build())
        return _lib


def _p(a, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def extract_patches(adc, nticks, hits, psize: int = PATCH, ds: int = DOWNSAMPLE, lib=None):
    """Sec. 2.1 patch cut.  ``adc`` [nwires][ld] float32 (first ``nticks``
    columns are data), ``hits`` [n][2] int32 (wire, peak tick).  Returns
    [n][psize][psize] float32."""
    lib = lib or load()
    adc = _c(adc, np.float32)
    hits = _c(hits, np.int32).reshape(-1, 2)
    out = np.zeros((hits.shape[0], psize, psize), np.float32)
    rc = lib.or_extract_patches(_p(adc, ctypes.c_float), adc.shape[0], int(nticks), adc.shape[1],
                                _p(hits, ctypes.c_int32), hits.shape[0], psize, ds,
                                _p(out, ctypes.c_float))
    if rc != 0:
        raise ValueError(f"or_extract_patches failed ({rc})")
    return out


_WKEYS = ("conv_w", "conv_b", "fc1_w", "fc1_b", "fc2_w", "fc2_b", "cls_w", "cls_b", "mic_w", "mic_b")


_EMULATE = {None: 0, "bf16": 1, "fp16": 2, "fp8": 3}


def forward(patches, weights: dict, dims: dict | None = None, emulate: str | None = None,
            threads: int | None = None, lib=None, fp8_scales: tuple = (1.0, 1.0)):
    """Sec. 2.2 network on [n][P][P] float32 patches.  Returns (logits, scores),
    each [n][NC+1] float64: softmax classes (track, em, none) then Michel.
    ``emulate`` = "bf16" or "fp16" rounds the operands of the conv and of
    dense-1 to that format first (a diagnostic reference for 16-bit paths);
    "fp8" rounds the conv operands to bf16 and the dense-1 operands to e4m3,
    as e4m3(a * s_a) / s_a and e4m3(w * s_w) / s_w with (s_a, s_w) =
    ``fp8_scales``."""
    lib = lib or load()
    lib.or_set_fp8_scales(float(fp8_scales[0]), float(fp8_scales[1]))
    d = dict(EMTK_DIMS if dims is None else dims)
    patches = _c(patches, np.float32).reshape(-1, d["P"], d["P"])
    n = patches.shape[0]
    ws = [_c(weights[k], np.float32) for k in _WKEYS]
    logits = np.zeros((n, d["NC"] + 1), np.float64)
    scores = np.zeros((n, d["NC"] + 1), np.float64)
    if threads is not None:
        lib.or_set_threads(int(threads))
    rc = lib.or_forward(ctypes.byref(_Dims(**d)), _p(patches, ctypes.c_float), n,
                        *[_p(w, ctypes.c_float) for w in ws], _EMULATE[emulate],
                        _p(logits, ctypes.c_double), _p(scores, ctypes.c_double))
    if rc != 0:
        raise ValueError(f"or_forward failed ({rc})")
    return logits, scores


def conv_relu(img, w, b, lib=None):
    """One conv+ReLU on a single image: img [P][P], w [R][R][F] (or [R][R][1][F]),
    b [F] -> [Q][Q][F] float64."""
    lib = lib or load()
    img = _c(img, np.float64)
    P = img.shape[0]
    w = _c(w, np.float64)
    R, F = w.shape[0], w.shape[-1]
    w = w.reshape(R, R, F)
    b = _c(b, np.float64)
    Q = P - R + 1
    out = np.zeros((Q, Q, F), np.float64)
    lib.or_conv_relu(_p(img, ctypes.c_double), P, _p(w, ctypes.c_double), _p(b, ctypes.c_double),
                     R, F, _p(out, ctypes.c_double))
    return out


def dense(x, W, b, relu: bool, lib=None):
    """y = x W + b (ReLU optional); x [K] float64, W [K][N] float32, b [N] float32."""
    lib = lib or load()
    x = _c(x, np.float64)
    W = _c(W, np.float32)
    b = _c(b, np.float32)
    y = np.zeros(W.shape[1], np.float64)
    lib.or_dense(_p(x, ctypes.c_double), W.shape[0], _p(W, ctypes.c_float), _p(b, ctypes.c_float),
                 W.shape[1], int(relu), _p(y, ctypes.c_double))
    return y


def heads(z, zm, lib=None):
    """Softmax over the class logits ``z`` and sigmoid of ``zm``."""
    lib = lib or load()
    z = _c(z, np.float64)
    out = np.zeros(z.size + 1, np.float64)
    lib.or_heads(_p(z, ctypes.c_double), z.size, float(zm), _p(out, ctypes.c_double))
    return out


def round_bf16(x, lib=None):
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bits."""
    lib = lib or load()
    x = _c(x, np.float32)
    out = np.zeros(x.shape, np.uint16)
    lib.or_round_bf16(_p(x, ctypes.c_float), _p(out, ctypes.c_uint16), x.size)
    return out


def round_fp16(x, lib=None):
    """Round float32 values to IEEE binary16 (nearest, ties to even); returns float32."""
    lib = lib or load()
    x = _c(x, np.float32)
    out = np.zeros(x.shape, np.float32)
    lib.or_round_fp16(_p(x, ctypes.c_float), _p(out, ctypes.c_float), x.size)
    return out


def round_e4m3(x, lib=None):
    """Round float32 values to FP8 E4M3 (nearest, ties to even, saturating at
    +-448); returns float32."""
    lib = lib or load()
    x = _c(x, np.float32)
    out = np.zeros(x.shape, np.float32)
    lib.or_round_e4m3(_p(x, ctypes.c_float), _p(out, ctypes.c_float), x.size)
    return out


HIT_FIELDS = ("wire", "tick", "start", "end", "peak", "charge")


def find_hits(adc, nticks, threshold, lib=None) -> dict:
    """Hit finding of Sec. 2.1.  The paper gives no algorithm (only that hits
    are found on each wire's waveform and carry a time and a charge); the
    plainest reading: per wire, each maximal run of ticks with adc > threshold
    is one hit at the run's largest value (earliest on ties).  ``adc`` [nwires][ld] float32, first ``nticks``
    columns are data.  Returns a dict of arrays (wire, tick, start, end: int32;
    peak: float32; charge: float64), ordered by wire then start tick."""
    lib = lib or load()
    adc = _c(adc, np.float32)
    nw, ld = adc.shape
    args = (_p(adc, ctypes.c_float), nw, int(nticks), ld, ctypes.c_float(threshold))

    def arrays(n):
        return dict(wire=np.zeros(n, np.int32), tick=np.zeros(n, np.int32), start=np.zeros(n, np.int32),
                    end=np.zeros(n, np.int32), peak=np.zeros(n, np.float32), charge=np.zeros(n, np.float64))

    def call(a, cap):
        return lib.or_find_hits(*args, cap, _p(a["wire"], ctypes.c_int32), _p(a["tick"], ctypes.c_int32),
                                _p(a["start"], ctypes.c_int32), _p(a["end"], ctypes.c_int32),
                                _p(a["peak"], ctypes.c_float), _p(a["charge"], ctypes.c_double))

    n = call(arrays(1), 0)
    if n < 0:
        raise ValueError("or_find_hits: invalid argument")
    out = arrays(n)
    if call(out, n) != n:
        raise RuntimeError("or_find_hits: count changed between calls")
    return out


def max_threads(lib=None) -> int:
    return int((lib or load()).or_max_threads())


def set_threads(n: int, lib=None) -> None:
    (lib or load()).or_set_threads(int(n))
