"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every entry point include/emtk.h declares, and rejects bad arguments before
touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2009_04509_gb300 import emtk, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "emtk.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2009_04509_gb300 import build
    build.build()
    return emtk.load_library()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"EMTK_API\s+[\w\s\*]+?\b(emtk_\w+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    assert set(names) == set(emtk.EXPORTED)
    for n in ("emtk_create", "emtk_infer", "emtk_infer_batch", "emtk_extract_patches", "emtk_infer_patches"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_library_exports_nothing_else(lib):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", emtk.LIB_PATH], capture_output=True, text=True)
    if out.returncode != 0:
        pytest.skip("nm not available")
    syms = {l.split()[-1] for l in out.stdout.splitlines() if " T " in l}
    assert {s for s in syms if s.startswith("emtk_")} == set(declared_functions())


def test_status_strings(lib):
    for code in range(7):
        s = emtk.status_string(code)
        assert s and s != "unknown status"
    assert emtk.status_string(99) == "unknown status"


def test_default_options(lib):
    o = emtk.emtk_default_options()
    assert o.precision == emtk.EMTK_BF16 and o.max_hits == 65536 and o.debug_logits == 0
    assert o.wait_timeout_ns == 2_000_000_000 and o.debug_stall == 0 and o.profile == 0


ABI_STRUCTS = ("emtk_request", "emtk_options", "emtk_weights", "emtk_stats", "emtk_hitfind_request")


def test_struct_layouts_match_header(lib, tmp_path):
    """Every struct the binding mirrors has the header's size and field
    offsets, as a C compiler lays them out."""
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    lines = ["#include <stddef.h>", "#include <stdio.h>", '#include "emtk.h"', "int main(void) {"]
    for name in ABI_STRUCTS:
        lines.append(f'printf("{name} %zu\\n", sizeof({name}));')
        for f, _ in getattr(emtk, name)._fields_:
            lines.append(f'printf("{name}.{f} %zu\\n", offsetof({name}, {f}));')
    lines.append("return 0; }")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", inc, str(src), "-o", str(exe)], check=True)
    want = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True,
                                                   check=True).stdout.splitlines())
    for name in ABI_STRUCTS:
        st = getattr(emtk, name)
        assert ctypes.sizeof(st) == int(want[name]), name
        for f, _ in st._fields_:
            assert getattr(st, f).offset == int(want[f"{name}.{f}"]), f"{name}.{f}"


def test_argument_errors_without_device(lib):
    null = None
    assert lib.emtk_infer(null, None, 1, 1, 4, None, 0, None, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_infer_batch(null, None, 0, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_extract_patches(null, None, 1, 1, 4, None, 0, None, 0, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_infer_patches(null, None, 0, None, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_check(null, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_get_stats(null, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_destroy(null) == emtk.EMTK_OK
    assert lib.emtk_find_hits(null, None, 0, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_infer_batch_host(null, None, 0, None) == emtk.EMTK_ERR_ARG
    out = ctypes.c_void_p()
    assert lib.emtk_create(None, None, 0, ctypes.byref(out)) == emtk.EMTK_ERR_ARG and not out.value
    w = synth.he_normal_weights(0, dims=dict(P=6, R=3, F=2, N1=2, N2=2, NC=3))
    keep = {k: np.ascontiguousarray(v, np.float32) for k, v in w.items()}
    ws = emtk.emtk_weights(**{k: v.ctypes.data_as(ctypes.POINTER(ctypes.c_float)) for k, v in keep.items()})
    o = emtk.emtk_default_options()
    o.precision = 7
    assert lib.emtk_create(ctypes.byref(ws), ctypes.byref(o), 0, ctypes.byref(out)) == emtk.EMTK_ERR_ARG
    o = emtk.emtk_default_options()
    o.max_hits = 0
    assert lib.emtk_create(ctypes.byref(ws), ctypes.byref(o), 0, ctypes.byref(out)) == emtk.EMTK_ERR_ARG
    o = emtk.emtk_default_options()
    o.debug_stall = 2
    assert lib.emtk_create(ctypes.byref(ws), ctypes.byref(o), 0, ctypes.byref(out)) == emtk.EMTK_ERR_ARG
    assert lib.emtk_create(ctypes.byref(ws), None, -1, ctypes.byref(out)) == emtk.EMTK_ERR_ARG


def test_create_without_gpu_reports_cuda_error(lib):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(emtk.EmtkError) as e:
        emtk.emtk_create(synth.he_normal_weights(0), precision="bf16")
    assert e.value.status == emtk.EMTK_ERR_CUDA


def test_every_precision_is_accepted_then_needs_a_device(lib):
    """All five precisions are valid arguments (EMTK_TF32 included); without a
    GPU, creation fails at the device, not at the argument check."""
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    for prec in ("fp32", "tf32", "bf16", "fp16", "fp8"):
        with pytest.raises(emtk.EmtkError) as e:
            emtk.emtk_create(synth.he_normal_weights(0), precision=prec)
        assert e.value.status == emtk.EMTK_ERR_CUDA, prec


def test_fault_injection_hooks_without_device(lib):
    """The test hooks are host-only: they work without a device."""
    emtk.emtk_debug_fail_alloc(3)
    emtk.emtk_debug_fail_alloc(-1)
    assert emtk.emtk_debug_alloc_counts() == (0, 0)
    assert lib.emtk_debug_batcher_stall(None, 1) == emtk.EMTK_ERR_ARG


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        emtk.load_library(str(tmp_path / "libemtk.so"))


def test_batcher_argument_errors_without_device(lib):
    """The batcher rejects null handles and bad sizes before touching a device."""
    out = ctypes.c_void_p()
    assert lib.emtk_batcher_create(None, 1, 1024, 100, ctypes.byref(out)) == emtk.EMTK_ERR_ARG
    assert out.value is None
    t = ctypes.c_uint64(7)
    req = emtk.emtk_request()
    assert lib.emtk_batcher_submit(None, ctypes.byref(req), ctypes.byref(t)) == emtk.EMTK_ERR_ARG
    assert t.value == 0
    assert lib.emtk_batcher_wait(None, 1, 0) == emtk.EMTK_ERR_ARG
    assert lib.emtk_batcher_stats(None, None, None, None) == emtk.EMTK_ERR_ARG
    assert lib.emtk_batcher_destroy(None) == emtk.EMTK_OK
