"""The allocation-free patch cut, emtk_extract_patches_static.

It exists for callers that cannot allocate device memory (their memory is
owned by another allocator or fixed at start-up, or they must avoid the
synchronisation an allocation can cause), so it takes no context and keeps
its scratch in a fixed array inside the library.  This file is collected last
on purpose: if it fails, a run that stops at the first failure has already
run every other test.  It passes alone in a fresh process too.
"""
import ctypes

import numpy as np
import pytest

import oracle
from paper_2009_04509_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    oracle.build()
    return m


def _static_call(m, adc, nticks, hits, out, fmt):
    """Straight through the C ABI with ctypes."""
    lib = m.load_library()
    return lib.emtk_extract_patches_static(
        ctypes.c_void_p(adc.data_ptr()), ctypes.c_int32(adc.shape[0]), ctypes.c_int32(nticks),
        ctypes.c_int64(adc.shape[1]), ctypes.c_void_p(hits.data_ptr()), ctypes.c_int32(hits.shape[0]),
        ctypes.c_void_p(out.data_ptr()), ctypes.c_int(m.PATCH_FORMATS[fmt]),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _want(plane, fmt):
    """The oracle's patch cut, in the output format (16-bit: round to nearest even)."""
    p = oracle.extract_patches(plane.adc, plane.nticks, plane.hits)
    return p.view(np.uint32) if fmt == "f32" else oracle.round_bf16(p)


@pytest.mark.parametrize("fmt", ["f32", "bf16"])
def test_static_patch_cut_matches_context_call(emtk, fmt):
    """Two calls in a row (a full-size 960-wire plane, then a smaller ragged
    one) give the oracle's patches bit for bit, and the same patches as the
    existing context-based entry point; the device's free memory does not
    change across the calls."""
    dev = torch.device("cuda:0")
    big = synth.full_event(seed=3, n_apa=1)[2]                 # 960 x 6000
    small = synth.single_plane(seed=4, nwires=37, nhits=300, nticks=1996)   # 1996 % 6 != 0
    ctx = emtk.emtk_create(synth.he_normal_weights(0), precision="bf16")
    try:
        bufs = []
        for plane in (big, small):
            adc = torch.from_numpy(plane.adc).to(dev)
            hits = torch.from_numpy(plane.hits).to(dev)
            dt = torch.float32 if fmt == "f32" else torch.int16
            got = torch.full((plane.nhits, 48, 48), -1, dtype=dt, device=dev)
            want = torch.zeros((plane.nhits, 48, 48), dtype=dt, device=dev)
            bufs.append((plane, adc, hits, got, want))
        # a first call loads the library's module holding the fixed array (the CUDA
        # runtime loads modules lazily) and looks up the array's address; it is
        # the calls after it that must leave the device's free memory unchanged
        plane, adc, hits, got, _ = bufs[1]
        assert _static_call(emtk, adc, plane.nticks, hits, got, fmt) == emtk.EMTK_OK
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        for plane, adc, hits, got, _ in bufs:
            assert _static_call(emtk, adc, plane.nticks, hits, got, fmt) == emtk.EMTK_OK
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0    # nothing was allocated on the device
        for plane, adc, hits, got, want in bufs:
            emtk.emtk_extract_patches(ctx, adc, plane.nticks, hits, want, fmt)
            torch.cuda.synchronize()
            assert torch.equal(got, want)      # the patch cut is exact: tolerance zero
            g = got.cpu().numpy()
            assert np.array_equal(g.view(np.uint32) if fmt == "f32" else g.view(np.uint16), _want(plane, fmt))
    finally:
        emtk.emtk_destroy(ctx)


def test_static_patch_cut_rejects_oversized_plane(emtk):
    dev = torch.device("cuda:0")
    limit = emtk.EMTK_STATIC_SCRATCH_BYTES
    nwires = limit // (1000 * 4) + 1                       # fp32 image of 1000 intervals per wire
    adc = torch.zeros((nwires, 6000), dtype=torch.float32, device=dev)
    hits = torch.zeros((1, 2), dtype=torch.int32, device=dev)
    out = torch.zeros((1, 48, 48), dtype=torch.float32, device=dev)
    assert _static_call(emtk, adc, 6000, hits, out, "f32") == emtk.EMTK_ERR_ARG
    # the same plane fits as a 16-bit image, which takes half the room
    out16 = torch.zeros((1, 48, 48), dtype=torch.int16, device=dev)
    assert _static_call(emtk, adc, 6000, hits, out16, "bf16") == emtk.EMTK_OK
    torch.cuda.synchronize()
