"""Failure detection without faulting the GPU.

Every mbarrier wait in the tensor-core kernels is bounded by the context's
wait_timeout_ns.  The debug_stall knob makes the kernel wait once on a
barrier that nothing ever arrives at; the wait must run out, every CTA must
leave its loops, free its tensor memory and return, and emtk_check must
report EMTK_ERR_TIMEOUT.  The device stays usable: the next call on a normal
context gives correct scores.
"""
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


@pytest.mark.parametrize("prec", ["bf16", "tf32"])
def test_bounded_wait_reports_timeout_and_device_stays_usable(emtk, prec):
    """Both tensor-core kernels: the 16-bit one and the split-fp16 (tf32) one."""
    w = synth.he_normal_weights(0)
    x = synth.inference_patches(300, seed=21) * np.float32(0.05)
    xd = torch.from_numpy(x).cuda()
    scores = torch.zeros((300, 4), device="cuda")
    stalled = emtk.emtk_create(w, precision=prec, wait_timeout_ns=50_000_000, debug_stall=True)
    try:
        emtk.emtk_infer_patches(stalled, xd, scores)
        assert emtk.emtk_check(stalled) == emtk.EMTK_ERR_TIMEOUT
        assert emtk.emtk_check(stalled) == emtk.EMTK_OK   # the status word was cleared
    finally:
        emtk.emtk_destroy(stalled)
    ctx = emtk.emtk_create(w, precision="bf16")
    try:
        emtk.emtk_infer_patches(ctx, xd, scores)
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        got = scores.cpu().numpy().astype(np.float64)
    finally:
        emtk.emtk_destroy(ctx)
    _, emu = oracle.forward(x, w, emulate="bf16")
    assert np.abs(got - emu).max() <= 2e-2


def test_bounded_wait_large_launch(emtk):
    """A launch large enough that each tile's head waits for that tile's
    counter instead of the whole network kernel (8,192 patches): when the
    network kernel gives up, the head kernels see its status bit and return
    at once (no second timeout per tile), emtk_check reports EMTK_ERR_TIMEOUT
    and clears the status and the tile counters."""
    import time
    w = synth.he_normal_weights(0)
    n = 8192
    x = synth.inference_patches(n, seed=22) * np.float32(0.05)
    xd = torch.from_numpy(x).cuda()
    scores = torch.zeros((n, 4), device="cuda")
    stalled = emtk.emtk_create(w, precision="bf16", wait_timeout_ns=50_000_000, debug_stall=True)
    try:
        t0 = time.perf_counter()
        emtk.emtk_infer_patches(stalled, xd, scores)
        assert emtk.emtk_check(stalled) == emtk.EMTK_ERR_TIMEOUT
        assert time.perf_counter() - t0 < 5.0
        assert emtk.emtk_check(stalled) == emtk.EMTK_OK
    finally:
        emtk.emtk_destroy(stalled)
    ctx = emtk.emtk_create(w, precision="bf16")
    try:
        emtk.emtk_infer_patches(ctx, xd, scores)
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        got = scores.cpu().numpy().astype(np.float64)
    finally:
        emtk.emtk_destroy(ctx)
    idx = np.arange(0, n, 16)
    _, emu = oracle.forward(x[idx], w, emulate="bf16")
    assert np.abs(got[idx] - emu).max() <= 2e-2
