"""Parity on the full 18-plane event, every hit (Sec. 2.1 patch cut and
Sec. 2.2 network): the benchmark's workload (6 APAs, planes of 800/800/960
wires x 6000 ticks, 60,000 hits) in its launch configuration, one
emtk_infer_batch over all planes, against the CPU oracle on all 60,000 hits.

References: the fp64 oracle (the definition), and for the reduced-precision
paths the oracle that rounds the same operands at the same points (patch,
conv weights, post-ReLU activations and dense-1 weights to bf16 / fp16, or
the dense-1 operands to e4m3 with the same power-of-two scales).  Bars:

* every path: finite scores, softmax rows summing to 1, scores in [0, 1];
* fp32 and tf32 (the fp32-accuracy paths): max |score - fp64| <= 1e-3 on
  every hit, and every logit within TOL_LOGIT_FP32 (1 + |z|) of the fp64
  logit;
* bf16 / fp16: argmax agreement with fp64 >= 99.5% over all 60,000 hits;
  max |score - emulation| <= 2e-2 on every hit; every logit within
  TOL_LOGIT_16 (1 + |z|) of the emulation's;
* fp8: max |score - emulation| <= 2e-2 and argmax agreement with the
  emulation >= 99.5%, with fp64 >= 95%; logits within TOL_LOGIT_8 (1 + |z|)
  of the emulation's.

Why the 16-bit score bar is taken against the emulation on raw ADC: the
synthetic network saturates (logits up to ~200, 74% of hits score above
0.99), and rounding the operands to 16 bits moves a near-tie hit's score by
more than 2e-2 in any implementation (measured on this event against
fp64: up to 0.175 for bf16, 0.026 for fp16, with argmax agreement 99.8% and
99.98%).

The logit bars.  The kernel and the emulation differ in the order and
precision of the sums (fp32 tensor-core or CUDA-core accumulation over
92,928 dense-1 terms, against fp64) and, in the reduced-precision paths, in
activations that the kernel's fp32 conv sum and the oracle's fp64 one round
to different neighbours (one bf16 / fp16 step is 2^-8 / 2^-11 of the value,
one e4m3 step 2^-3: a few such flips per hit move a logit by 1e-3 to 1e-1).
The bars sit 3-5x above the largest error measured over these 60,000 hits
(relative to 1 + |z|): fp32 3.7e-4 against fp64; bf16 6.8e-3, fp16 6.4e-3
and fp8 2.9e-2 against their emulations.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2009_04509_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL_FP32 = 1e-3
TOL_LOGIT_FP32 = 2e-3
TOL_16 = 2e-2
TOL_LOGIT_16 = 2e-2
TOL_LOGIT_8 = 8e-2
ARGMAX_MIN = 0.995
ARGMAX_FP8_FP64 = 0.95


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    oracle.build()
    return m


@pytest.fixture(scope="module")
def event():
    """The event, the oracle's patches of all its hits and the fp64 network on them."""
    planes = synth.full_event(seed=0)
    w = synth.he_normal_weights(0)
    patches = np.concatenate([oracle.extract_patches(p.adc, p.nticks, p.hits) for p in planes])
    lo, sc = oracle.forward(patches, w)
    return dict(planes=planes, weights=w, patches=patches, fp64=(lo, sc), emu={})


def emulation(event, mode):
    if mode not in event["emu"]:
        scales = (1.0, 1.0)
        if mode == "fp8":
            m = float(np.abs(event["weights"]["fc1_w"]).max())
            k = math.floor(math.log2(448.0 / m))
            while m * 2.0 ** (k + 1) <= 448.0:
                k += 1
            while m * 2.0 ** k > 448.0:
                k -= 1
            scales = (2.0 ** -4, 2.0 ** k)
        event["emu"][mode] = oracle.forward(event["patches"], event["weights"], emulate=mode, fp8_scales=scales)
    return event["emu"][mode]


def run_event(emtk, event, prec):
    planes = event["planes"]
    ctx = emtk.emtk_create(event["weights"], precision=prec, debug_logits=True)
    try:
        items, outs = [], []
        for p in planes:
            s = torch.full((p.nhits, 8), float("nan"), device="cuda")
            items.append((torch.from_numpy(p.adc).cuda(), p.nticks, torch.from_numpy(p.hits).cuda(), s))
            outs.append(s)
        emtk.emtk_infer_batch(ctx, items)
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    finally:
        emtk.emtk_destroy(ctx)
    got = np.concatenate([s.cpu().numpy().astype(np.float64) for s in outs])
    assert got.shape == (60000, 8)
    s = got[:, :4]
    assert np.all(np.isfinite(got))
    assert np.all(np.abs(s[:, :3].sum(1) - 1.0) <= 1e-5)
    assert np.all((s >= 0.0) & (s <= 1.0))
    return got[:, :4], got[:, 4:]


def logit_err(z, ref):
    """Largest |z - ref| / (1 + |ref|) over all hits and logits."""
    return float((np.abs(z - ref) / (1.0 + np.abs(ref))).max())


@pytest.mark.parametrize("prec", ["fp32", "tf32"])
def test_full_event_fp32_every_hit(emtk, event, prec):
    """The fp32 bar for both fp32-accuracy paths: CUDA-core fp32 and the
    tensor-core split-fp16 path (EMTK_TF32)."""
    s, z = run_event(emtk, event, prec)
    lo, ref = event["fp64"]
    d = np.abs(s - ref)
    assert d.max() <= TOL_FP32, f"max |score - fp64| = {d.max():.3g} at hit {np.unravel_index(d.argmax(), d.shape)}"
    assert logit_err(z, lo) <= TOL_LOGIT_FP32


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
def test_full_event_16bit_every_hit(emtk, event, prec):
    s, z = run_event(emtk, event, prec)
    lo, ref = event["fp64"]
    lo_e, emu = emulation(event, prec)
    agree = (s[:, :3].argmax(1) == ref[:, :3].argmax(1)).mean()
    d = np.abs(s - emu)
    msg = (f"{prec}: argmax vs fp64 {agree:.5f}, max |score - emulation| {d.max():.3g}, "
           f"logit error vs emulation {logit_err(z, lo_e):.3g}, max |score - fp64| {np.abs(s - ref).max():.3g}")
    assert agree >= ARGMAX_MIN, msg
    assert d.max() <= TOL_16, msg
    assert logit_err(z, lo_e) <= TOL_LOGIT_16, msg


def test_full_event_fp8_every_hit(emtk, event):
    s, z = run_event(emtk, event, "fp8")
    lo, ref = event["fp64"]
    lo_e, emu = emulation(event, "fp8")
    d = np.abs(s - emu)
    a_emu = (s[:, :3].argmax(1) == emu[:, :3].argmax(1)).mean()
    a_ref = (s[:, :3].argmax(1) == ref[:, :3].argmax(1)).mean()
    msg = (f"fp8: max |score - emulation| {d.max():.3g}, argmax vs emulation {a_emu:.5f}, vs fp64 {a_ref:.5f}, "
           f"logit error vs emulation {logit_err(z, lo_e):.3g}")
    assert d.max() <= TOL_16, msg
    assert a_emu >= ARGMAX_MIN, msg
    assert a_ref >= ARGMAX_FP8_FP64, msg
    assert logit_err(z, lo_e) <= TOL_LOGIT_8, msg


def test_full_event_patch_cut_bit_exact(emtk, event):
    """The patch cut of every hit of every full-size plane, fp32 and bf16."""
    ctx = emtk.emtk_create(event["weights"], precision="bf16")
    try:
        k = 0
        for p in event["planes"]:
            adc, hits = torch.from_numpy(p.adc).cuda(), torch.from_numpy(p.hits).cuda()
            want = event["patches"][k:k + p.nhits]
            k += p.nhits
            f32 = torch.zeros((p.nhits, 48, 48), dtype=torch.float32, device="cuda")
            b16 = torch.zeros((p.nhits, 48, 48), dtype=torch.int16, device="cuda")
            emtk.emtk_extract_patches(ctx, adc, p.nticks, hits, f32, "f32")
            emtk.emtk_extract_patches(ctx, adc, p.nticks, hits, b16, "bf16")
            assert emtk.emtk_check(ctx) == emtk.EMTK_OK
            assert np.array_equal(f32.cpu().numpy().view(np.uint32), want.view(np.uint32))
            assert np.array_equal(b16.cpu().numpy().view(np.uint16), oracle.round_bf16(want))
    finally:
        emtk.emtk_destroy(ctx)


def test_launch_counts(emtk, event):
    """The library's launch count is the number of its kernels launched: a
    full-event call is four (tile marks, the touched image tiles with the window
    descriptors, the network, the head), a small single-plane call three (the
    whole-plane images with the descriptors, the network, the head), and a
    hit-finding call two (find, place)."""
    planes = event["planes"]
    ctx = emtk.emtk_create(event["weights"], precision="bf16")
    try:
        items = [(torch.from_numpy(p.adc).cuda(), p.nticks, torch.from_numpy(p.hits).cuda(),
                  torch.empty((p.nhits, 4), device="cuda")) for p in planes]
        base = emtk.emtk_get_stats(ctx)["launches"]
        emtk.emtk_infer_batch(ctx, items)
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        assert emtk.emtk_get_stats(ctx)["launches"] - base == 4
        adc, nticks, hits, _ = items[2]
        small = torch.empty((256, 4), device="cuda")
        base = emtk.emtk_get_stats(ctx)["launches"]
        emtk.emtk_infer(ctx, adc, nticks, hits[:256], small)
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        assert emtk.emtk_get_stats(ctx)["launches"] - base == 3
        cap = 65536
        req = [(adc, nticks, 15.0, torch.empty((cap, 2), dtype=torch.int32, device="cuda"), None)]
        base = emtk.emtk_get_stats(ctx)["launches"]
        emtk.emtk_find_hits(ctx, req)
        assert emtk.emtk_get_stats(ctx)["launches"] - base == 2
    finally:
        emtk.emtk_destroy(ctx)
