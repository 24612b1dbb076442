"""emtk_infer_batch_host: the batch with host buffers (copies in on the
context's copy stream, two staging areas used in turn, scores copied back).
Its scores must be bit-identical to emtk_infer_batch on device copies of the
same inputs, also when several calls are in flight at once."""
import numpy as np
import pytest

from paper_2009_04509_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    return m


@pytest.fixture(scope="module")
def ctx(emtk):
    c = emtk.emtk_create(synth.he_normal_weights(0), precision="bf16")
    yield c
    emtk.emtk_destroy(c)


def device_scores(emtk, ctx, planes):
    items, outs = [], []
    for p in planes:
        s = torch.zeros((p.nhits, 4), device="cuda")
        items.append((torch.from_numpy(p.adc).cuda(), p.nticks, torch.from_numpy(p.hits).cuda(), s))
        outs.append(s)
    emtk.emtk_infer_batch(ctx, items)
    torch.cuda.synchronize()
    return [o.cpu() for o in outs]


def host_items(planes, pin=True):
    mk = (lambda t: t.pin_memory()) if pin else (lambda t: t)
    return [(mk(torch.from_numpy(p.adc)), p.nticks, mk(torch.from_numpy(p.hits)),
             mk(torch.full((p.nhits, 4), float("nan")))) for p in planes]


def test_matches_device_call(emtk, ctx):
    planes = synth.apa(seed=3)
    want = device_scores(emtk, ctx, planes)
    items = host_items(planes)
    emtk.emtk_infer_batch_host(ctx, items)
    torch.cuda.synchronize()
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    for (_, _, _, s), w in zip(items, want):
        assert torch.equal(s, w)


def test_calls_in_flight(emtk, ctx):
    """Four events enqueued back to back (the copy of one overlapping the
    kernels of the one before), synchronised once."""
    events = [synth.apa(seed=10 + k, hits=(900, 700, 400)) for k in range(4)]
    want = [device_scores(emtk, ctx, ev) for ev in events]
    items = [host_items(ev) for ev in events]
    for it in items:
        emtk.emtk_infer_batch_host(ctx, it)
    torch.cuda.synchronize()
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    for it, w in zip(items, want):
        for (_, _, _, s), ws in zip(it, w):
            assert torch.equal(s, ws)


def test_pageable_memory_and_empty_requests(emtk, ctx):
    planes = synth.apa(seed=5, hits=(300, 0, 200))
    want = device_scores(emtk, ctx, planes)
    items = host_items(planes, pin=False)
    emtk.emtk_infer_batch_host(ctx, items)
    torch.cuda.synchronize()
    for (_, _, _, s), w in zip(items, want):
        assert torch.equal(s, w)
