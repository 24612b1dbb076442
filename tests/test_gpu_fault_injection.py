"""Host-side fault injection (the paper's service survives failed workers by
replacing them, Sec. 2.4; here the library itself must survive the failures
a long-running service meets): an allocation that fails as on an exhausted
device, and a batch dispatcher that stops making progress.  Every failure is
made on the host (emtk_debug_fail_alloc, emtk_debug_batcher_stall); no test
here faults, traps or hangs the GPU.

Checked for each allocation of emtk_create, of a workspace growth
(ensure the interval-image buffer grows), of a staging-area growth of
emtk_infer_batch_host and of emtk_batcher_create: the entry point returns
EMTK_ERR_OOM, the library's live allocation counts return to what they were
(nothing leaked), and the context then scores a plane exactly as a context
that never failed.
"""
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
    yield m
    m.emtk_debug_fail_alloc(-1)


@pytest.fixture(scope="module")
def setup(emtk):
    w = synth.he_normal_weights(0)
    small = synth.single_plane(seed=1, nwires=120, nhits=200, nticks=1200)
    big = synth.single_plane(seed=2, nwires=480, nhits=300, nticks=6000)
    dev = torch.device("cuda:0")
    ref = emtk.emtk_create(w, precision="bf16", max_hits=512)
    want = {}
    try:
        for name, p in (("small", small), ("big", big)):
            sc = torch.zeros((p.nhits, 4), device=dev)
            emtk.emtk_infer(ref, torch.from_numpy(p.adc).to(dev), p.nticks, torch.from_numpy(p.hits).to(dev), sc)
            assert emtk.emtk_check(ref) == emtk.EMTK_OK
            want[name] = sc.cpu().numpy()
    finally:
        emtk.emtk_destroy(ref)
    return dict(w=w, planes={"small": small, "big": big}, want=want, dev=dev)


def score(emtk, ctx, p, dev):
    sc = torch.zeros((p.nhits, 4), device=dev)
    emtk.emtk_infer(ctx, torch.from_numpy(p.adc).to(dev), p.nticks, torch.from_numpy(p.hits).to(dev), sc)
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    return sc.cpu().numpy()


def create_rc(emtk, w, **kw):
    try:
        return emtk.EMTK_OK, emtk.emtk_create(w, **kw)
    except emtk.EmtkError as e:
        return e.status, None


@pytest.mark.parametrize("prec", ["bf16", "fp32"])
def test_create_fails_cleanly_at_every_allocation(emtk, setup, prec):
    w, dev = setup["w"], setup["dev"]
    torch.cuda.synchronize()
    base = emtk.emtk_debug_alloc_counts()
    failures = 0
    for after in range(64):
        emtk.emtk_debug_fail_alloc(after)
        rc, ctx = create_rc(emtk, w, precision=prec, max_hits=512)
        emtk.emtk_debug_fail_alloc(-1)
        if rc == emtk.EMTK_OK:        # `after` exceeds the number of allocations emtk_create makes
            try:
                if prec == "bf16":
                    assert np.array_equal(score(emtk, ctx, setup["planes"]["small"], dev), setup["want"]["small"])
            finally:
                emtk.emtk_destroy(ctx)
            break
        assert rc == emtk.EMTK_ERR_OOM, emtk.status_string(rc)
        assert emtk.emtk_debug_alloc_counts() == base, f"allocation {after}: leaked"
        failures += 1
    assert failures >= 10                  # weights and workspace: every one of them was made to fail
    assert emtk.emtk_debug_alloc_counts() == base


def test_workspace_growth_fails_then_recovers(emtk, setup):
    """The interval-image buffer grows on the first call and again for a
    larger plane; both growths fail once, return EMTK_ERR_OOM with nothing
    enqueued, and the next call scores correctly."""
    dev = setup["dev"]
    ctx = emtk.emtk_create(setup["w"], precision="bf16", max_hits=512)
    try:
        for name in ("small", "big"):
            p = setup["planes"][name]
            before = emtk.emtk_debug_alloc_counts()
            emtk.emtk_debug_fail_alloc(0)
            sc = torch.full((p.nhits, 4), -7.0, device=dev)
            with pytest.raises(emtk.EmtkError) as ei:
                emtk.emtk_infer(ctx, torch.from_numpy(p.adc).to(dev), p.nticks, torch.from_numpy(p.hits).to(dev), sc)
            emtk.emtk_debug_fail_alloc(-1)
            assert ei.value.status == emtk.EMTK_ERR_OOM
            torch.cuda.synchronize()
            assert bool((sc == -7.0).all())    # nothing was written
            # the old buffer was given back before the failed growth: one fewer, never more
            assert emtk.emtk_debug_alloc_counts()[0] <= before[0]
            assert np.array_equal(score(emtk, ctx, p, dev), setup["want"][name])
    finally:
        emtk.emtk_destroy(ctx)


def test_host_staging_growth_fails_then_recovers(emtk, setup):
    dev = setup["dev"]
    p = setup["planes"]["big"]
    ctx = emtk.emtk_create(setup["w"], precision="bf16", max_hits=512)
    try:
        items = [(torch.from_numpy(p.adc).pin_memory(), p.nticks, torch.from_numpy(p.hits).pin_memory(),
                  torch.zeros((p.nhits, 4)).pin_memory())]
        for after in (0, 1):     # the device staging area, then the pinned hit-list area
            emtk.emtk_debug_fail_alloc(after)
            with pytest.raises(emtk.EmtkError) as ei:
                emtk.emtk_infer_batch_host(ctx, items)
            emtk.emtk_debug_fail_alloc(-1)
            assert ei.value.status == emtk.EMTK_ERR_OOM
            torch.cuda.synchronize()
        emtk.emtk_infer_batch_host(ctx, items)
        torch.cuda.synchronize()
        assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        assert np.array_equal(items[0][3].numpy(), setup["want"]["big"])
    finally:
        emtk.emtk_destroy(ctx)
    emtk.emtk_debug_fail_alloc(-1)


def test_batcher_create_fails_cleanly(emtk, setup):
    ctx = emtk.emtk_create(setup["w"], precision="bf16", max_hits=512)
    try:
        base = emtk.emtk_debug_alloc_counts()
        n = 0
        for after in range(64):
            emtk.emtk_debug_fail_alloc(after)
            try:
                b = emtk.emtk_batcher_create(ctx, nstreams=2, max_hits=4096, max_delay_us=100)
            except emtk.EmtkError as e:
                emtk.emtk_debug_fail_alloc(-1)
                assert e.status == emtk.EMTK_ERR_OOM
                assert emtk.emtk_debug_alloc_counts() == base, f"allocation {after}: leaked"
                n += 1
                continue
            emtk.emtk_debug_fail_alloc(-1)
            emtk.emtk_batcher_destroy(b)
            break
        assert n >= 3                      # the pinned status words and both lanes' workspaces
        assert emtk.emtk_debug_alloc_counts() == base
        # the context still scores correctly
        assert np.array_equal(score(emtk, ctx, setup["planes"]["small"], setup["dev"]), setup["want"]["small"])
    finally:
        emtk.emtk_destroy(ctx)


def test_stalled_dispatcher_times_out_and_keeps_the_ticket(emtk, setup):
    dev = setup["dev"]
    p = setup["planes"]["small"]
    ctx = emtk.emtk_create(setup["w"], precision="bf16", max_hits=512)
    try:
        b = emtk.emtk_batcher_create(ctx, nstreams=2, max_hits=4096, max_delay_us=0)
        try:
            adc, hits = torch.from_numpy(p.adc).to(dev), torch.from_numpy(p.hits).to(dev)
            sc = torch.full((p.nhits, 4), -7.0, device=dev)
            torch.cuda.synchronize()
            emtk.emtk_debug_batcher_stall(b, True)
            t = emtk.emtk_batcher_submit(b, adc, p.nticks, hits, sc)
            for _ in range(3):
                assert emtk.emtk_batcher_wait(b, t, 50) == emtk.EMTK_ERR_TIMEOUT
            assert emtk.emtk_batcher_stats(b)["batches"] == 0
            torch.cuda.synchronize()
            assert bool((sc == -7.0).all())
            emtk.emtk_debug_batcher_stall(b, False)
            assert emtk.emtk_batcher_wait(b, t, 10_000) == emtk.EMTK_OK
            assert emtk.emtk_batcher_wait(b, t, 0) == emtk.EMTK_ERR_ARG    # consumed once
            assert np.abs(sc.cpu().numpy() - setup["want"]["small"]).max() <= 1e-3
            # a stalled batcher still launches its queue when destroyed
            sc2 = torch.full((p.nhits, 4), -7.0, device=dev)
            emtk.emtk_debug_batcher_stall(b, True)
            emtk.emtk_batcher_submit(b, adc, p.nticks, hits, sc2)
        finally:
            emtk.emtk_batcher_destroy(b)
        torch.cuda.synchronize()
        assert np.abs(sc2.cpu().numpy() - setup["want"]["small"]).max() <= 1e-3
        with pytest.raises(emtk.EmtkError):
            emtk.emtk_debug_batcher_stall(None, True)
    finally:
        emtk.emtk_destroy(ctx)
