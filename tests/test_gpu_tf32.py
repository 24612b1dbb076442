"""GPU parity of EMTK_TF32, the fp32-accuracy tensor-core path (split fp16
operands, three products per fp32 product; include/emtk.h), against the fp64
oracle on every hit.  The bar is the fp32 one: max |score - fp64| <= 1e-3 on
every hit, and every logit within 2e-3 (1 + |z|) of the fp64 logit (the same
bars as the CUDA-core fp32 path).

Cases: the single-plane workload (480 x 6000, 256 hits on tracks); the
inference-only workload's largest batch, 65,536 pre-cut patches in one
emtk_infer_patches call (every hit); unsaturated inputs; hit counts off the
128-hit tile; hits on the plane's corners, outside it and duplicated; run to
run determinism.  The full 18-plane event is in test_gpu_full_event.py, the
window read in test_gpu_window_probe.py.
"""
import numpy as np
import pytest

import oracle
from paper_2009_04509_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-3
TOL_LOGIT = 2e-3


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    oracle.build()
    return m


@pytest.fixture(scope="module")
def weights():
    return synth.he_normal_weights(0)


@pytest.fixture(scope="module")
def ctx(emtk, weights):
    c = emtk.emtk_create(weights, precision="tf32", debug_logits=True)
    yield c
    emtk.emtk_destroy(c)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_infer(emtk, ctx, adc, nticks, hits):
    out = torch.full((hits.shape[0], 8), float("nan"), device="cuda")
    emtk.emtk_infer(ctx, dev(adc), nticks, dev(hits), out)
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    return out.cpu().numpy().astype(np.float64)


def check(got, lo, ref):
    s, z = got[:, :4], got[:, 4:]
    assert np.all(np.isfinite(got))
    assert np.all(np.abs(s[:, :3].sum(1) - 1.0) <= 1e-5)
    d = np.abs(s - ref)
    rel = np.abs(z - lo) / (1.0 + np.abs(lo))
    assert d.max() <= TOL, f"max |score - fp64| = {d.max():.3g}"
    assert rel.max() <= TOL_LOGIT, f"logit error {rel.max():.3g}"
    return d.max()


def test_tf32_single_plane(emtk, ctx, weights):
    plane = synth.single_plane(seed=0)
    got = run_infer(emtk, ctx, plane.adc, plane.nticks, plane.hits)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, plane.hits), weights)
    check(got, lo, ref)


def test_tf32_unsaturated(emtk):
    w = synth.he_normal_weights(0, bias_std=0.1)
    c = emtk.emtk_create(w, precision="tf32", debug_logits=True)
    try:
        plane = synth.scaled(synth.single_plane(seed=3), 0.01)
        got = run_infer(emtk, c, plane.adc, plane.nticks, plane.hits)
    finally:
        emtk.emtk_destroy(c)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, plane.hits), w)
    check(got, lo, ref)


@pytest.mark.parametrize("n", [1, 127, 128, 129, 383])
def test_tf32_tile_edges(emtk, ctx, weights, n):
    plane = synth.single_plane(seed=5, nhits=n, nticks=1200)
    got = run_infer(emtk, ctx, plane.adc, plane.nticks, plane.hits)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, plane.hits), weights)
    check(got, lo, ref)


def test_tf32_edge_and_outside_hits(emtk, ctx, weights):
    """Hits on the corners, outside the plane in every direction, at the
    trailing partial interval, and duplicated; ld > nticks with large values
    past nticks that must not be read."""
    base = synth.single_plane(seed=6, nhits=8, nticks=1199)
    nw, nt = base.nwires, base.nticks
    adc = np.full((nw, 1204), 3e4, np.float32)
    adc[:, :nt] = base.adc[:, :nt]
    edge = [[0, 0], [nw - 1, nt - 1], [0, nt - 1], [nw - 1, 0], [-100, 300], [20, 10_000_000], [5, -7],
            [5, -1], [nw + 23, 50], [nw + 24, 50], [-24, 100], [-25, 100], [nw // 2, nt], [nw // 2, nt - 1],
            [nw // 2, 6 * (nt // 6) - 1], [nw // 2, 6 * (nt // 6)]]
    rng = np.random.default_rng(9)
    rand = np.stack([rng.integers(-60, nw + 60, 60), rng.integers(-400, nt + 400, 60)], 1)
    hits = np.concatenate([np.array(edge), rand]).astype(np.int32)
    hits = np.concatenate([hits, hits[:5]])
    got = run_infer(emtk, ctx, adc, nt, hits)
    lo, ref = oracle.forward(oracle.extract_patches(adc, nt, hits), weights)
    check(got, lo, ref)
    assert np.array_equal(got[-5:], got[:5])


def test_tf32_largest_sweep_batch_every_hit(emtk, weights):
    """65,536 pre-cut fp32 patches (70% zeros, else lognormal(2, 1)) in one
    emtk_infer_patches call on a context with default options, as the
    inference-only sweep runs it; every hit against the fp64 oracle."""
    n = 65536
    x = synth.inference_patches(n, seed=0)
    c = emtk.emtk_create(weights, precision="tf32", debug_logits=True)
    try:
        out = torch.full((n, 8), float("nan"), device="cuda")
        emtk.emtk_infer_patches(c, dev(x), out)
        assert emtk.emtk_check(c) == emtk.EMTK_OK
        got = out.cpu().numpy().astype(np.float64)
    finally:
        emtk.emtk_destroy(c)
    lo, ref = oracle.forward(x, weights)
    check(got, lo, ref)


def test_tf32_deterministic(emtk, ctx):
    plane = synth.single_plane(seed=9, nhits=500, nticks=1200)
    a = run_infer(emtk, ctx, plane.adc, plane.nticks, plane.hits)
    b = run_infer(emtk, ctx, plane.adc, plane.nticks, plane.hits)
    assert np.array_equal(a, b)


@pytest.mark.parametrize("scale", [200.0, 0.001])
def test_tf32_range_ends(emtk, ctx, weights, scale):
    """The path's range: ADC x 200 puts the largest interval values near 4e4
    and the largest conv activations near 5e5 (below the 2^20 limit of the
    head/tail scales); ADC x 0.001 puts most pixel tails in fp16's subnormal
    range.  Both keep the fp32 bars."""
    plane = synth.scaled(synth.single_plane(seed=11, nhits=300), scale)
    got = run_infer(emtk, ctx, plane.adc, plane.nticks, plane.hits)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, plane.hits), weights)
    check(got, lo, ref)


def test_tf32_chunked_call(emtk, weights):
    """A context whose workspace holds 256 hits runs a 700-hit call in chunks."""
    c = emtk.emtk_create(weights, precision="tf32", debug_logits=True, max_hits=256)
    try:
        plane = synth.single_plane(seed=10, nhits=700, nticks=1200)
        got = run_infer(emtk, c, plane.adc, plane.nticks, plane.hits)
        assert emtk.emtk_get_stats(c)["chunks"] >= 3
    finally:
        emtk.emtk_destroy(c)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, plane.hits), weights)
    check(got, lo, ref)


def test_tf32_batcher_and_host_call(emtk, ctx, weights):
    """The request batcher and the host-buffer call on a tf32 context: every
    hit within the fp32 bars of the oracle."""
    planes = synth.apa(seed=12, hits=(400, 300, 200), n_tracks=6, n_showers=2)
    want = [oracle.forward(oracle.extract_patches(p.adc, p.nticks, p.hits), weights) for p in planes]
    b = emtk.emtk_batcher_create(ctx, nstreams=2, max_hits=600, max_delay_us=200)
    try:
        outs, tickets, keep = [], [], []
        for p in planes:
            # the request's buffers must stay alive until its ticket has been waited for
            adc, hits = dev(p.adc), dev(p.hits)
            out = torch.full((p.nhits, 8), float("nan"), device="cuda")
            keep.append((adc, hits))
            tickets.append(emtk.emtk_batcher_submit(b, adc, p.nticks, hits, out))
            outs.append(out)
        for t in tickets:
            assert emtk.emtk_batcher_wait(b, t, 60_000) == emtk.EMTK_OK
    finally:
        emtk.emtk_batcher_destroy(b)
    for out, (lo, ref) in zip(outs, want):
        check(out.cpu().numpy().astype(np.float64), lo, ref)
    items = [(torch.from_numpy(p.adc).pin_memory(), p.nticks, torch.from_numpy(p.hits).pin_memory(),
              torch.full((p.nhits, 8), float("nan")).pin_memory()) for p in planes]
    emtk.emtk_infer_batch_host(ctx, items)
    torch.cuda.synchronize()
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    for it, (lo, ref) in zip(items, want):
        check(it[3].numpy().astype(np.float64), lo, ref)


def test_tf32_on_found_hits(emtk, ctx, weights):
    """Hits found on the plane by emtk_find_hits, scored unchanged."""
    plane = synth.single_plane(seed=13, nhits=10, nticks=1200)
    adc = dev(plane.adc)
    cap = 4096
    fh = torch.zeros((cap, 2), dtype=torch.int32, device="cuda")
    n = emtk.emtk_find_hits(ctx, [(adc, plane.nticks, 15.0, fh, None)])[0]
    assert 0 < n <= cap
    hits = fh[:n].cpu().numpy()
    got = run_infer(emtk, ctx, plane.adc, plane.nticks, hits)
    lo, ref = oracle.forward(oracle.extract_patches(plane.adc, plane.nticks, hits), weights)
    check(got, lo, ref)
