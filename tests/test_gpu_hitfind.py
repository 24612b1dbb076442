"""GPU parity of hit finding (emtk_find_hits) against the oracle on the same
seeded planes.

Bars: the number of hits and every integer field (wire, peak tick, start,
end) bit-exact, the peak value bit-exact (it is an input value); the charge,
an fp32 sum in the kernel's fixed order against the oracle's double sum,
within 1e-5 x sum|values| + 1e-3.  Hits found on a plane then go through
emtk_infer unchanged, and the scores match the oracle's on the oracle's
hits.
"""
import numpy as np
import pytest

import oracle
from paper_2009_04509_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

THR = 15.0  # 5 sigma of the synthetic noise


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    oracle.build()
    return m


@pytest.fixture(scope="module")
def ctx(emtk):
    c = emtk.emtk_create(synth.he_normal_weights(0), precision="bf16", debug_logits=True)
    yield c
    emtk.emtk_destroy(c)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def gpu_find(emtk, ctx, planes, capacity=None):
    """planes: list of (adc [nwires][ld] float32, nticks, threshold)."""
    items, outs = [], []
    for adc, nticks, thr in planes:
        most = adc.shape[0] * ((nticks + 1) // 2)  # one run per two ticks on every wire
        cap = capacity if capacity is not None else max(1, min(most, max(65536, adc.shape[0] * 256)))
        h = torch.full((cap, 2), -7, dtype=torch.int32, device="cuda")
        inf = torch.full((cap, 4), -7, dtype=torch.int32, device="cuda")
        items.append((dev(adc), nticks, thr, h, inf))
        outs.append((h, inf))
    n = emtk.emtk_find_hits(ctx, items)
    res = []
    for k, (h, inf) in zip(n, outs):
        m = min(k, h.shape[0])
        hh, ii = h[:m].cpu().numpy(), inf[:m].cpu().numpy()
        res.append(dict(n=k, wire=hh[:, 0], tick=hh[:, 1], start=ii[:, 0], end=ii[:, 1],
                        peak=ii[:, 2].view(np.float32), charge=ii[:, 3].view(np.float32), rest=h[m:].cpu().numpy()))
    return res


def check_plane(got, adc, nticks, thr):
    want = oracle.find_hits(adc, nticks, thr)
    n = want["wire"].size
    assert got["n"] == n
    m = got["wire"].size
    for f in ("wire", "tick", "start", "end"):
        assert np.array_equal(got[f], want[f][:m]), f
    assert np.array_equal(got["peak"], want["peak"][:m])
    if m:
        sab = np.array([np.abs(adc[w, s:e + 1].astype(np.float64)).sum()
                        for w, s, e in zip(want["wire"][:m], want["start"][:m], want["end"][:m])])
        assert np.all(np.abs(got["charge"] - want["charge"][:m]) <= 1e-5 * sab + 1e-3)
    return n


def test_one_apa(emtk, ctx):
    planes = synth.apa(seed=0)
    got = gpu_find(emtk, ctx, [(p.adc, p.nticks, THR) for p in planes])
    total = sum(check_plane(g, p.adc, p.nticks, THR) for g, p in zip(got, planes))
    assert total > 10_000


def test_full_event_one_call(emtk, ctx):
    """The 18 planes of the full event in one call (one launch group)."""
    planes = synth.full_event(seed=1)
    got = gpu_find(emtk, ctx, [(p.adc, p.nticks, THR) for p in planes])
    for g, p in zip(got, planes):
        check_plane(g, p.adc, p.nticks, THR)


def test_edges(emtk, ctx):
    nt = 1001  # not a multiple of 4 or of the 512-tick load block
    rng = np.random.default_rng(3)
    adc = np.full((7, 1024), 999.0, np.float32)  # pitch past nticks holds large values
    adc[:, :nt] = rng.standard_normal((7, nt)).astype(np.float32)
    adc[0, :nt] = 5.0                                   # the whole wire above
    adc[1, :nt] = 0.0
    adc[1, 0] = 4.0
    adc[1, nt - 1] = 4.0                                # first and last tick
    adc[2, :nt] = 0.0
    adc[2, 100:110] = [3, 4, 6, 6, 2, 6, 1, 0.5, 3, 3]  # ties; a value equal to the threshold
    adc[3, :nt] = 0.0
    adc[3, 127:130] = 2.0                               # across a 128-tick block edge
    adc[3, 511:514] = 2.0                               # across a 512-tick load edge
    adc[4, :nt] = np.where(np.arange(nt) % 2 == 0, 3.0, 0.0)  # the most runs a wire can hold
    thr = 1.0
    got = gpu_find(emtk, ctx, [(adc, nt, thr)])[0]
    check_plane(got, adc, nt, thr)
    assert (got["start"][0], got["end"][0]) == (0, nt - 1)


def test_segment_edges(emtk, ctx):
    """Runs across the 2048-tick work segments: one crossing 2048, one
    starting exactly there, a wire above everywhere (three segments, one
    hit), one crossing 4096 up to the last tick, and a wire with more runs per
    segment than the first pass keeps."""
    nt = 4200
    adc = np.zeros((6, 4208), np.float32)
    adc[0, 2040:2061] = np.linspace(2, 9, 21)
    adc[1, 2048:2051] = [5, 7, 5]
    adc[1, 2047] = 1.0  # equal to the threshold: below
    adc[2, :nt] = 3.0
    adc[2, 3000] = 4.0
    adc[3, 4090:nt] = 2.0
    adc[4, :nt] = np.where(np.arange(nt) % 3 == 0, 2.0, 0.0)
    adc[5, 2047] = 6.0
    adc[5, 2049] = 6.0
    got = gpu_find(emtk, ctx, [(adc, nt, 1.0)])[0]
    n = check_plane(got, adc, nt, 1.0)
    assert n == 1 + 1 + 1 + 1 + 1400 + 2
    assert (got["start"][2], got["end"][2], got["tick"][2]) == (0, nt - 1, 3000)


def test_degenerate_planes(emtk, ctx):
    z = np.zeros((0, 64), np.float32)
    one = np.zeros((1, 64), np.float32)
    one[0, 10:12] = 9.0
    notick = np.ones((3, 64), np.float32)
    got = gpu_find(emtk, ctx, [(z, 64, 0.0), (one, 64, 1.0), (notick, 0, 0.0), (one, 64, 20.0)], capacity=4)
    assert [g["n"] for g in got] == [0, 1, 0, 0]
    assert (got[1]["wire"][0], got[1]["tick"][0], got[1]["start"][0], got[1]["end"][0]) == (0, 10, 10, 11)


def test_capacity_overflow(emtk, ctx):
    """Many short runs (threshold 0 on noise); a short output keeps the first
    hits in order and reports the full count."""
    rng = np.random.default_rng(4)
    adc = (rng.standard_normal((64, 2000)) * 3).astype(np.float32)
    full = gpu_find(emtk, ctx, [(adc, 2000, 0.0)])[0]
    n = check_plane(full, adc, 2000, 0.0)
    assert n > 30_000
    short = gpu_find(emtk, ctx, [(adc, 2000, 0.0)], capacity=n // 3)[0]
    assert short["n"] == n
    check_plane(short, adc, 2000, 0.0)


def test_argument_errors(emtk, ctx):
    flat = torch.zeros(4 * 64 + 1, device="cuda")
    adc = flat[:256].view(4, 64)
    h = torch.zeros((8, 2), dtype=torch.int32, device="cuda")
    with pytest.raises(emtk.EmtkError):
        emtk.emtk_find_hits(ctx, [(flat[1:].view(4, 64), 64, 0.0, h, None)])  # base not 16-byte aligned
    with pytest.raises(emtk.EmtkError):
        emtk.emtk_find_hits(ctx, [(adc, 65, 0.0, h, None)])  # nticks > ld


def test_found_hits_feed_inference(emtk, ctx):
    """Raw plane in, scores out: the found hits go to emtk_infer as they are."""
    p = synth.single_plane(seed=2, nwires=480, nhits=1)
    got = gpu_find(emtk, ctx, [(p.adc, p.nticks, THR)])[0]
    n = check_plane(got, p.adc, p.nticks, THR)
    assert n > 100
    hits = np.stack([got["wire"], got["tick"]], 1).astype(np.int32)
    scores = torch.zeros((n, 8), device="cuda")
    emtk.emtk_infer(ctx, dev(p.adc), p.nticks, dev(hits), scores)
    assert emtk.emtk_check(ctx) == emtk.EMTK_OK
    want = oracle.find_hits(p.adc, p.nticks, THR)
    sel = np.random.default_rng(0).choice(n, min(n, 96), replace=False)
    wh = np.stack([want["wire"][sel], want["tick"][sel]], 1).astype(np.int32)
    _, emu = oracle.forward(oracle.extract_patches(p.adc, p.nticks, wh), synth.he_normal_weights(0), emulate="bf16")
    assert np.abs(scores.cpu().numpy()[sel, :4] - emu).max() <= 2e-2


def test_run_lengths_and_phases(emtk, ctx):
    """Runs of every length 1..70 starting at every phase of the 4-tick lane
    groups (short runs measured in registers, longer ones walked by the
    warp), some across the 512-tick stretch edges, with tied maxima."""
    rng = np.random.default_rng(7)
    nt = 6000
    adc = np.zeros((40, nt), np.float32)
    for w in range(40):
        t = int(rng.integers(0, 8))
        while t < nt - 80:
            ln = int(rng.integers(1, 71))
            vals = rng.integers(2, 9, ln).astype(np.float32)  # small integers: many ties
            adc[w, t:t + ln] = vals
            t += ln + int(rng.integers(1, 40))
    for w in range(40):  # runs across the stretch edges 512k
        e = 512 * (1 + w % 10)
        adc[w, e - 1 - w % 7:e + 3 + w % 5] = 5.0
    got = gpu_find(emtk, ctx, [(adc, nt, 1.0)])[0]
    assert check_plane(got, adc, nt, 1.0) > 2000


def test_slots_and_overflow_mix(emtk, ctx):
    """Units with 33..128 runs (kept in the slots) next to units with more
    (scanned again) and units with none, in one chunk."""
    nt = 4096
    adc = np.zeros((64, nt), np.float32)
    t = np.arange(nt)
    adc[0::3] = np.where(t % 20 == 0, 3.0, 0.0)   # 103 runs per segment
    adc[1::3] = np.where(t % 5 == 0, 3.0, 0.0)    # 410 runs per segment
    got = gpu_find(emtk, ctx, [(adc, nt, 1.0)])[0]
    assert check_plane(got, adc, nt, 1.0) == 22 * 205 + 21 * 820


def test_negative_threshold_signed_zero(emtk, ctx):
    """A negative threshold: zeros of both signs are above it and tie at the
    peak; the first of them is the hit."""
    adc = np.full((3, 256), -5.0, np.float32)
    adc[0, 10:14] = [-0.0, 0.0, -1.0, 0.0]
    adc[1, 100:140] = -0.5
    adc[1, 120] = 0.0
    adc[1, 125] = -0.0
    adc[2, 0:256] = -1.0
    got = gpu_find(emtk, ctx, [(adc, 256, -2.0)])[0]
    check_plane(got, adc, 256, -2.0)
    assert list(got["tick"]) == [10, 120, 0]
    assert np.signbit(got["peak"][0])


def test_planes_of_odd_unit_counts(emtk, ctx):
    """Several planes in one call whose unit counts are not multiples of the
    place kernel's 128-unit chunk, with empty planes between them."""
    rng = np.random.default_rng(11)
    planes = []
    for nw, ntk in [(1, 2049), (0, 100), (130, 700), (300, 4100), (5, 0), (77, 2048), (129, 6000)]:
        ld = max(4, (ntk + 3) // 4 * 4)
        adc = (rng.standard_normal((nw, ld)) * 3).astype(np.float32)
        adc[:, ntk:] = 99.0
        planes.append((adc, ntk, 6.0))
    got = gpu_find(emtk, ctx, planes)
    for g, (adc, ntk, thr) in zip(got, planes):
        check_plane(g, adc, ntk, thr)
    assert got[1]["n"] == 0 and got[4]["n"] == 0 and got[3]["n"] > 1000


def test_more_planes_than_one_group(emtk, ctx):
    """70 planes in one call: more than a launch group holds (64), so the
    call runs two groups; every plane's hits and count must still match."""
    rng = np.random.default_rng(13)
    planes = []
    for i in range(70):
        nw, nt = 1 + i % 5, 300 + 37 * i
        ld = (nt + 3) // 4 * 4
        adc = (rng.standard_normal((nw, ld)) * 3).astype(np.float32)
        planes.append((adc, nt, 4.0))
    got = gpu_find(emtk, ctx, planes)
    for g, (adc, nt, thr) in zip(got, planes):
        check_plane(g, adc, nt, thr)
