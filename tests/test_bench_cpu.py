"""The benchmark's host-side arithmetic on CPU: the patch cut's algorithmic
bytes (the union of the hits' windows, each sample once) against a brute-force
mask, and the peaks the rooflines divide by."""
import numpy as np

import bench
from paper_2009_04509_gb300 import synth


class _Plane:
    def __init__(self, nwires, nticks, hits):
        self.nwires, self.nticks = nwires, nticks
        self.hits = np.asarray(hits, np.int32).reshape(-1, 2)
        self.nhits = len(self.hits)


def _brute_union_bytes(planes, patch=48, ds=6):
    total = 0
    for p in planes:
        nint = p.nticks // ds
        m = np.zeros((p.nwires, nint), bool)
        for w, t in p.hits:
            b = t // ds  # floor division, as the cut centres on interval floor(t / 6)
            for r in range(w - patch // 2, w + patch // 2):
                for c in range(b - patch // 2, b + patch // 2):
                    if 0 <= r < p.nwires and 0 <= c < nint:
                        m[r, c] = True
        total += int(m.sum()) * ds * 4
    return total


def test_union_of_one_interior_window():
    p = _Plane(100, 600, [[50, 300]])
    assert bench.window_union_bytes([p]) == 48 * 48 * 6 * 4


def test_union_clipped_and_overlapping_windows():
    rng = np.random.default_rng(0)
    cases = [
        _Plane(30, 200, [[0, 0], [29, 199], [5, -40], [-10, 50]]),   # corners, negative tick, off-plane wire
        _Plane(64, 607, rng.integers(-5, 70, (40, 2)) * [1, 9]),     # many overlaps, a trailing partial interval
        _Plane(10, 60, []),                                           # no hits
    ]
    for p in cases:
        assert bench.window_union_bytes([p]) == _brute_union_bytes([p])
    assert bench.window_union_bytes(cases) == _brute_union_bytes(cases)


def test_union_on_a_synthetic_plane():
    p = synth.single_plane(seed=0, nwires=120, nhits=40, nticks=1200)
    assert bench.window_union_bytes([p]) == _brute_union_bytes([p])


def test_network_peaks():
    peaks = {"hbm": 6000.0, "bf16": 1900.0, "bf16_sus": 1700.0, "source": "measured"}
    # the network kernel is one ~1 ms launch timed alone: the burst figure by default
    p16, _ = bench.network_peak("bf16", peaks)
    assert p16 == 1900.0
    assert bench.network_peak("fp16", peaks)[0] == 1900.0
    assert bench.network_peak("bf16", peaks, sustained=True)[0] == 1700.0
    p8, _ = bench.network_peak("fp8", peaks)
    # conv at the bf16 rate, dense-1 at twice it: the FLOP-weighted harmonic mix
    want = (bench.FLOP_CONV + bench.FLOP_FC1) / (bench.FLOP_CONV / 1900.0 + bench.FLOP_FC1 / 3800.0)
    assert abs(p8 - want) < 1e-9 and 1900.0 < p8 < 3800.0
    # the split-fp16 path runs three 16-bit products per fp32 product
    assert abs(bench.network_peak("tf32", peaks)[0] - 1900.0 / 3.0) < 1e-9
    p32, src = bench.network_peak("fp32", peaks)
    assert abs(p32 - 152 * 128 * 2 * 2.07e9 / 1e12) < 1e-9 and "derived" in src


def test_tiled_cut_label_follows_the_library_threshold():
    """The benchmark names the patch-cut kernels from the planes' size with the
    library's rule: the tiled cut from 96 MiB of planes with hits.  The
    threshold is read from the library source so that the two cannot drift."""
    import os
    import re
    src = open(os.path.join(os.path.dirname(bench.__file__), "paper_2009_04509_gb300", "csrc", "api.cu")).read()
    m = re.search(r"constexpr int64_t kTiledCutMinBytes = \(int64_t\)(\d+) << (\d+);", src)
    assert m, "the threshold's definition moved"
    limit = int(m.group(1)) << int(m.group(2))
    words = limit // 4

    class P:  # a plane of `nwires` x 6000 fp32 ticks with or without hits
        def __init__(self, nwires, nhits):
            self.nwires, self.nticks, self.nhits = nwires, 6000, nhits

    at = -(-words // 6000)   # wires that just reach the threshold
    assert bench.tiled_cut([P(at, 1)])
    assert not bench.tiled_cut([P(at - 1, 1)])
    assert not bench.tiled_cut([P(at, 0)])                  # planes without hits do not count
    assert bench.tiled_cut([P(at // 2, 3), P(at - at // 2, 5)])
    full = synth.full_event(seed=0)
    assert bench.tiled_cut(full)                              # 368.6 MB: the tiled cut
    assert not bench.tiled_cut([synth.single_plane(seed=0)])  # 11.5 MB: whole planes
