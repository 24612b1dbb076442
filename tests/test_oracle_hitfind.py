"""Pins for the oracle's hit finding (Sec. 2.1, read as: per wire, each
maximal run of ticks above a threshold is one hit at the run's largest value,
the earliest on ties; charge = the run's sum).

* closed forms: rectangular pulses (start, end, height x width), ties, a
  sampled Gaussian pulse whose run ends follow from the threshold;
* the plane's edges: runs touching tick 0 and the last tick, a wire that is
  above everywhere, data past nticks in the row pitch, runs on neighbouring
  wires that must not merge, a value equal to the threshold;
* a library restatement: scipy.ndimage.label / find_objects / sum_labels /
  maximum_position per wire, on tie-free random waveforms;
* capacity: a short output keeps the first hits and still reports the count.

``test_planted_mistakes`` compiles copies of the oracle with one plausible
mistake in the hit finder each and checks that some pin fails on every copy.
"""
import math
import os
import shutil
import subprocess

import numpy as np
import pytest
import scipy.ndimage as ndi

import oracle


def rows_to_plane(rows, ld=None, pad_value=0.0):
    rows = [np.asarray(r, np.float32) for r in rows]
    nticks = len(rows[0])
    ld = ld or nticks
    a = np.full((len(rows), ld), pad_value, np.float32)
    for i, r in enumerate(rows):
        a[i, :nticks] = r
    return a, nticks


def as_tuples(h):
    return list(zip(h["wire"].tolist(), h["tick"].tolist(), h["start"].tolist(), h["end"].tolist(),
                    h["peak"].tolist(), h["charge"].tolist()))


# --------------------------------------------------------------------- pins
def pin_rectangles(lib):
    """Rectangular pulses of known height and width on a zero baseline."""
    row = np.zeros(40, np.float32)
    row[3:8] = 4.0          # width 5, flat: peak at its first tick
    row[12] = 9.0           # one tick
    row[20:26] = [1, 2, 6, 6, 2, 1]  # tie at 22/23 -> 22
    a, nt = rows_to_plane([row])
    h = oracle.find_hits(a, nt, 0.5, lib=lib)
    assert as_tuples(h) == [(0, 3, 3, 7, 4.0, 20.0), (0, 12, 12, 12, 9.0, 9.0), (0, 22, 20, 25, 6.0, 18.0)]


def pin_edges(lib):
    """Runs that touch the first and the last tick, a wire above everywhere,
    neighbouring wires that must stay separate, and data past nticks."""
    nt = 16
    r0 = np.zeros(nt); r0[:3] = [5, 3, 2]; r0[-2:] = [1.5, 8]
    r1 = np.full(nt, 2.0); r1[7] = 2.5
    r2 = np.zeros(nt); r2[0] = 7
    a, _ = rows_to_plane([r0, r1, r2], ld=24, pad_value=100.0)  # the pitch holds large values past nticks
    h = oracle.find_hits(a, nt, 1.0, lib=lib)
    assert as_tuples(h) == [(0, 0, 0, 2, 5.0, 10.0), (0, 15, 14, 15, 8.0, 9.5),
                            (1, 7, 0, 15, 2.5, 32.5), (2, 0, 0, 0, 7.0, 7.0)]


def pin_threshold_is_strict(lib):
    t = np.float32(3.0)
    up = np.nextafter(t, np.float32(np.inf))
    row = np.array([3.0, up, 3.0, 3.0, 5.0, 3.0], np.float32)
    a, nt = rows_to_plane([row])
    h = oracle.find_hits(a, nt, float(t), lib=lib)
    assert h["start"].tolist() == [1, 4] and h["end"].tolist() == [1, 4]
    assert oracle.find_hits(a, nt, 5.0, lib=lib)["wire"].size == 0


def pin_gaussian_pulse(lib):
    """A pulse A exp(-(t - tau)^2 / (2 s^2)) sampled at integer ticks: the
    run is the set of ticks with |t - tau| < s sqrt(2 ln(A / T)), its peak the
    tick nearest tau."""
    A, tau, s, T = 150.0, 37.3, 3.0, 15.0
    t = np.arange(80)
    row = (A * np.exp(-0.5 * ((t - tau) / s) ** 2)).astype(np.float32)
    half = s * math.sqrt(2.0 * math.log(A / T))
    a, nt = rows_to_plane([row])
    h = oracle.find_hits(a, nt, T, lib=lib)
    assert h["start"].tolist() == [math.floor(tau - half) + 1]
    assert h["end"].tolist() == [math.ceil(tau + half) - 1]
    assert h["tick"].tolist() == [round(tau)]
    assert h["charge"][0] == pytest.approx(float(row[row > T].astype(np.float64).sum()), rel=1e-15)


def pin_scipy_label(lib):
    """Per wire, the same runs from scipy.ndimage's labelling routines."""
    rng = np.random.default_rng(3)
    a = (rng.standard_normal((37, 333)) * 3.0).astype(np.float32)
    a[:, 100:140] += np.linspace(0, 40, 40, dtype=np.float32)
    nt = 321  # the last 12 columns are pitch
    T = 2.5
    want = []
    for w in range(a.shape[0]):
        x = a[w, :nt].astype(np.float64)
        lab, n = ndi.label(x > T)
        if n == 0:
            continue
        idx = np.arange(1, n + 1)
        objs = ndi.find_objects(lab)
        pos = ndi.maximum_position(x, lab, idx)
        sums = ndi.sum_labels(x, lab, idx)
        for k in range(n):
            want.append((w, int(pos[k][0]), objs[k][0].start, objs[k][0].stop - 1, float(a[w, pos[k][0]]),
                         float(sums[k])))
    got = as_tuples(oracle.find_hits(a, nt, T, lib=lib))
    assert len(got) == len(want) > 500
    for g, e in zip(got, want):
        assert g[:5] == e[:5]
        assert g[5] == pytest.approx(e[5], rel=1e-12, abs=1e-12)


def pin_empty(lib):
    a = np.zeros((4, 10), np.float32)
    assert oracle.find_hits(a, 10, 0.0, lib=lib)["wire"].size == 0
    assert oracle.find_hits(np.zeros((0, 8), np.float32), 8, 0.0, lib=lib)["wire"].size == 0
    assert oracle.find_hits(np.ones((3, 8), np.float32), 0, 0.0, lib=lib)["wire"].size == 0


def pin_capacity(lib):
    """A short output keeps the first hits and reports the full count."""
    import ctypes
    rng = np.random.default_rng(5)
    a = (rng.standard_normal((6, 200)) * 3).astype(np.float32)
    full = oracle.find_hits(a, 200, 2.0, lib=lib)
    n = full["wire"].size
    cap = n // 3
    w, t, s, e = (np.zeros(cap, np.int32) for _ in range(4))
    pk, q = np.zeros(cap, np.float32), np.zeros(cap, np.float64)
    p32 = lambda x: x.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))  # noqa: E731
    got = lib.or_find_hits(a.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), 6, 200, 200, ctypes.c_float(2.0), cap,
                           p32(w), p32(t), p32(s), p32(e), pk.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                           q.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    assert got == n
    assert np.array_equal(w, full["wire"][:cap]) and np.array_equal(t, full["tick"][:cap])
    assert np.array_equal(q, full["charge"][:cap])


PINS = [pin_rectangles, pin_edges, pin_threshold_is_strict, pin_gaussian_pulse, pin_scipy_label, pin_empty,
        pin_capacity]


@pytest.fixture(scope="module")
def oracle_lib():
    return oracle.load()


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin, oracle_lib):
    pin(oracle_lib)


# ---------------------------------------------------------- planted mistakes
MUTATIONS = {
    "threshold_inclusive": ("    return v > threshold;", "    return v >= threshold;"),
    "ties_latest": ("if (row[t] > row[best])", "if (row[t] >= row[best])"),
    "charge_skips_first": ("q += (double)row[t];", "if (t > first) q += (double)row[t];"),
    "end_one_past": ("end[n] = t - 1;", "end[n] = t;"),
    "peak_value_at_start": ("peak[n] = row[best];", "peak[n] = row[first];"),
    "last_wire_skipped": ("for (int w = 0; w < nwires; ++w) {\n        const float *row = plane + (long)w * ld;",
                          "for (int w = 0; w < nwires - 1; ++w) {\n        const float *row = plane + (long)w * ld;"),
    "pitch_ignored": ("const float *row = plane + (long)w * ld;\n        int t = 0;",
                      "const float *row = plane + (long)w * nticks;\n        int t = 0;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistakes(name, tmp_path, oracle_lib):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    old, new = MUTATIONS[name]
    src = open(os.path.join(os.path.dirname(oracle.__file__), "oracle.c")).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not found exactly once"
    mutated = tmp_path / "oracle_mut.c"
    mutated.write_text(src.replace(old, new))
    so = tmp_path / "liboracle_mut.so"
    subprocess.run(["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared", str(mutated),
                    "-o", str(so), "-lm"], check=True)
    lib = oracle.load(str(so))
    failed = []
    for pin in PINS:
        try:
            pin(lib)
        except (AssertionError, ValueError, RuntimeError):
            failed.append(pin.__name__)
    assert failed, f"planted mistake {name} passed every pin"
