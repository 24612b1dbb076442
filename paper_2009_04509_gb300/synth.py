"""Seeded synthetic ProtoDUNE-SP-shaped inputs: wire planes, hit lists, patches, weights.

This module only draws random numbers and lays them out; it holds none of the
hit-identification arithmetic (no downsampling, no patch cut, no network), so
it can feed both the CUDA library and the CPU oracle without coupling them.

What it stands in for (Sec. 3.1 of the paper): Corsika cosmic-ray Monte Carlo
with RadioGen backgrounds, 15,360 channels read out for 3 ms at 0.5 us per
tick (6000 ticks), and the trained EmTrackMichelId network (Sec. 2.2).  None
of that is available, so:

* ADC plane: white Gaussian noise N(0, 3^2) per sample plus unipolar pulses
  (Gaussian in time, sigma 3 ticks, cut at +-4 sigma, amplitude U(20, 200)).
* Tracks: straight lines between uniform (wire, tick) endpoints; every wire a
  track crosses gets one pulse at the interpolated tick; track hits are
  (wire, round(tick)) samples on a track.
* EM showers: uniform apex, axis angle U(0, 2 pi), half-opening 0.2 rad,
  length U(50, 200) wires, 6 ticks ~ 1 wire; a hit sits at depth d ~ U(0, L)
  with transverse offset N(0, (d tan 0.2)^2) and adds its own pulse.
* Michel-like segments: short straight segments of U(5, 20) wires.
* Weights: He-normal N(0, 2/fan_in), drawn from numpy's PCG64 with seed 0 in
  the order conv, fc1, fc2, cls, mic, C order over the layouts below; biases 0
  unless asked for.

Layouts (Sec. 2.2, 11,900,420 parameters):
  conv_w [5][5][1][48] (tap row i, tap col j, in-channel, filter) + conv_b [48]
  fc1_w  [92928][128]  (input index (y*44+x)*48+c, output)        + fc1_b [128]
  fc2_w  [128][32]                                                 + fc2_b [32]
  cls_w  [32][3]  (track, em, none)                                + cls_b [3]
  mic_w  [32][1]                                                   + mic_b [1]
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

PATCH = 48            # patch side (Sec. 2.1)
DOWNSAMPLE = 6        # ticks per time bin
KSIZE = 5             # conv kernel side (Sec. 2.2)
NFILT = 48            # conv filters
CONV_OUT = PATCH - KSIZE + 1          # 44
FC1_IN = CONV_OUT * CONV_OUT * NFILT  # 92,928
FC1_OUT = 128
FC2_OUT = 32
NCLASS = 3
NTICKS = 6000         # 3 ms at 0.5 us per tick (Sec. 3.1)

NOISE_SIGMA = 3.0
PULSE_SIGMA = 3.0
PULSE_HALF = 12       # +-4 sigma
AMP_LO, AMP_HI = 20.0, 200.0
SHOWER_HALF_ANGLE = 0.2
TICKS_PER_WIRE = 6.0

WEIGHT_SHAPES = (
    ("conv_w", (KSIZE, KSIZE, 1, NFILT), KSIZE * KSIZE),
    ("fc1_w", (FC1_IN, FC1_OUT), FC1_IN),
    ("fc2_w", (FC1_OUT, FC2_OUT), FC1_OUT),
    ("cls_w", (FC2_OUT, NCLASS), FC2_OUT),
    ("mic_w", (FC2_OUT, 1), FC2_OUT),
)
BIAS_SHAPES = (("conv_b", NFILT), ("fc1_b", FC1_OUT), ("fc2_b", FC2_OUT),
               ("cls_b", NCLASS), ("mic_b", 1))


def he_normal_weights(seed: int = 0, bias_std: float = 0.0, bias_seed: int = 12345,
                      dims: dict | None = None) -> dict:
    """He-normal weights (float32) in the layouts of the module docstring.

    ``dims`` may shrink the network for tiny tests: keys P (patch side), R
    (kernel side), F (filters), N1, N2, NC.  Biases are zero when
    ``bias_std == 0`` else N(0, bias_std^2) from their own generator.
    """
    if dims is None:
        shapes = WEIGHT_SHAPES
        bshapes = BIAS_SHAPES
    else:
        P, R, F = dims["P"], dims["R"], dims["F"]
        N1, N2, NC = dims["N1"], dims["N2"], dims["NC"]
        Q = P - R + 1
        shapes = (("conv_w", (R, R, 1, F), R * R), ("fc1_w", (Q * Q * F, N1), Q * Q * F),
                  ("fc2_w", (N1, N2), N1), ("cls_w", (N2, NC), N2), ("mic_w", (N2, 1), N2))
        bshapes = (("conv_b", F), ("fc1_b", N1), ("fc2_b", N2), ("cls_b", NC), ("mic_b", 1))
    rng = np.random.default_rng(seed)
    out = {}
    for name, shape, fan_in in shapes:
        std = math.sqrt(2.0 / fan_in)
        out[name] = (rng.standard_normal(shape) * std).astype(np.float32)
    brng = np.random.default_rng(bias_seed)
    for name, n in bshapes:
        if bias_std == 0.0:
            out[name] = np.zeros(n, np.float32)
        else:
            out[name] = (brng.standard_normal(n) * bias_std).astype(np.float32)
    return out


def parameter_count(weights: dict) -> int:
    return int(sum(np.asarray(v).size for v in weights.values()))


@dataclasses.dataclass
class Plane:
    """One wire plane: ADC samples ``adc[nwires][ld]`` (float32, only the first
    ``nticks`` columns of a row are data) and its hits ``hits[n][2]`` = (wire,
    peak tick), int32.  ``kind[n]`` is 0 track, 1 shower, 2 Michel-like."""
    adc: np.ndarray
    nticks: int
    hits: np.ndarray
    kind: np.ndarray

    @property
    def nwires(self) -> int:
        return int(self.adc.shape[0])

    @property
    def ld(self) -> int:
        return int(self.adc.shape[1])

    @property
    def nhits(self) -> int:
        return int(self.hits.shape[0])


def _pulses(nwires, ld, wires, ticks, amps):
    """Sum of Gaussian pulses as a dense [nwires][ld] float64 array."""
    wires = np.asarray(wires, np.int64)
    ticks = np.asarray(ticks, np.float64)
    amps = np.asarray(amps, np.float64)
    acc = np.zeros(nwires * ld, np.float64)
    if wires.size == 0:
        return acc.reshape(nwires, ld)
    base = np.floor(ticks).astype(np.int64)
    offs = np.arange(-PULSE_HALF, PULSE_HALF + 2, dtype=np.int64)
    t = base[:, None] + offs[None, :]
    val = amps[:, None] * np.exp(-0.5 * ((t - ticks[:, None]) / PULSE_SIGMA) ** 2)
    keep = (np.abs(t - ticks[:, None]) <= 4.0 * PULSE_SIGMA) & (t >= 0) & (t < ld)
    idx = (wires[:, None] * ld + t)[keep]
    acc += np.bincount(idx, weights=val[keep], minlength=nwires * ld)
    return acc.reshape(nwires, ld)


def _line_wires(w0, t0, w1, t1, nwires):
    """Integer wires crossed by the segment (w0,t0)-(w1,t1) and the
    interpolated tick on each."""
    lo, hi = min(w0, w1), max(w0, w1)
    ws = np.arange(max(0, math.ceil(lo)), min(nwires - 1, math.floor(hi)) + 1, dtype=np.int64)
    if ws.size == 0 or w1 == w0:
        return ws[:0], np.zeros(0)
    ts = t0 + (ws - w0) * (t1 - t0) / (w1 - w0)
    return ws, ts


def make_plane(rng: np.random.Generator, nwires: int, nticks: int = NTICKS, *,
               n_tracks: int = 30, n_showers: int = 5, n_michel: int = 0,
               hits_track: int = 0, hits_shower: int = 0, hits_michel: int = 0,
               ld: int | None = None, noise_sigma: float = NOISE_SIGMA) -> Plane:
    ld = nticks if ld is None else ld
    assert ld >= nticks
    adc = np.zeros((nwires, ld), np.float32)
    adc[:, :nticks] = rng.standard_normal((nwires, nticks), dtype=np.float32) * np.float32(noise_sigma)

    pw, pt, pa = [], [], []

    def add_segment(w0, t0, w1, t1):
        ws, ts = _line_wires(w0, t0, w1, t1, nwires)
        keep = (ts >= 0) & (ts <= nticks - 1)
        ws, ts = ws[keep], ts[keep]
        pw.append(ws)
        pt.append(ts)
        pa.append(rng.uniform(AMP_LO, AMP_HI, ws.size))
        return ws, ts

    tracks = []
    for _ in range(n_tracks):
        w0, w1 = rng.uniform(0, nwires, 2)
        t0, t1 = rng.uniform(0, nticks, 2)
        tracks.append(add_segment(w0, t0, w1, t1))
    michels = []
    for _ in range(n_michel):
        w0 = rng.uniform(0, nwires)
        t0 = rng.uniform(0, nticks)
        ang = rng.uniform(0, 2 * math.pi)
        length = rng.uniform(5, 20)
        w1 = w0 + length * math.cos(ang)
        t1 = t0 + TICKS_PER_WIRE * length * math.sin(ang)
        michels.append(add_segment(w0, t0, w1, t1))

    hits, kinds = [], []

    def sample_on(objs, n, kind):
        objs = [o for o in objs if o[0].size > 0]
        if n <= 0:
            return
        if not objs:
            raise ValueError("no object crosses a wire; cannot place hits")
        which = rng.integers(0, len(objs), n)
        for k in range(len(objs)):
            sel = np.nonzero(which == k)[0]
            if sel.size == 0:
                continue
            ws, ts = objs[k]
            j = rng.integers(0, ws.size, sel.size)
            hits.append(np.stack([ws[j], np.rint(ts[j]).astype(np.int64)], 1))
            kinds.append(np.full(sel.size, kind, np.int8))

    sample_on(tracks, hits_track, 0)
    sample_on(michels, hits_michel, 2)

    # EM showers: every hit is its own deposit
    if hits_shower > 0:
        if n_showers <= 0:
            raise ValueError("shower hits requested without showers")
        per = np.bincount(rng.integers(0, n_showers, hits_shower), minlength=n_showers)
        for s in range(n_showers):
            wa = rng.uniform(0, nwires)
            ta = rng.uniform(0, nticks)
            th = rng.uniform(0, 2 * math.pi)
            L = rng.uniform(50, 200)
            got = []
            need = int(per[s])
            while need > 0:
                m = 2 * need + 8
                d = rng.uniform(0, L, m)
                u = rng.standard_normal(m) * d * math.tan(SHOWER_HALF_ANGLE)
                w = wa + d * math.cos(th) - u * math.sin(th)
                t = ta + TICKS_PER_WIRE * (d * math.sin(th) + u * math.cos(th))
                wi = np.rint(w).astype(np.int64)
                ok = (wi >= 0) & (wi < nwires) & (t >= 0) & (t <= nticks - 1)
                wi, t = wi[ok][:need], t[ok][:need]
                if wi.size == 0 and not ok.any():
                    # shower fully outside the plane: re-centre it
                    wa = rng.uniform(0, nwires)
                    ta = rng.uniform(0, nticks)
                    continue
                got.append((wi, t))
                need -= wi.size
            wi = np.concatenate([g[0] for g in got])
            t = np.concatenate([g[1] for g in got])
            pw.append(wi)
            pt.append(t)
            pa.append(rng.uniform(AMP_LO, AMP_HI, wi.size))
            hits.append(np.stack([wi, np.rint(t).astype(np.int64)], 1))
            kinds.append(np.full(wi.size, 1, np.int8))

    pulses = _pulses(nwires, ld, np.concatenate(pw) if pw else [], np.concatenate(pt) if pt else [],
                     np.concatenate(pa) if pa else [])
    adc[:, :nticks] = (adc[:, :nticks].astype(np.float64) + pulses[:, :nticks]).astype(np.float32)

    if hits:
        h = np.concatenate(hits).astype(np.int32)
        k = np.concatenate(kinds)
        order = rng.permutation(h.shape[0])
        h, k = np.ascontiguousarray(h[order]), k[order]
    else:
        h, k = np.zeros((0, 2), np.int32), np.zeros(0, np.int8)
    return Plane(adc=adc, nticks=nticks, hits=h, kind=k)


def _split(total, fracs):
    counts = [int(round(total * f)) for f in fracs]
    counts[0] += total - sum(counts)
    return counts


# ---------------------------------------------------------------- workloads
def single_plane(seed: int = 0, nwires: int = 480, nhits: int = 256, n_tracks: int = 5,
                 nticks: int = NTICKS) -> Plane:
    """One collection plane, hits sampled on straight tracks only
    (480 wires x 6000 ticks, 5 tracks, 256 hits by default)."""
    rng = np.random.default_rng(seed)
    return make_plane(rng, nwires, nticks, n_tracks=n_tracks, n_showers=0, hits_track=nhits)


def apa(seed: int = 0, wires=(800, 800, 480), hits=(7692, 7692, 4616),
        fracs=(0.7, 0.3, 0.0), n_tracks=30, n_showers=5, n_michel=0,
        rng: np.random.Generator | None = None) -> list[Plane]:
    """One APA: three planes, hits split over planes in proportion to wires
    and over tracks/showers/Michel-like segments by ``fracs``."""
    rng = np.random.default_rng(seed) if rng is None else rng
    planes = []
    for nw, nh in zip(wires, hits):
        ht, hs, hm = _split(nh, fracs)
        planes.append(make_plane(rng, nw, NTICKS, n_tracks=n_tracks, n_showers=n_showers,
                                 n_michel=n_michel, hits_track=ht, hits_shower=hs, hits_michel=hm))
    return planes


def full_event(seed: int = 0, n_apa: int = 6) -> list[Plane]:
    """Full synthetic event: 6 APAs x (800, 800, 960) wires = 18 planes,
    15,360 wires, 6000 ticks; 10,000 hits per APA split 3125/3125/3750,
    60% track, 30% shower, 10% Michel-like."""
    rng = np.random.default_rng(seed)
    planes = []
    for _ in range(n_apa):
        planes += apa(wires=(800, 800, 960), hits=(3125, 3125, 3750), fracs=(0.6, 0.3, 0.1),
                      n_tracks=30, n_showers=5, n_michel=10, rng=rng)
    return planes


def inference_patches(n: int, seed: int = 0) -> np.ndarray:
    """Pre-extracted 48x48 float32 patches: 70% zeros, the rest
    exp(N(2, 1)) (lognormal mu=2 sigma=1)."""
    rng = np.random.default_rng(seed)
    mask = rng.random((n, PATCH, PATCH)) < 0.3
    val = np.exp(rng.normal(2.0, 1.0, (n, PATCH, PATCH)))
    return np.where(mask, val, 0.0).astype(np.float32)


def scaled(plane: Plane, factor: float) -> Plane:
    """The same plane with ADC multiplied by ``factor`` (unsaturated tests)."""
    return Plane(adc=(plane.adc * np.float32(factor)).astype(np.float32), nticks=plane.nticks,
                 hits=plane.hits.copy(), kind=plane.kind.copy())

