"""Pins for the CPU oracle: facts fixed by the paper and by mathematics,
checked without the oracle restating itself.

* shapes and the parameter count printed in Sec. 2.2, and the 4.1 Gbit per
  event of Sec. 3.3 (tests/golden/paper_facts.json);
* the patch cut of Sec. 2.1 on planes whose interval means are known in
  closed form (constant, ramps, impulses), at the plane's edges, beyond them,
  with a trailing partial interval and with negative ticks, and against a
  brute-force numpy/slicing restatement;
* each layer of Sec. 2.2 against a library routine that computes the same
  thing (scipy.signal.correlate2d, numpy matmul, scipy.special.softmax and
  expit), and the whole network against their composition;
* special cases: zero weights give exactly 1/3 and 1/2, a one-hot dense-1
  weight pins the flatten order.

``test_planted_mistakes`` compiles copies of the oracle with one plausible
mistake each and checks that some pin here fails on every copy.
"""
import json
import os
import shutil
import subprocess

import numpy as np
import pytest
import scipy.signal
import scipy.special

import oracle
from paper_2009_04509_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_facts.json")
FACTS = {k: v["value"] for k, v in json.load(open(GOLDEN)).items() if not k.startswith("_")}


# ------------------------------------------------------------------ helpers
def seq_interval_means(adc, nticks, ds=6):
    """Brute force: the fp32 left-to-right sum of each 6-tick interval,
    divided once by 6, for every complete interval of every wire."""
    nint = nticks // ds
    a = adc[:, : nint * ds].reshape(adc.shape[0], nint, ds).astype(np.float32)
    s = a[:, :, 0].copy()
    for j in range(1, ds):
        s = (s + a[:, :, j]).astype(np.float32)
    return (s / np.float32(ds)).astype(np.float32)


def brute_patches(adc, nticks, hits, psize=48, ds=6):
    """Brute force: pad the interval-mean image with zeros and slice windows."""
    D = seq_interval_means(adc, nticks, ds)
    half = psize // 2
    pad = psize + 8 + int(np.abs(hits).max() if hits.size else 0) // ds
    Dp = np.zeros((D.shape[0] + 2 * pad, D.shape[1] + 2 * pad), np.float32)
    Dp[pad: pad + D.shape[0], pad: pad + D.shape[1]] = D
    out = np.zeros((hits.shape[0], psize, psize), np.float32)
    for h, (w, t) in enumerate(hits):
        b = int(np.floor(t / ds))
        r0, c0 = w - half + pad, b - half + pad
        if r0 < 0 or c0 < 0 or r0 + psize > Dp.shape[0] or c0 + psize > Dp.shape[1]:
            continue  # fully outside the padded image: stays zero
        out[h] = Dp[r0: r0 + psize, c0: c0 + psize]
    return out


def library_forward(patches, wt, dims):
    """The network of Sec. 2.2 composed from library routines (float64)."""
    P, R, F = dims["P"], dims["R"], dims["F"]
    Q = P - R + 1
    cw = wt["conv_w"].astype(np.float64).reshape(R, R, F)
    outs_l, outs_s = [], []
    for img in patches.astype(np.float64):
        maps = np.stack([scipy.signal.correlate2d(img, cw[:, :, f], mode="valid") for f in range(F)], -1)
        act = np.maximum(maps + wt["conv_b"].astype(np.float64), 0.0).reshape(Q * Q * F)
        h1 = np.maximum(act @ wt["fc1_w"].astype(np.float64) + wt["fc1_b"], 0.0)
        h2 = np.maximum(h1 @ wt["fc2_w"].astype(np.float64) + wt["fc2_b"], 0.0)
        z = h2 @ wt["cls_w"].astype(np.float64) + wt["cls_b"]
        m = (h2 @ wt["mic_w"].astype(np.float64) + wt["mic_b"])[0]
        outs_l.append(np.concatenate([z, [m]]))
        outs_s.append(np.concatenate([scipy.special.softmax(z), [scipy.special.expit(m)]]))
    return np.array(outs_l), np.array(outs_s)


TINY = dict(P=9, R=3, F=4, N1=6, N2=5, NC=3)


# --------------------------------------------------------------------- pins
def pin_parameter_count(lib):
    w = synth.he_normal_weights(0)
    assert synth.parameter_count(w) == FACTS["trainable_parameters"]
    P, R, F = FACTS["patch_side"], FACTS["conv_kernel"], FACTS["conv_filters"]
    Q = (P - R) // FACTS["conv_stride"] + 1
    assert Q == FACTS["conv_map_side"]
    n = (R * R * F + F) + (Q * Q * F * FACTS["fc1_width"] + FACTS["fc1_width"]) + \
        (FACTS["fc1_width"] * FACTS["fc2_width"] + FACTS["fc2_width"]) + \
        (FACTS["fc2_width"] * FACTS["softmax_outputs"] + FACTS["softmax_outputs"]) + \
        (FACTS["fc2_width"] * FACTS["sigmoid_outputs"] + FACTS["sigmoid_outputs"])
    assert n == FACTS["trainable_parameters"]


def pin_conv_shape(lib):
    rng = np.random.default_rng(1)
    img = rng.standard_normal((48, 48))
    out = oracle.conv_relu(img, rng.standard_normal((5, 5, 48)), np.zeros(48), lib=lib)
    assert out.shape == (FACTS["conv_map_side"], FACTS["conv_map_side"], FACTS["conv_filters"])
    assert out.size == 92928


def pin_constant_plane(lib):
    for a in (7.0, 3.25, -1.5):
        adc = np.full((100, 600), a, np.float32)
        hits = np.array([[50, 300]], np.int32)
        p = oracle.extract_patches(adc, 600, hits, lib=lib)[0]
        assert np.all(p == np.float32(a))
        # hit at wire 0, tick 0: wires -24..-1 and intervals -24..-1 are zero
        p = oracle.extract_patches(adc, 600, np.array([[0, 0]], np.int32), lib=lib)[0]
        assert np.all(p[:24, :] == 0) and np.all(p[:, :24] == 0)
        assert np.all(p[24:, 24:] == np.float32(a))


def pin_ramps(lib):
    nw, nt = 70, 600
    tick_ramp = np.tile(np.arange(nt, dtype=np.float32), (nw, 1))
    wire_ramp = np.tile(np.arange(nw, dtype=np.float32)[:, None], (1, nt))
    hits = np.array([[35, 301], [30, 150]], np.int32)
    p = oracle.extract_patches(tick_ramp, nt, hits, lib=lib)
    for h, (w, t) in enumerate(hits):
        bc = t // 6
        for c in range(48):
            b = bc - 24 + c
            # mean of 6b..6b+5 = 6b + 2.5
            expect = np.float32(6 * b + 2.5) if 0 <= b < nt // 6 else 0.0
            rows = [r for r in range(48) if 0 <= w - 24 + r < nw]
            assert np.all(p[h, rows, c] == expect)
    p = oracle.extract_patches(wire_ramp, nt, hits, lib=lib)
    for h, (w, t) in enumerate(hits):
        for r in range(48):
            wr = w - 24 + r
            expect = np.float32(wr) if 0 <= wr < nw else 0.0
            assert np.all(p[h, r, :] == expect)


def pin_impulse(lib):
    adc = np.zeros((60, 600), np.float32)
    adc[31, 299] = 6.0            # interval 49
    hits = np.array([[30, 290]], np.int32)   # interval 48: pixel row 25, col 25
    p = oracle.extract_patches(adc, 600, hits, lib=lib)[0]
    nz = np.argwhere(p != 0)
    assert nz.tolist() == [[25, 25]] and p[25, 25] == np.float32(1.0)


def pin_outside_and_partial(lib):
    rng = np.random.default_rng(2)
    nw, nticks, ld = 40, 597, 600          # 99 complete intervals, ticks 594..596 partial
    adc = rng.standard_normal((nw, ld)).astype(np.float32)
    adc[:, nticks:] = 1e30                  # data beyond nticks must never be read
    hits = np.array([[-100, 300], [20, 10_000], [20, 596], [39, 594]], np.int32)
    p = oracle.extract_patches(adc, nticks, hits, lib=lib)
    assert np.all(p[0] == 0) and np.all(p[1] == 0)
    # hit at tick 596 -> interval 99 (partial, absent) at column 24: columns >= 24 are zero
    assert np.all(p[2][:, 24:] == 0) and np.any(p[2][:, :24] != 0)
    assert np.all(np.abs(p) < 1e29)


def pin_negative_ticks(lib):
    nw, nt = 50, 600
    tick_ramp = np.tile(np.arange(nt, dtype=np.float32), (nw, 1)) + 1.0
    # tick -1 lies in interval -1 (floor), so interval 0 appears at column 25
    p = oracle.extract_patches(tick_ramp, nt, np.array([[25, -1]], np.int32), lib=lib)[0]
    assert np.all(p[:, :25] == 0)
    assert np.all(p[1:, 25] == np.float32(3.5))   # (1+2+...+6)/6


def pin_patches_brute_force(lib):
    rng = np.random.default_rng(3)
    for nw, nticks, ld in ((37, 301, 304), (64, 600, 600)):
        adc = (rng.standard_normal((nw, ld)) * 50).astype(np.float32)
        hits = np.stack([rng.integers(-30, nw + 30, 60), rng.integers(-200, nticks + 200, 60)], 1).astype(np.int32)
        hits = np.concatenate([hits, hits[:3]])   # duplicates are ordinary hits
        got = oracle.extract_patches(adc, nticks, hits, lib=lib)
        want = brute_patches(adc, nticks, hits)
        assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def pin_conv_library(lib):
    rng = np.random.default_rng(4)
    for P, R, F in ((9, 3, 4), (48, 5, 48)):
        img = rng.standard_normal((P, P))
        w = rng.standard_normal((R, R, F))
        b = rng.standard_normal(F)
        got = oracle.conv_relu(img, w, b, lib=lib)
        want = np.stack([scipy.signal.correlate2d(img, w[:, :, f], mode="valid") for f in range(F)], -1)
        np.testing.assert_allclose(got, np.maximum(want + b, 0.0), rtol=1e-12, atol=1e-12)


def pin_dense_library(lib):
    rng = np.random.default_rng(5)
    for K, N in ((7, 5), (1000, 128)):
        x = rng.standard_normal(K)
        W = rng.standard_normal((K, N)).astype(np.float32)
        b = rng.standard_normal(N).astype(np.float32)
        for relu in (False, True):
            want = x @ W.astype(np.float64) + b
            want = np.maximum(want, 0.0) if relu else want
            np.testing.assert_allclose(oracle.dense(x, W, b, relu, lib=lib), want, rtol=1e-12, atol=1e-11)


def pin_heads(lib):
    for z, m in (([0.3, -1.2, 2.0], 0.7), ([800.0, 0.0, -5.0], -40.0), ([0.0, 0.0, 0.0], 0.0)):
        s = oracle.heads(np.array(z), m, lib=lib)
        np.testing.assert_allclose(s[:3], scipy.special.softmax(z), rtol=1e-13, atol=1e-300)
        np.testing.assert_allclose(s[3], scipy.special.expit(m), rtol=1e-13)
        assert abs(s[:3].sum() - 1.0) < 1e-12 and 0.0 <= s[3] <= 1.0


def pin_forward_library(lib):
    rng = np.random.default_rng(6)
    wt = synth.he_normal_weights(7, bias_std=0.1, dims=TINY)
    x = (rng.standard_normal((5, TINY["P"], TINY["P"])) * 3).astype(np.float32)
    lo, sc = oracle.forward(x, wt, dims=TINY, lib=lib)
    wl, ws = library_forward(x, wt, TINY)
    np.testing.assert_allclose(lo, wl, rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(sc, ws, rtol=1e-10, atol=1e-12)


def pin_forward_full_size(lib):
    rng = np.random.default_rng(8)
    wt = synth.he_normal_weights(0, bias_std=0.1)
    x = synth.inference_patches(2, seed=9) * np.float32(0.05)
    x[1] = (rng.standard_normal((48, 48)) * 2).astype(np.float32)
    lo, sc = oracle.forward(x, wt, lib=lib)
    wl, ws = library_forward(x, wt, oracle.EMTK_DIMS)
    np.testing.assert_allclose(lo, wl, rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(sc, ws, rtol=1e-9, atol=1e-12)


def pin_zero_weights(lib):
    wt = {k: np.zeros_like(v) for k, v in synth.he_normal_weights(0, dims=TINY).items()}
    x = np.ones((3, TINY["P"], TINY["P"]), np.float32)
    lo, sc = oracle.forward(x, wt, dims=TINY, lib=lib)
    assert np.all(lo == 0.0)
    assert np.all(sc[:, :3] == 1.0 / 3.0) and np.all(sc[:, 3] == 0.5)


def pin_flatten_order(lib):
    d = dict(P=12, R=5, F=6, N1=4, N2=3, NC=3)
    Q = d["P"] - d["R"] + 1
    rng = np.random.default_rng(10)
    wt = synth.he_normal_weights(3, dims=d)
    y, x, c = 2, 5, 4
    wt["fc1_w"][:] = 0
    wt["fc1_w"][(y * Q + x) * d["F"] + c, 1] = 1.0    # dense-1 unit 1 reads map c at (y, x)
    wt["fc2_w"][:] = 0
    wt["fc2_w"][1, 0] = 1.0
    wt["cls_w"][:] = 0
    wt["cls_w"][0, 0] = 1.0
    img = (rng.standard_normal((1, d["P"], d["P"])) * 4).astype(np.float32)
    lo, _ = oracle.forward(img, wt, dims=d, lib=lib)
    ref = scipy.signal.correlate2d(img[0].astype(np.float64),
                                   wt["conv_w"][:, :, 0, c].astype(np.float64), mode="valid")[y, x]
    assert abs(lo[0, 0] - max(ref, 0.0)) < 1e-12


def pin_bf16_rounding(lib):
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(11)
    x = np.concatenate([(rng.standard_normal(4000) * 100).astype(np.float32),
                        np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 0.0, -0.0,
                                  65504.0, 1e-30], np.float32)])
    got = oracle.round_bf16(x, lib=lib)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, want)


def pin_fp16_rounding(lib):
    rng = np.random.default_rng(13)
    x = np.concatenate([(rng.standard_normal(4000) * 100).astype(np.float32),
                        (rng.standard_normal(1000) * 1e-5).astype(np.float32),
                        np.array([1.0 + 2.0 ** -11, 1.0 + 3 * 2.0 ** -11, 65504.0, 65519.0, 65520.0,
                                  -70000.0, 2.0 ** -25, 3 * 2.0 ** -26, 1e-30, 0.0], np.float32)])
    got = oracle.round_fp16(x, lib=lib)
    with np.errstate(over="ignore"):
        want = x.astype(np.float16).astype(np.float32)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def pin_transmit_volume(lib):
    bits = FACTS["patches_per_event"] * FACTS["patch_side"] ** 2 * FACTS["bits_per_pixel"]
    assert abs(bits / 1e9 - FACTS["transmit_gbit_per_event"]) < 0.06


# ------------------------------------------------------------- fp8 (e4m3)
def e4m3_table():
    """Every finite FP8 E4M3 value, from the format's definition: sign, 4-bit
    exponent (bias 7), 3-bit mantissa; exponent 0 is subnormal; the code with
    all exponent and mantissa bits set is NaN, so 448 is the largest."""
    vals = set()
    for e in range(16):
        for m in range(8):
            if e == 15 and m == 7:
                continue
            v = (m / 8.0) * 2.0 ** -6 if e == 0 else (1 + m / 8.0) * 2.0 ** (e - 7)
            vals.add(v)
            vals.add(-v)
    return np.array(sorted(vals))


def test_e4m3_table_facts():
    t = e4m3_table()
    assert t.max() == 448.0 and np.min(t[t > 0]) == 2.0 ** -9
    assert len(t) == 2 * 127 - 1  # 127 non-negative finite codes each side, +-0 merged


def pin_e4m3_rounding(lib):
    t = e4m3_table()
    # representable values map to themselves
    assert np.array_equal(oracle.round_e4m3(t.astype(np.float32), lib=lib), t.astype(np.float32))
    rng = np.random.default_rng(7)
    x = np.concatenate([rng.standard_normal(20000) * s for s in (0.003, 0.1, 3.0, 100.0)]).astype(np.float32)
    got = oracle.round_e4m3(x, lib=lib).astype(np.float64)
    xs = np.clip(x.astype(np.float64), -448.0, 448.0)
    dist = np.abs(t[None, :] - xs[:, None])
    best = dist.min(1)
    assert np.allclose(np.abs(got - xs), best, rtol=0, atol=0)  # a nearest value
    # ties (midpoints between neighbours) go to the even mantissa
    pos = t[t > 0]
    mids = ((pos[:-1] + pos[1:]) / 2).astype(np.float32)
    r = oracle.round_e4m3(mids, lib=lib).astype(np.float64)
    for mval, rv in zip(mids.astype(np.float64), r):
        lo, hi = pos[pos < mval].max(), pos[pos > mval].min()
        even = lo if int(round(lo / 2.0 ** (np.floor(np.log2(max(lo, 2.0 ** -6))) - 3))) % 2 == 0 else hi
        assert rv == even, (mval, rv, lo, hi)
    assert oracle.round_e4m3(np.array([1e4, -1e4], np.float32), lib=lib).tolist() == [448.0, -448.0]



PINS = [pin_parameter_count, pin_conv_shape, pin_constant_plane, pin_ramps, pin_impulse,
        pin_outside_and_partial, pin_negative_ticks, pin_patches_brute_force, pin_conv_library,
        pin_dense_library, pin_heads, pin_forward_library, pin_forward_full_size, pin_zero_weights,
        pin_flatten_order, pin_bf16_rounding, pin_fp16_rounding, pin_transmit_volume, pin_e4m3_rounding]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin, oracle_lib):
    pin(oracle_lib)


@pytest.mark.parametrize("mode", ["bf16", "fp16"])
def test_emulated_mode_is_rounding_only(mode, oracle_lib):
    """An emulating mode equals the plain mode on inputs that are already
    values of that format with activations that need no rounding (one-filter
    identity conv on rounded patches, rounded weights)."""
    rnd = (lambda a: (oracle.round_bf16(a).astype(np.uint32) << 16).view(np.float32).reshape(a.shape)) \
        if mode == "bf16" else (lambda a: oracle.round_fp16(a))
    rng = np.random.default_rng(12)
    d = dict(P=6, R=1, F=1, N1=4, N2=3, NC=3)
    wt = synth.he_normal_weights(5, bias_std=0.1, dims=d)
    wt["conv_w"][:] = 1.0
    wt["conv_b"][:] = 0.0
    wt["fc1_w"] = rnd(wt["fc1_w"])
    x = rnd((rng.standard_normal((4, 6, 6)) * 5).astype(np.float32))
    a = oracle.forward(x, wt, dims=d)
    b = oracle.forward(x, wt, dims=d, emulate=mode)
    assert np.array_equal(a[0], b[0])
    c = oracle.forward((rng.standard_normal((4, 6, 6)) * 5).astype(np.float32), wt, dims=d, emulate=mode)
    assert np.all(np.isfinite(c[1]))


# ---------------------------------------------------------- planted mistakes
MUTATIONS = {
    "transposed_taps": ("img[(y + i) * P + (x + j)]", "img[(y + j) * P + (x + i)]"),
    "dropped_dense_bias": ("y[n] = b ? (double)b[n] : 0.0;", "y[n] = 0.0;"),
    "off_by_one_centre": ("const int half = psize / 2;", "const int half = psize / 2 - 1;"),
    "short_interval_sum": ("for (int j = 1; j < ds; ++j)\n        s = s + a[j];",
                           "for (int j = 1; j < ds - 1; ++j)\n        s = s + a[j];"),
    "truncating_division": ("const long bc = floor_div(hits[2 * h + 1], ds);",
                            "const long bc = hits[2 * h + 1] / ds;"),
    "softmax_without_shift": ("scores[c] = exp(logits[c] - mx);", "scores[c] = exp(logits[c]);"),
    "sigmoid_sign": ("1.0 / (1.0 + exp(-logit_m))", "1.0 / (1.0 + exp(logit_m))"),
    "no_relu_after_fc2": ("or_dense(h1, N1, fc2_w, fc2_b, N2, 1, h2);",
                          "or_dense(h1, N1, fc2_w, fc2_b, N2, 0, h2);"),
    "flatten_chw": ("out[((long)y * Q + x) * F + f]", "out[((long)f * Q + y) * Q + x]"),
    "partial_interval_read": ("const long nint = nticks / ds;", "const long nint = (nticks + ds - 1) / ds;"),
    "e4m3_four_mantissa_bits": ("int qexp = e - 4;           /* 4 significant bits */",
                                "int qexp = e - 5;           /* 4 significant bits */"),
    "e4m3_no_subnormals": ("if (qexp < -9)\n        qexp = -9;", "if (qexp < -6)\n        qexp = -6;"),
    "e4m3_no_saturation": ("if (r > 448.0f)\n        r = 448.0f;", "if (r > 480.0f)\n        r = 480.0f;"),
    "wire_col_swap": ("v = interval_value(plane + w * ld, b, ds);",
                      "v = (w < nint && b < nwires) ? interval_value(plane + b * ld, w, ds) : 0.0f;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistakes(name, tmp_path, oracle_lib):
    """A copy of the oracle with one planted mistake must fail at least one pin."""
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
            with np.errstate(all="ignore"):
                pin(lib)
        except (AssertionError, ValueError, FloatingPointError):
            failed.append(pin.__name__)
    assert failed, f"planted mistake {name} passed every pin"


def test_fp8_emulation_is_rounding_only(oracle_lib):
    """The fp8 mode equals the plain mode on inputs whose bf16 conv operands,
    scaled activations and scaled dense-1 weights are already e4m3 values."""
    rng = np.random.default_rng(13)
    d = dict(P=6, R=1, F=1, N1=4, N2=3, NC=3)
    wt = synth.he_normal_weights(5, bias_std=0.1, dims=d)
    wt["conv_w"][:] = 1.0
    wt["conv_b"][:] = 0.0
    t = e4m3_table()
    sa, sw = 0.25, 16.0
    wt["fc1_w"] = (rng.choice(t[np.abs(t) <= 100], wt["fc1_w"].shape) / sw).astype(np.float32)
    x = (rng.choice(t[(t >= 0) & (t <= 200)], (4, 6, 6)) / sa).astype(np.float32)  # bf16 values too
    a = oracle.forward(x, wt, dims=d)
    b = oracle.forward(x, wt, dims=d, emulate="fp8", fp8_scales=(sa, sw))
    assert np.array_equal(a[0], b[0])
    c = oracle.forward(x * 1.1, wt, dims=d, emulate="fp8", fp8_scales=(sa, sw))  # beyond e4m3 spacing
    assert not np.array_equal(a[0], c[0]) and np.all(np.isfinite(c[1]))
