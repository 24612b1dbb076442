"""Bit-exact probe of the window read inside the tensor-core kernel (Sec. 2.1
patch definition, as the fused bf16 / fp16 / fp8 network path performs it).

The tensor-core path never writes patches: its builder warps read each hit's
48 x 48 window straight from the plane's interval image (aligned 16-byte
loads, then selects and a funnel shift for the window's phase; a per-pixel
checked read for hits outside their plane).  The score tolerances of the
network tests cannot see a misplaced pixel, so this test makes each logit an
exact, decodable function of known window pixels:

* plane: every time interval of every wire holds a small integer v in 0..15
  (its six ticks are v+a, v-a, v+b, v-b, v, v, so the fp32 sum and the
  division by 6 are exact), the ticks of the trailing partial interval hold
  1e30 (they must never be read);
* conv: filter 5i + j is one-hot at tap (i, j), bias 0, so conv map 5i + j at
  position (y, x) is the pixel (y + i, x + j), an exact 16-bit value;
* dense-1: neuron L sums six chosen (position, filter) inputs with weights
  2^(4k - 8), k = 0..5 (three inputs, k = 0..2, in e4m3), so it holds
  sum_k 2^(4k-8) p_k exactly (fewer than 24 significant bits);
* dense-2 and the heads pass neuron L through to logit L.

In tf32 (split fp16 heads and tails) every value above is an fp16 head with
a zero tail, after the power-of-two scales, so the sums stay exact; that
path reads its windows with code of its own (32-bit pixels), probed here over
every pixel as bf16's is.

The logits must then equal, bit for bit, the same sums of the oracle's patch
pixels; the oracle's own fp64 network on the same weights must agree too
(a check of the test's decoding).  Across the contexts every pixel of the
window is probed, through taps that vary over all 25, for hits at every
phase of the image row (e0 % 8), hits whose window reaches into the zero
border, hits outside the plane, and through pre-cut patches.

Each probe runs twice: alone (a small launch, whose interval image is built
from the whole plane) and batched with a 105.6 MB plane holding one hit (a
launch large enough that only the image tiles some window touches are
built).  Before the second, two decoy calls on the same context fill the
image area with other values: one with a plane of another size and row
pitch, so that most of what becomes the probe image's zero border holds
data, then one with the probe plane's own layout whose windows rebuild every
tile that holds probe pixels.  A tile that a window reads but the marking
missed would then still hold decoy values.
"""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

NW, NT = 101, 2399          # 399 complete intervals and a partial one (5 ticks)
NINT = NT // 6
BIG_NW, BIG_NT = 4400, 6000  # 105.6 MB of ADC: a launch holding it cuts only the touched image tiles


@pytest.fixture(scope="module")
def emtk():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2009_04509_gb300 import build, emtk as m
    build.build()
    oracle.build()
    return m


@pytest.fixture(scope="module")
def big(emtk):
    adc = torch.zeros((BIG_NW, BIG_NT), dtype=torch.float32, device="cuda")
    hits = torch.tensor([[BIG_NW // 2, BIG_NT // 2]], dtype=torch.int32, device="cuda")
    return adc, hits


def probe_plane(seed=77):
    rng = np.random.default_rng(seed)
    v = rng.integers(0, 16, (NW, NINT)).astype(np.float32)
    a = rng.integers(0, 4, (NW, NINT)).astype(np.float32)
    b = rng.integers(0, 4, (NW, NINT)).astype(np.float32)
    ticks = np.stack([v + a, v - a, v + b, v - b, v, v], axis=2).reshape(NW, NINT * 6)
    adc = np.full((NW, 2404), 1e30, np.float32)     # ld > nticks; poison past the complete intervals
    adc[:, :NINT * 6] = ticks
    return adc, v


def probe_hits():
    h = []
    for m in range(8):                   # interior hits at every phase of the interval (e0 % 8)
        for w in (30, 50, 70):
            h.append([w, 6 * (8 * (10 + w % 7) + m) + (w % 6)])
    for w, b in [(0, 0), (NW - 1, NINT - 1), (0, NINT - 1), (NW - 1, 0), (3, 5), (97, 391), (23, 23),
                 (24, 24), (77, 376), (50, 1), (50, NINT - 2), (1, 200), (NW - 2, 200)]:
        h.append([w, 6 * b + 5])           # in the plane, window reaching into the zero border
    for w, t in [(-1, 600), (NW, 600), (50, -1), (50, NT), (50, 6 * NINT), (-24, 700), (-23, 700),
                 (NW + 23, 900), (NW + 24, 900), (-500, -500), (60, 10 ** 7), (-3, 6 * 397 + 2)]:
        h.append([w, t])                   # outside the plane: the checked read
    h = np.array(h, np.int32)
    reps = -(-150 // len(h))
    return np.concatenate([h] * reps)[:150]   # two 128-hit tiles, the second ragged


DA_NW, DA_NT, DA_LD = NW + 48, NT + 240, 2644   # the first decoy's plane: other rows, other pitch


def decoy_a():
    """A plane of another shape and windows covering all of its image."""
    adc = np.random.default_rng(79).integers(1, 16, (DA_NW, DA_LD)).astype(np.float32)
    hits = [[w, 6 * b + 3] for w in range(0, DA_NW + 48, 40) for b in range(0, DA_NT // 6 + 48, 40)]
    return adc, np.array(hits, np.int32)


def decoy_b_hits():
    """Windows of in-plane hits covering every image tile that holds probe
    pixels (wires 0..NW-1, intervals 0..NINT-1) and fewer of the border tiles."""
    ws = [24, 64, NW - 24]
    bs = list(range(24, NINT - 24, 40)) + [NINT - 24]
    return np.array([[w, 6 * b + 3] for w in ws for b in bs], np.int32)


def probe_pixels(per_logit):
    """Every window pixel once, in groups of 4 logits x per_logit pixels."""
    order = np.random.default_rng(5).permutation(48 * 48)
    group = 4 * per_logit
    return [order[i:i + group] for i in range(0, order.size, group)]


def tap_for(r, c):
    """A tap (i, j) reading pixel (r, c) from a valid conv position; varied over the 25 taps."""
    i = min(max((r + c) % 5, r - 43, 0), r, 4)
    j = min(max((r + 2 * c) % 5, c - 43, 0), c, 4)
    return i, j


def probe_weights(pixels, per_logit):
    w = {"conv_w": np.zeros((5, 5, 1, 48), np.float32), "conv_b": np.zeros(48, np.float32),
         "fc1_w": np.zeros((92928, 128), np.float32), "fc1_b": np.zeros(128, np.float32),
         "fc2_w": np.zeros((128, 32), np.float32), "fc2_b": np.zeros(32, np.float32),
         "cls_w": np.zeros((32, 3), np.float32), "cls_b": np.zeros(3, np.float32),
         "mic_w": np.zeros((32, 1), np.float32), "mic_b": np.zeros(1, np.float32)}
    for i in range(5):
        for j in range(5):
            w["conv_w"][i, j, 0, 5 * i + j] = 1.0
    where = []
    for idx, pix in enumerate(pixels):
        L, k = divmod(idx, per_logit)
        r, c = divmod(int(pix), 48)
        i, j = tap_for(r, c)
        y, x = r - i, c - j
        w["fc1_w"][(y * 44 + x) * 48 + 5 * i + j, L] = 2.0 ** (4 * k - 8)
        where.append((L, k, r, c))
    for L in range(4):
        w["fc2_w"][L, L] = 1.0
    for L in range(3):
        w["cls_w"][L, L] = 1.0
    w["mic_w"][3, 0] = 1.0
    return w, where


def expected_logits(patches, where, n):
    z = np.zeros((n, 4), np.float64)
    for L, k, r, c in where:
        z[:, L] += 2.0 ** (4 * k - 8) * patches[:, r, c].astype(np.float64)
    return z


@pytest.mark.parametrize("prec", ["bf16", "fp16", "fp8", "tf32"])
def test_window_read_bit_exact(emtk, big, prec):
    adc_np, _ = probe_plane()
    hits_np = probe_hits()
    n = hits_np.shape[0]
    want_p = oracle.extract_patches(adc_np, NT, hits_np)
    # the probe plane really holds small integers (the test's own premise)
    assert np.array_equal(want_p, np.round(want_p)) and want_p.min() >= 0 and want_p.max() <= 15
    adc = torch.from_numpy(adc_np).cuda()
    hits = torch.from_numpy(hits_np).cuda()
    patches = torch.from_numpy(want_p).cuda()
    da_np, da_hits_np = decoy_a()
    da, da_hits = torch.from_numpy(da_np).cuda(), torch.from_numpy(da_hits_np).cuda()
    db_np, _ = probe_plane(seed=78)
    assert (db_np[:, :NINT * 6] != adc_np[:, :NINT * 6]).any()
    db, db_hits = torch.from_numpy(db_np).cuda(), torch.from_numpy(decoy_b_hits()).cuda()
    big_adc, big_hits = big
    big_out = torch.empty((1, 8), dtype=torch.float32, device="cuda")
    da_out = torch.empty((da_hits.shape[0], 8), dtype=torch.float32, device="cuda")
    db_out = torch.empty((db_hits.shape[0], 8), dtype=torch.float32, device="cuda")
    per_logit = 3 if prec == "fp8" else 6
    groups = probe_pixels(per_logit)
    if prec in ("fp16", "fp8"):
        groups = groups[::7]               # the window read of bf16, fp16 and fp8 is one code
    for gi, pixels in enumerate(groups):
        w, where = probe_weights(pixels, per_logit)
        ctx = emtk.emtk_create(w, precision=prec, debug_logits=True, max_hits=256)
        try:
            out = torch.full((n, 8), float("nan"), dtype=torch.float32, device="cuda")
            emtk.emtk_infer(ctx, adc, NT, hits, out)
            emtk.emtk_infer_batch(ctx, [(da, DA_NT, da_hits, da_out), (big_adc, BIG_NT, big_hits, big_out)])
            emtk.emtk_infer_batch(ctx, [(db, NT, db_hits, db_out), (big_adc, BIG_NT, big_hits, big_out)])
            tiled = torch.full((n, 8), float("nan"), dtype=torch.float32, device="cuda")
            emtk.emtk_infer_batch(ctx, [(adc, NT, hits, tiled), (big_adc, BIG_NT, big_hits, big_out)])
            # the pre-cut patch path reads the same windows (from the fp32 patches themselves)
            via_patches = torch.full((n, 8), float("nan"), dtype=torch.float32, device="cuda")
            emtk.emtk_infer_patches(ctx, patches, via_patches)
            assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        finally:
            emtk.emtk_destroy(ctx)
        got = out[:, 4:].cpu().numpy().astype(np.float64)
        want = expected_logits(want_p, where, n)
        bad = np.argwhere(got != want)
        assert bad.size == 0, (f"{prec}, pixel group {gi}: {len(bad)} logits differ, first at hit "
                               f"{hits_np[bad[0][0]].tolist()} logit {bad[0][1]}: {got[tuple(bad[0])]} "
                               f"!= {want[tuple(bad[0])]}")
        got_t = tiled[:, 4:].cpu().numpy().astype(np.float64)
        bad = np.argwhere(got_t != want)
        assert bad.size == 0, (f"{prec}, tiled cut, pixel group {gi}: {len(bad)} logits differ, first at hit "
                               f"{hits_np[bad[0][0]].tolist()} logit {bad[0][1]}: {got_t[tuple(bad[0])]} "
                               f"!= {want[tuple(bad[0])]}")
        assert np.array_equal(via_patches[:, 4:].cpu().numpy().astype(np.float64), want), \
            f"{prec}, pre-cut patches, pixel group {gi}"
        if gi % 16 == 0:                   # the oracle's own network on these weights gives the same sums
            lo, _ = oracle.forward(want_p, w)
            assert np.array_equal(lo, want)


def rounding_patches(n, fmt, seed):
    """Positive fp32 patch values (the conv's ReLU keeps them) that need rounding
    to 16 bit: random ones, and as many exact halfway cases of the format, with
    the kept part's last bit even and odd."""
    rng = np.random.default_rng(seed)
    x = np.exp2(rng.uniform(-6.0, 10.0, (n, 48, 48))).astype(np.float32)
    b = x.view(np.uint32)
    tie = rng.random((n, 48, 48)) < 0.5
    if fmt == "bf16":   # 16 dropped bits: halfway is 0x8000
        b[tie] = (b[tie] & np.uint32(0xFFFF0000)) | np.uint32(0x8000)
    else:               # fp16 keeps 10 of fp32's 23 mantissa bits here: halfway is 0x1000
        b[tie] = (b[tie] & np.uint32(0xFFFFE000)) | np.uint32(0x1000)
    return b.view(np.float32)


@pytest.mark.parametrize("prec", ["bf16", "fp16"])
def test_precut_patch_rounding_bit_exact(emtk, prec):
    """The 16-bit network kernels round pre-cut fp32 patches as they load them:
    to nearest, ties to even, as the oracle's rounding.  With one pixel per logit
    (weights as in the window probe, the dense-1 weight 2^-8), each logit is
    2^-8 times that pixel rounded, exactly."""
    n = 300
    x = rounding_patches(n, prec, seed=93 if prec == "bf16" else 94)
    if prec == "bf16":
        r = (oracle.round_bf16(x).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    else:
        r = oracle.round_fp16(x).astype(np.float64)
    assert (r != x).mean() > 0.5      # most values are changed by the rounding
    xd = torch.from_numpy(x).cuda()
    groups = probe_pixels(1)[::48]     # 12 contexts of 4 pixels, spread over the window
    for gi, pixels in enumerate(groups):
        w, where = probe_weights(pixels, 1)
        ctx = emtk.emtk_create(w, precision=prec, debug_logits=True, max_hits=512)
        try:
            out = torch.full((n, 8), float("nan"), dtype=torch.float32, device="cuda")
            emtk.emtk_infer_patches(ctx, xd, out)
            assert emtk.emtk_check(ctx) == emtk.EMTK_OK
        finally:
            emtk.emtk_destroy(ctx)
        got = out[:, 4:].cpu().numpy().astype(np.float64)
        want = np.zeros((n, 4))
        for L, k, rr, cc in where:
            want[:, L] += 2.0 ** (4 * k - 8) * r[:, rr, cc]
        bad = np.argwhere(got != want)
        assert bad.size == 0, (f"{prec}, group {gi}: {len(bad)} logits differ, first hit {bad[0][0]} logit "
                               f"{bad[0][1]}: {got[tuple(bad[0])]} != {want[tuple(bad[0])]}")
