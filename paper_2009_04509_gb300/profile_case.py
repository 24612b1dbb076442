"""Profiling driver: a small, self-checking run of the hot path to capture
with ncu.  A tool, not part of the library: nothing in the package imports
it; the commands in profiles/ run it.

    python -m paper_2009_04509_gb300.profile_case --mode event   # one APA, 20,000 hits
    python -m paper_2009_04509_gb300.profile_case --mode patches --hits 30000
    python -m paper_2009_04509_gb300.profile_case --mode hitfind          # full event, threshold 15

`event` runs one APA (6 planes, 800/800/480 wires x 6000 ticks, 20,000 hits)
through emtk_infer_batch, the call the benchmark times on a full event;
`patches` runs N pre-cut patches through emtk_infer_patches; `hitfind` runs
emtk_find_hits on the 18 planes of the full event (368.6 MB of samples) and
checks the hit counts against a first run.  The path runs
twice (capture the second launch with `ncu -s 1 -c 1`), and the context's
status word is checked, so that a run that ends with exit code 0 was a
correct, complete one.  Inputs are synthetic and seeded; the device holds a
few hundred MB.
"""
from __future__ import annotations

import argparse
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from paper_2009_04509_gb300 import emtk, synth  # noqa: E402


def main() -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--mode", default="event", choices=["event", "patches", "hitfind"])
    ap.add_argument("--hits", type=int, default=30000, help="patches mode: number of patches")
    ap.add_argument("--precision", default="bf16", choices=["bf16", "fp16", "fp8", "fp32", "tf32"])
    ap.add_argument("--runs", type=int, default=2)
    args = ap.parse_args()

    import torch
    dev = torch.device("cuda:0")
    w = synth.he_normal_weights(0)
    if args.mode == "hitfind":
        planes = synth.full_event(seed=0)
        ctx = emtk.emtk_create(w, precision="bf16")
        cap = 262_144
        items = [(torch.from_numpy(p.adc).to(dev), p.nticks, 15.0, torch.empty((cap, 2), dtype=torch.int32, device=dev),
                  torch.empty((cap, 4), dtype=torch.int32, device=dev)) for p in planes]
        try:
            counts = [emtk.emtk_find_hits(ctx, items) for _ in range(args.runs)]
        finally:
            emtk.emtk_destroy(ctx)
        if any(c != counts[0] for c in counts):
            print("hit counts differ between runs", file=sys.stderr)
            return 1
        print(f"ok: hitfind, {sum(counts[0])} hits on {len(planes)} planes, {args.runs} runs")
        return 0
    if args.mode == "event":
        planes = synth.apa(seed=0)
        ctx = emtk.emtk_create(w, precision=args.precision)
        items = [(torch.from_numpy(p.adc).to(dev), p.nticks, torch.from_numpy(p.hits).to(dev),
                  torch.zeros((p.nhits, 4), device=dev)) for p in planes]
        n = sum(p.nhits for p in planes)
        run = lambda: emtk.emtk_infer_batch(ctx, items)  # noqa: E731
    else:
        n = args.hits
        ctx = emtk.emtk_create(w, precision=args.precision, max_hits=min(n, 1 << 20))
        x = torch.from_numpy(synth.inference_patches(n, seed=1)).to(dev)
        sc = torch.zeros((n, 4), device=dev)
        run = lambda: emtk.emtk_infer_patches(ctx, x, sc)  # noqa: E731
    try:
        for _ in range(args.runs):
            run()
        rc = emtk.emtk_check(ctx)
    finally:
        emtk.emtk_destroy(ctx)
    if rc != emtk.EMTK_OK:
        print(f"status {emtk.status_string(rc)}", file=sys.stderr)
        return 1
    print(f"ok: {args.mode}, {n} hits, {args.precision}, {args.runs} runs")
    return 0


if __name__ == "__main__":
    sys.exit(main())
