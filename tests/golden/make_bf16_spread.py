"""Write tests/golden/bf16_spread.json: on fixed seeded samples of the bf16
workloads, the per-track error of the fp32 emulation of the oracle against the
fp64 oracle, in each accumulation order (mean, 50th, 90th, 99th percentile,
maximum).

It calls only oracle/ (and the seeded input generators).  These numbers are the
spread a correct fp32-accumulating implementation with bf16 operands shows; the
GPU gate (tests/helpers.py) recomputes the same statistics on its own tracks and
allows BF16_BULK_FACTOR / BF16_MAX_FACTOR above the worse order.

  python tests/golden/make_bf16_spread.py
"""
import dataclasses
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import fp32_emulation as E  # noqa: E402
from oracle import trackfit_oracle as O  # noqa: E402
from paper_2609_32479_gb300 import workloads as W  # noqa: E402

# (workload, tracks, hit count for every track or None for the generated counts)
SAMPLES = [("medium", 300, None), ("large", 300, None), ("sweep8", 1000, None), ("sweep64", 200, None),
           ("medium", 500, 1)]


def per_track(got, ref):
    rms = np.sqrt(np.mean(ref * ref, axis=0))
    return np.max(np.abs(got - ref) / np.maximum(np.abs(ref), rms[None, :]), axis=1)


def main():
    out = {"metric": "per track: max over the 5 outputs of |g - r| / max(|r|, column RMS of r)",
           "reference": "fp64 oracle with bf16 operand rounding", "samples": []}
    for name, n, n_fixed in SAMPLES:
        w = W.workload(name, n_tracks=n)
        tb = W.gen_tracks(w)
        n_hits = tb.n_hits if n_fixed is None else np.full(n, n_fixed, np.int32)
        blob = W.gen_weights(w.model, w.weight_seed)
        cfg = dataclasses.asdict(w.model)
        ref = O.forward(cfg, blob, tb.hits, n_hits)
        entry = {"workload": name, "n_tracks": n, "hits_per_track": n_fixed}
        for order in E.ORDERS:
            e = per_track(E.forward(cfg, blob, tb.hits, n_hits, order=order), ref)
            entry[order] = {k: float(v) for k, v in (("mean", e.mean()), ("p50", np.percentile(e, 50)),
                                                     ("p90", np.percentile(e, 90)), ("p99", np.percentile(e, 99)),
                                                     ("max", e.max()))}
        out["samples"].append(entry)
        print(entry, flush=True)
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "bf16_spread.json"), "w") as fh:
        json.dump(out, fh, indent=1)


if __name__ == "__main__":
    main()
