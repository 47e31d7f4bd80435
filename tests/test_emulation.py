"""Pins for the fp32 emulation of the oracle (oracle/fp32_emulation.py), no GPU.

The emulation sets the bf16 parity bars, so it is checked against the fp64
oracle where the answer is fixed: without 16-bit operands it must agree with
the oracle to fp32 rounding (in both accumulation orders); with bf16 operands it
must round the same operands as the oracle (it lands far closer to the bf16
oracle than to the unrounded one, and a version with the rounding taken out
does not); and the spread it reports on fixed samples is the one recorded in
tests/golden/bf16_spread.json by tests/golden/make_bf16_spread.py."""
import dataclasses
import json
import os

import numpy as np
import pytest

from oracle import fp32_emulation as E
from oracle import trackfit_oracle as O
from paper_2609_32479_gb300 import workloads as W
from tests.helpers import track_errors

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "bf16_spread.json")


def _case(name, n, **kw):
    w = W.workload(name, n_tracks=n, **kw)
    tb = W.gen_tracks(w)
    return w, W.gen_weights(w.model, w.weight_seed), tb


@pytest.mark.parametrize("name,n", [("tiny", 128), ("small", 128), ("medium", 48), ("large", 24)])
@pytest.mark.parametrize("order", E.ORDERS)
def test_fp32_emulation_matches_the_oracle_without_16_bit_operands(name, n, order):
    w, blob, tb = _case(name, n, precision=W.PRECISION_FP32)
    cfg = dataclasses.asdict(w.model)
    ref = O.forward(cfg, blob, tb.hits, tb.n_hits)
    got = E.forward(cfg, blob, tb.hits, tb.n_hits, order=order)
    assert track_errors(got, ref).max() < 2e-5


def test_emulation_rounds_the_same_operands_as_the_oracle(monkeypatch):
    w, blob, tb = _case("medium", 64)
    cfg = dataclasses.asdict(w.model)
    ref16 = O.forward(cfg, blob, tb.hits, tb.n_hits)
    ref32 = O.forward(dict(cfg, precision=0), blob, tb.hits, tb.n_hits)
    em = E.forward(cfg, blob, tb.hits, tb.n_hits)
    near, far = np.median(track_errors(em, ref16)), np.median(track_errors(em, ref32))
    assert near < 0.2 * far, (near, far)
    # planted mistake: the operand rounding taken out of the emulation
    monkeypatch.setattr(E, "_op", lambda x, prec: np.asarray(x, dtype=np.float32))
    bad = E.forward(cfg, blob, tb.hits, tb.n_hits)
    assert np.median(track_errors(bad, ref16)) > 3 * near


def test_accumulation_orders_differ_only_by_rounding():
    w, blob, tb = _case("medium", 32, precision=W.PRECISION_FP32)
    cfg = dataclasses.asdict(w.model)
    a = E.forward(cfg, blob, tb.hits, tb.n_hits, order="blas")
    b = E.forward(cfg, blob, tb.hits, tb.n_hits, order="k16")
    assert 0 < np.max(np.abs(a - b)) and track_errors(a, b).max() < 2e-5


def test_recorded_bf16_spread_reproduces():
    """The first recorded sample (medium) recomputed here gives the recorded mean,
    90th percentile and maximum of the per-track error of every accumulation order
    (to 5 %: the BLAS library may block the products differently on another
    host, which moves individual rounding flips)."""
    with open(GOLDEN) as fh:
        rec = json.load(fh)
    entry = rec["samples"][0]
    w, blob, tb = _case(entry["workload"], entry["n_tracks"])
    cfg = dataclasses.asdict(w.model)
    ref = O.forward(cfg, blob, tb.hits, tb.n_hits)
    for order in E.ORDERS:
        e = track_errors(E.forward(cfg, blob, tb.hits, tb.n_hits, order=order), ref)
        got = {"mean": float(e.mean()), "p90": float(np.percentile(e, 90)), "max": float(e.max())}
        for k in ("mean", "p90", "max"):
            want = entry[order][k]
            assert abs(got[k] - want) <= 0.05 * want, (order, k, got[k], want)
