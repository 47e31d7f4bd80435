"""Shared test helpers: config conversion and the parity metric."""
import dataclasses

import numpy as np


def cfg_dict(model):
    """The oracle takes the model configuration as a plain dict."""
    return dataclasses.asdict(model)


def normalised_errors(got, ref):
    """Per track b and output column j: |g_bj - r_bj| / max(|r_bj|, RMS_b(r_.j)).

    A plain relative error is unbounded for outputs near zero; the floor at the
    column's RMS makes it a relative error for outputs at or above the typical
    magnitude and an error relative to that magnitude below it."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    rms = np.sqrt(np.mean(ref * ref, axis=0))
    return np.abs(got - ref) / np.maximum(np.abs(ref), rms[None, :])


def track_errors(got, ref):
    """Per track: the largest normalised error over its output columns."""
    return np.max(normalised_errors(got, ref), axis=1)


def parity_error(got, ref):
    """Max over tracks of the normalised error, per output column."""
    return np.max(normalised_errors(got, ref), axis=0)


FP32_TOL = 1e-5         # every track, fp32 path
FP16_TOL = 2e-3         # every track, fp16 operands
# bf16 operands: the bars come from the fp32 emulation of the oracle on the same
# tracks (oracle/fp32_emulation.py), in each of its accumulation orders: steps
# of 16 products rounding to nearest, or toward zero as the tensor core does,
# the second MLP product accumulating onto x' as on the tensor-core path.  Per
# track error e_b = max over the outputs of the normalised error.  The gate
# holds the mean and the 90th percentile of e_b within BF16_BULK_FACTOR of the
# worse emulation's (the measured spread between correct fp32 evaluations of
# the same arithmetic: the tensor-core path's mean and p90 came within 1.02-1.25
# of the emulation's on every 500-track chunk of medium and sweep8) and the
# maximum within
# BF16_MAX_FACTOR (the maximum of a few hundred tracks is an extreme value that
# scatters by tens of percent between two correct evaluations; the bar catches
# a wrong track, whose error is of order one).  No bar need be below BF16_FLOOR.
BF16_BULK_FACTOR = 1.3
BF16_MAX_FACTOR = 2.0
BF16_FLOOR = 1e-4
EVERY_TRACK_BAR = 2e-3  # the stated bar for every track, reported beside the gate


def emulations(model, blob, hits, n_hits):
    """The fp32 emulation of the oracle in each accumulation order (mean pooling)."""
    from oracle import fp32_emulation as E
    cfg = dataclasses.asdict(model)
    return [E.forward(cfg, blob, hits, n_hits, order=o) for o in E.ORDERS]


def bf16_bars(ref, emuls):
    """(mean bar, p90 bar, max bar) of the per-track error, from emulation outputs
    on the same tracks."""
    es = [track_errors(e, ref) for e in emuls]
    mean = max(float(e.mean()) for e in es)
    p90 = max(float(np.percentile(e, 90)) for e in es)
    mx = max(float(e.max()) for e in es)
    return (max(BF16_BULK_FACTOR * mean, BF16_FLOOR), max(BF16_BULK_FACTOR * p90, BF16_FLOOR),
            max(BF16_MAX_FACTOR * mx, BF16_FLOOR))


def parity_ok(got, ref, precision, emul=None):
    """The parity gate of one precision; returns (ok, summary string).  For bf16
    operands emul must hold the fp32 emulation's outputs on the same tracks (one
    array or a list, see emulations())."""
    e = track_errors(got, ref)
    mx = float(e.max())
    if precision == 0:
        return bool(mx <= FP32_TOL), f"max {mx:.3e} (tol {FP32_TOL})"
    if precision == 2:
        return bool(mx <= FP16_TOL), f"max {mx:.3e} (tol {FP16_TOL})"
    if emul is None:
        raise ValueError("the bf16 gate needs the fp32 emulation's outputs on the same tracks")
    emuls = list(emul) if isinstance(emul, (list, tuple)) else [emul]
    bmean, b90, bmx = bf16_bars(ref, emuls)
    mean, p90 = float(e.mean()), float(np.percentile(e, 90))
    return bool(mean <= bmean and p90 <= b90 and mx <= bmx), \
        (f"per-track mean {mean:.3e} (bar {bmean:.3e}), p90 {p90:.3e} (bar {b90:.3e}), "
         f"max {mx:.3e} (bar {bmx:.3e}); every track within {EVERY_TRACK_BAR}: {'yes' if mx <= EVERY_TRACK_BAR else 'no'}")
