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


FP32_TOL = 1e-5
BF16_TOL = 2e-3          # bulk bar (90th percentile of tracks) for bf16 operands
BF16_TAIL_TOL = 1e-2     # every track, bf16 operands (rounding-boundary flips)
FP16_TOL = 2e-3          # every track, fp16 operands


def parity_ok(got, ref, precision):
    """The parity gate of one precision; returns (ok, summary string)."""
    e = normalised_errors(got, ref)
    mx = e.max()
    if precision == 0:
        return bool(mx <= FP32_TOL), f"max {mx:.3e} (tol {FP32_TOL})"
    if precision == 2:
        return bool(mx <= FP16_TOL), f"max {mx:.3e} (tol {FP16_TOL})"
    p90 = np.percentile(e, 90)
    return bool(p90 <= BF16_TOL and mx <= BF16_TAIL_TOL), \
        f"p90 {p90:.3e} (tol {BF16_TOL}), max {mx:.3e} (tol {BF16_TAIL_TOL})"
