"""Shared test helpers: config conversion and the parity metric."""
import dataclasses

import numpy as np


def cfg_dict(model):
    """The oracle takes the model configuration as a plain dict."""
    return dataclasses.asdict(model)


def parity_error(got, ref):
    """Per output column j: max_b |g_bj - r_bj| / max(|r_bj|, RMS_b(r_.j)).

    A plain relative error is unbounded for outputs near zero; the floor at the
    column's RMS makes it a relative error for outputs at or above the typical
    magnitude and an error relative to that magnitude below it."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    rms = np.sqrt(np.mean(ref * ref, axis=0))
    den = np.maximum(np.abs(ref), rms[None, :])
    return np.max(np.abs(got - ref) / den, axis=0)


FP32_TOL = 1e-5
BF16_TOL = 2e-3
