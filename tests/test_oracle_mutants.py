"""Planted mistakes in the oracle must be caught by its pins.

Each mutant rewrites one expression of one oracle function: a dropped term, a wrong
sign, a swapped operand, an index off by one, the kinds of slip a restatement of
Sec. 3.2 / Eq. 2 can make.  The rewritten function is installed in the oracle
module for the duration of the test (CPU only, nothing else is touched) and every
pin of tests/test_oracle_units.py and tests/test_oracle_model.py (for the
analytic-seed oracle: tests/test_oracle_seed.py) runs against it; at least one pin
must fail.  A mutant that survives marks a gap in the pins."""
import inspect
import textwrap

import pytest

from oracle import seed_oracle as SO
from oracle import trackfit_oracle as O
from tests import test_oracle_attention as PA
from tests import test_oracle_concat as PC
from tests import test_oracle_model as PM
from tests import test_oracle_seed as PS
from tests import test_oracle_units as PU

# mutants may overflow or cast NaN on the way to failing a pin
pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")

# (id, oracle function, original text, mutated text)
MUTANTS = [
    ("bf16-truncates", "bf16_round", "((bits + half + lsb) >> drop) << drop", "(bits >> drop) << drop"),
    ("bf16-ties-up", "bf16_round", "((bits + half + lsb) >> drop)", "((bits + half + np.uint64(1)) >> drop)"),
    ("sigmoid-sign", "sigmoid", "np.exp(-x)", "np.exp(x)"),
    ("silu-drops-x", "silu", "return x * sigmoid(x)", "return sigmoid(x)"),
    ("rmsnorm-no-sqrt", "rmsnorm", "np.sqrt(ms + eps)", "(ms + eps)"),
    ("rmsnorm-divides-by-gain", "rmsnorm", "* g", "/ g"),
    ("rmsnorm-sum-not-mean", "rmsnorm", "np.mean(x * x", "np.sum(x * x"),
    ("normalise-sign", "normalise", "- lo) / (hi - lo)", "+ lo) / (hi - lo)"),
    ("normalise-range-from-max", "normalise", "/ (hi - lo)", "/ hi"),
    ("fourier-no-pi", "fourier", "np.pi * u", "u"),
    ("fourier-sin-cos-swapped", "fourier", "[np.sin(arg), np.cos(arg)]", "[np.cos(arg), np.sin(arg)]"),
    ("fourier-feature-major-flipped", "fourier", "arg = np.pi * u[..., :, None] * s",
     "arg = np.swapaxes(np.pi * s[:, None] * u[..., None, :], -1, -2)[..., ::-1, :]"),
    ("scan-no-mask", "linear_scan", "h = np.where(v, a[:, t] * h + b[:, t] * x[:, t], h)",
     "h = a[:, t] * h + b[:, t] * x[:, t]"),
    ("scan-pads-keep-state", "linear_scan", "out[:, t] = np.where(v, h, 0.0)", "out[:, t] = h"),
    ("scan-drops-b", "linear_scan", "b[:, t] * x[:, t]", "x[:, t]"),
    ("scan-ignores-reverse", "linear_scan", "steps = range(T - 1, -1, -1) if reverse else range(T)",
     "steps = range(T)"),
    ("mingru-gates-swapped", "mingru_layer_scans", "linear_scan(1.0 - z_f, z_f, n_f", "linear_scan(z_f, 1.0 - z_f, n_f"),
    ("mingru-reverse-takes-forward-gate", "mingru_layer_scans", "linear_scan(1.0 - z_b, z_b, n_b",
     "linear_scan(1.0 - z_f, z_f, n_b"),
    ("mingru-reverse-not-reversed", "mingru_layer_scans", "valid, reverse=True", "valid, reverse=False"),
    ("layer-no-prenorm", "encoder_layer", 'xh = rmsnorm(x, W[p + "g"], cfg["rms_eps"])', "xh = x"),
    ("layer-z-not-gated", "encoder_layer", "z_f = sigmoid(proj[..., 0:H])", "z_f = proj[..., 0:H]"),
    ("layer-n-rows-swapped", "encoder_layer", "n_f = proj[..., H:2 * H]", "n_f = proj[..., 3 * H:4 * H]"),
    ("layer-gate-rows-offset", "encoder_layer", "proj[..., 4 * H:4 * H + D]", "proj[..., 4 * H - D:4 * H]"),
    ("layer-no-output-gate", "encoder_layer", "x1 = x + m * gate", "x1 = x + m"),
    ("layer-no-merge-residual", "encoder_layer", "x1 = x + m * gate", "x1 = m * gate"),
    ("layer-directions-swapped", "encoder_layer", "[h_f, h_b]", "[h_b, h_f]"),
    ("layer-mlp-residual-dropped", "encoder_layer", "x2 = x1 + _lin(", "x2 = _lin("),
    ("layer-mlp-reads-x", "encoder_layer", 'u = silu(_lin(x1, W[p + "w1"]', 'u = silu(_lin(x, W[p + "w1"]'),
    ("layer-pads-not-zeroed", "encoder_layer", "np.where(valid[..., None], x2, 0.0)", "x2"),
    ("lin-weight-not-transposed", "_lin", "prec).T + b", "prec) + b"),
    ("lin-drops-bias", "_lin", "prec).T + b", "prec).T"),
    ("embed-no-silu", "embed", "hdn = silu(", "hdn = ("),
    ("pool-divides-by-T", "pool", "s / n_hits[:, None].astype(np.float64)", "s / x.shape[1]"),
    ("pool-sums-pads", "pool", "np.sum(np.where(valid[..., None], x, 0.0), axis=1)", "np.sum(x, axis=1)"),
    ("pool-endpoint-index", "pool", "h_f[idx, n_hits - 1]", "h_f[idx, n_hits - 2]"),
    ("pool-endpoint-reverse-index", "pool", "h_b[:, 0]", "h_b[:, 1]"),
    ("head-median-index", "head", "q[:, :, nq // 2]", "q[:, :, nq // 2 + 1]"),
    ("head-quantile-major", "head", "q.reshape(q.shape[0], q.shape[1] // nq, nq)",
     "q.reshape(q.shape[0], nq, q.shape[1] // nq).transpose(0, 2, 1)"),
    ("head-no-norm", "head", 'hn = rmsnorm(pv, W["head.g"], cfg["rms_eps"])', "hn = pv"),
    ("head-no-silu", "head", "hid = silu(", "hid = ("),
    ("concat-directions-swapped", "encoder_layer_concat", "np.concatenate([h_f, h_b]", "np.concatenate([h_b, h_f]"),
    ("concat-z-not-gated", "encoder_layer_concat", "z_f = sigmoid(proj[..., 0:H])", "z_f = proj[..., 0:H]"),
    ("concat-candidate-activated", "encoder_layer_concat", "n_f = proj[..., H:2 * H]", "n_f = np.tanh(proj[..., H:2 * H])"),
    ("concat-reverse-reads-forward", "encoder_layer_concat", "n_b = proj[..., 3 * H:4 * H]", "n_b = proj[..., H:2 * H]"),
    ("concat-normalised", "encoder_layer_concat", 'proj = _lin(x, W[p + "w_in"]', 'proj = _lin(rmsnorm(x, 1.0, 1e-6), W[p + "w_in"]'),
    ("attention-scaled-by-width", "attention", "/ np.sqrt(dh)", "/ np.sqrt(D)"),
    ("attention-no-key-mask", "attention", "sc = np.where(valid[:, None, None, :], sc, -np.inf)", "sc = sc"),
    ("attention-scores-transposed", "attention", '"bthd,bshd->bhts"', '"bthd,bshd->bhst"'),
    ("attention-not-normalised", "attention", "w = w / np.sum(w, axis=-1, keepdims=True)", "w = w"),
    ("attention-heads-interleaved", "attention", ".reshape(B, T, n_heads, dh) for a in (q, k, v)",
     ".reshape(B, T, dh, n_heads).swapaxes(2, 3) for a in (q, k, v)"),
    ("attention-pads-not-zeroed", "attention", "return np.where(valid[..., None], o, 0.0)", "return o"),
    ("attnlayer-no-prenorm", "encoder_layer_attention", 'qkv = _lin(rmsnorm(x, W[p + "g1"], cfg["rms_eps"])',
     "qkv = _lin(x"),
    ("attnlayer-k-v-swapped", "encoder_layer_attention", "qkv[..., D:2 * D], qkv[..., 2 * D:3 * D]",
     "qkv[..., 2 * D:3 * D], qkv[..., D:2 * D]"),
    ("attnlayer-no-attention-residual", "encoder_layer_attention", "x1 = x + _lin(o", "x1 = _lin(o"),
    ("attnlayer-mlp-reads-x", "encoder_layer_attention", 'rmsnorm(x1, W[p + "g2"]', 'rmsnorm(x, W[p + "g2"]'),
    ("attnlayer-no-mlp-residual", "encoder_layer_attention", "x2 = x1 + _lin(u", "x2 = _lin(u"),
    ("attnlayer-pads-not-zeroed", "encoder_layer_attention", "return np.where(valid[..., None], x2, 0.0), None, None",
     "return x2, None, None"),
]


# mutants of the analytic-seed oracle (Sec. 3.1), caught by tests/test_oracle_seed.py
SEED_MUTANTS = [
    ("circle-centre-sign", "circle_through_three", "cy = (u1 - u2) / (2.0 * det)", "cy = (u2 - u1) / (2.0 * det)"),
    ("circle-no-inversion", "circle_through_three", "u1, v1 = a[..., 0] / na, a[..., 1] / na", "u1, v1 = a[..., 0], a[..., 1]"),
    ("seed-charge-sign", "seed_perigee", "q = -np.sign(cross)", "q = np.sign(cross)"),
    ("seed-perigee-far-side", "seed_perigee", "px, py = centre[..., 0] - R * ux, centre[..., 1] - R * uy",
     "px, py = centre[..., 0] + R * ux, centre[..., 1] + R * uy"),
    ("seed-d0-sign", "seed_perigee", "d0 = -px * np.sin(phi0) + py * np.cos(phi0)", "d0 = px * np.sin(phi0) + py * np.cos(phi0)"),
    ("seed-turning-reversed", "seed_perigee", "np.mod(-q * (g_h - g_p)", "np.mod(q * (g_h - g_p)"),
    ("seed-z0-from-h2", "seed_perigee", "z0 = h0[..., 2] - s0 * cot", "z0 = h0[..., 2] - s2 * cot"),
    ("seed-theta-complement", "seed_perigee", "theta = np.arctan2(1.0, cot)", "theta = np.arctan2(cot, 1.0)"),
    ("seed-pt-units", "seed_perigee", "pt = C_LIGHT * b_field * R / 1000.0", "pt = C_LIGHT * b_field * R / 100.0"),
    ("seed-qop-no-sin", "seed_perigee", "qop = q * np.sin(theta) / pt", "qop = q / pt"),
    ("triplet-no-separation", "seed_triplet", "> min_sep", "> -1.0"),
    ("helix-turns-wrong-way", "helix_point", "phi = phi0 - q * alpha", "phi = phi0 + q * alpha"),
    ("tangent-no-polar-angle", "helix_tangent", "st = np.sin(theta)", "st = 1.0"),
    ("residual-axes-swapped", "curvilinear_residuals", "return np.sum(r * U, axis=-1), np.sum(r * V, axis=-1)",
     "return np.sum(r * V, axis=-1), np.sum(r * U, axis=-1)"),
    ("residual-v-sign", "curvilinear_residuals", "V = np.cross(t, U)", "V = np.cross(U, t)"),
    ("residual-no-foot-search", "curvilinear_residuals", "a_new = a - step", "a_new = a"),
    ("residual-transverse-path", "curvilinear_residuals", "R * a / np.sin(theta)", "R * a"),
    ("residual-no-turn-choice", "curvilinear_residuals", "a = np.where(resolved, a + 2.0 * np.pi * turns, a)",
     "a = a"),
    ("residual-start-from-zero", "curvilinear_residuals", "np.mod(-q * (gh - g0) + np.pi, 2.0 * np.pi) - np.pi",
     "np.mod(-q * (gh - g0), 2.0 * np.pi)"),
    ("features-no-asinh", "seed_features", "np.arcsinh(du / scale_mm)", "du / scale_mm"),
    ("decode-phi-unwrapped", "decode", "out[..., 2] = np.pi - np.mod(np.pi - out[..., 2], 2.0 * np.pi)",
     "out[..., 2] = out[..., 2]"),
    ("decode-qop-absolute", "decode", "delta[..., 4] * (np.abs(seed[..., 4]) + QOP_EPS)", "delta[..., 4]"),
    ("decode-qop-no-floor", "decode", "(np.abs(seed[..., 4]) + QOP_EPS)", "np.abs(seed[..., 4])"),
]


def _pins(mods=None):
    """Every pin of the oracle test modules, parametrised cases expanded."""
    out = []
    for mod in (mods or (PU, PM, PC, PA)):
        for name, fn in sorted(vars(mod).items()):
            if not (name.startswith("test_") and callable(fn)):
                continue
            cases = [{}]
            for mark in getattr(fn, "pytestmark", []):
                if mark.name == "parametrize":
                    names = [n.strip() for n in mark.args[0].split(",")]
                    vals = mark.args[1]
                    cases = [dict(c, **dict(zip(names, v if len(names) > 1 else (v,)))) for c in cases for v in vals]
            for kw in cases:
                out.append((f"{mod.__name__.split('.')[-1]}::{name}{kw or ''}", fn, kw))
    return out


def _install(monkeypatch, fname, old, new, mod=O):
    src = textwrap.dedent(inspect.getsource(getattr(mod, fname)))
    assert src.count(old) == 1, f"mutation text not found once in {fname}: {old}"
    ns = {}
    exec(compile(src.replace(old, new, 1), f"<mutant of {fname}>", "exec"), vars(mod), ns)
    monkeypatch.setattr(mod, fname, ns[fname])


@pytest.mark.parametrize("mid,fname,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(monkeypatch, mid, fname, old, new):
    _install(monkeypatch, fname, old, new)
    caught = []
    for pid, fn, kw in _pins():
        try:
            fn(**kw)
        except Exception:   # an assertion, or the mutant breaking a shape
            caught.append(pid)
            break
    assert caught, f"mutant {mid} passes every oracle pin"


def test_unmutated_oracle_passes_every_pin():
    for pid, fn, kw in _pins():
        fn(**kw)


@pytest.mark.parametrize("mid,fname,old,new", SEED_MUTANTS, ids=[m[0] for m in SEED_MUTANTS])
def test_seed_pins_catch_mutant(monkeypatch, mid, fname, old, new):
    _install(monkeypatch, fname, old, new, mod=SO)
    for pid, fn, kw in _pins((PS,)):
        try:
            fn(**kw)
        except Exception:
            return
    raise AssertionError(f"mutant {mid} passes every seed pin")
