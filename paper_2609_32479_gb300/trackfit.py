"""Thin ctypes binding of the C-ABI in include/trackfit.h.

Argument marshalling only: every step of the encoder runs in the CUDA kernels of
libtrackfit.so.  There is no CPU fallback; if the library is missing, load()
raises.  Device buffers are torch CUDA tensors (torch supplies memory and
streams), host buffers are numpy arrays."""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

from . import workloads as W

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libtrackfit.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_OOM, ERR_BAD_HITS, ERR_TIMEOUT = range(7)
ABI_VERSION = 3
MAX_FEATURES = 16

# every function declared in include/trackfit.h
EXPORTS = ("trackfit_weight_count", "trackfit_create", "trackfit_forward", "trackfit_forward_ex",
           "trackfit_forward_host", "trackfit_device_errors", "trackfit_path_name", "trackfit_set_path",
           "trackfit_destroy", "trackfit_strerror", "trackfit_debug_scan", "trackfit_debug_umma",
           "trackfit_profile", "trackfit_profile_read", "trackfit_forward_noalloc",
           "trackfit_debug_schedule", "trackfit_debug_wait_limit", "trackfit_debug_alloc", "trackfit_seed",
           "trackfit_decode", "trackfit_forward_packed", "trackfit_last_error")


class Config(ctypes.Structure):
    _fields_ = [("abi_version", ctypes.c_int32), ("max_hits", ctypes.c_int32),
                ("n_features", ctypes.c_int32), ("n_fourier", ctypes.c_int32),
                ("d_model", ctypes.c_int32), ("d_hidden", ctypes.c_int32), ("n_layers", ctypes.c_int32),
                ("head_hidden", ctypes.c_int32), ("n_quantiles", ctypes.c_int32),
                ("precision", ctypes.c_int32), ("pool", ctypes.c_int32), ("topology", ctypes.c_int32),
                ("n_heads", ctypes.c_int32),
                ("feat_min", ctypes.c_float * MAX_FEATURES), ("feat_max", ctypes.c_float * MAX_FEATURES),
                ("fourier_scale", ctypes.c_float * 16), ("rms_eps", ctypes.c_float)]


class TrackfitError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        detail = ""
        if status in (ERR_CUDA, ERR_OOM):
            detail = load().trackfit_last_error().decode()
        super().__init__(f"{what}: {strerror(status)} (status {status})" + (f" [{detail}]" if detail else ""))


_lib: Optional[ctypes.CDLL] = None


def load() -> ctypes.CDLL:
    """Open libtrackfit.so (built by paper_2609_32479_gb300.build); raise if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; "
                           f"g.build()'` (there is no CPU fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.trackfit_weight_count.argtypes = [ctypes.POINTER(Config)]
    lib.trackfit_weight_count.restype = ctypes.c_size_t
    lib.trackfit_create.argtypes = [ctypes.POINTER(Config), vp, ctypes.c_size_t, ctypes.POINTER(vp)]
    lib.trackfit_create.restype = ctypes.c_int
    lib.trackfit_forward.argtypes = [vp, vp, vp, i64, vp, vp]
    lib.trackfit_forward.restype = ctypes.c_int
    lib.trackfit_forward_ex.argtypes = [vp, vp, vp, i64, vp, vp, vp, vp]
    lib.trackfit_forward_ex.restype = ctypes.c_int
    lib.trackfit_forward_host.argtypes = [vp, vp, vp, i64, vp, vp]
    lib.trackfit_forward_host.restype = ctypes.c_int
    lib.trackfit_device_errors.argtypes = [vp, vp, ctypes.POINTER(i64)]
    lib.trackfit_device_errors.restype = ctypes.c_int
    lib.trackfit_path_name.argtypes = [vp]
    lib.trackfit_path_name.restype = ctypes.c_char_p
    lib.trackfit_set_path.argtypes = [vp, ctypes.c_int]
    lib.trackfit_set_path.restype = ctypes.c_int
    lib.trackfit_destroy.argtypes = [vp]
    lib.trackfit_destroy.restype = None
    lib.trackfit_strerror.argtypes = [ctypes.c_int]
    lib.trackfit_strerror.restype = ctypes.c_char_p
    lib.trackfit_last_error.argtypes = []
    lib.trackfit_last_error.restype = ctypes.c_char_p
    lib.trackfit_debug_scan.argtypes = [vp, vp, vp, vp, i64, i32, i32, vp, vp, vp]
    lib.trackfit_debug_scan.restype = ctypes.c_int
    lib.trackfit_debug_umma.argtypes = [vp, vp, vp, i32, vp, vp]
    lib.trackfit_debug_umma.restype = ctypes.c_int
    lib.trackfit_profile.argtypes = [vp, ctypes.c_int]
    lib.trackfit_profile.restype = ctypes.c_int
    lib.trackfit_profile_read.argtypes = [vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64)]
    lib.trackfit_profile_read.restype = ctypes.c_int
    lib.trackfit_forward_noalloc.argtypes = [ctypes.POINTER(Config), vp, vp, vp, i64, vp, vp]
    lib.trackfit_forward_noalloc.restype = ctypes.c_int
    lib.trackfit_debug_schedule.argtypes = [ctypes.POINTER(Config), ctypes.POINTER(i64), i32, vp, i64]
    lib.trackfit_debug_schedule.restype = ctypes.c_int
    lib.trackfit_debug_wait_limit.argtypes = [vp, i64, i32]
    lib.trackfit_debug_wait_limit.restype = ctypes.c_int
    lib.trackfit_debug_alloc.argtypes = [i64, ctypes.POINTER(i64)]
    lib.trackfit_debug_alloc.restype = i64
    lib.trackfit_seed.argtypes = [vp, i32, vp, i64, i32, ctypes.c_double, vp, vp, i32, vp]
    lib.trackfit_seed.restype = ctypes.c_int
    lib.trackfit_decode.argtypes = [vp, vp, i64, vp, vp]
    lib.trackfit_decode.restype = ctypes.c_int
    lib.trackfit_forward_packed.argtypes = [vp, vp, i64, vp, i64, vp, vp]
    lib.trackfit_forward_packed.restype = ctypes.c_int
    _lib = lib
    return lib


def strerror(status: int) -> str:
    return load().trackfit_strerror(int(status)).decode()


def make_config(m: W.ModelConfig) -> Config:
    c = Config()
    c.abi_version = ABI_VERSION
    c.max_hits, c.n_features, c.n_fourier = m.max_hits, m.n_features, m.n_fourier
    c.d_model, c.d_hidden, c.n_layers = m.d_model, m.d_hidden, m.n_layers
    c.head_hidden, c.n_quantiles = m.head_hidden, m.n_quantiles
    c.precision, c.pool, c.topology = m.precision, m.pool, m.topology
    c.n_heads = m.n_heads
    for i in range(m.n_features):
        c.feat_min[i], c.feat_max[i] = m.feat_min[i], m.feat_max[i]
    for i in range(16):
        c.fourier_scale[i] = m.fourier_scale[i]
    c.rms_eps = m.rms_eps
    return c


def weight_count(m: W.ModelConfig) -> int:
    c = make_config(m)
    return int(load().trackfit_weight_count(ctypes.byref(c)))


def schedule_counts(m: W.ModelConfig, with_codes: bool = False):
    """Per-tile totals of the tensor-core path's block schedule (host only): dict
    with blocks, mmas, w_e, w_h, c_acc, c_hb (and, with_codes, "codes": each block's
    wait | commit << 2 in issue order); None when m does not run on that path."""
    c = make_config(m)
    out = (ctypes.c_int64 * 6)()
    lib = load()
    st = lib.trackfit_debug_schedule(ctypes.byref(c), out, 6, None, 0)
    if st == ERR_UNSUPPORTED:
        return None
    if st != OK:
        raise TrackfitError(st, "trackfit_debug_schedule")
    res = dict(zip(("blocks", "mmas", "w_e", "w_h", "c_acc", "c_hb"), (int(v) for v in out)))
    if with_codes:
        codes = (ctypes.c_uint8 * res["blocks"])()
        st = lib.trackfit_debug_schedule(ctypes.byref(c), out, 6, codes, res["blocks"])
        if st != OK:
            raise TrackfitError(st, "trackfit_debug_schedule")
        res["codes"] = list(codes)
    return res


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def _dev(t, dtype_name: str):
    if t is None:
        return None
    if not (t.is_cuda and t.is_contiguous() and str(t.dtype) == dtype_name):
        raise ValueError(f"expected a contiguous CUDA {dtype_name} tensor, got {t.dtype} on {t.device}")
    return t.data_ptr()


class Trackfit:
    """A library handle: trackfit_create on construction, trackfit_destroy on close()."""

    def __init__(self, model: W.ModelConfig, weights: np.ndarray):
        self.lib = load()
        self.model = model
        self._cfg = make_config(model)
        w = np.ascontiguousarray(weights, dtype=np.float32)
        h = ctypes.c_void_p()
        st = self.lib.trackfit_create(ctypes.byref(self._cfg), w.ctypes.data, w.size, ctypes.byref(h))
        if st != OK:
            raise TrackfitError(st, "trackfit_create")
        self._h = h

    @property
    def handle(self) -> int:
        return self._h.value

    @property
    def path(self) -> str:
        return self.lib.trackfit_path_name(self._h).decode()

    def set_path(self, path: int) -> None:
        st = self.lib.trackfit_set_path(self._h, int(path))
        if st != OK:
            raise TrackfitError(st, "trackfit_set_path")

    def forward(self, hits, n_hits, out, stream=None, quantiles=None, pooled=None) -> None:
        """Device tensors: hits [B, T, F] f32 (F = n_features), n_hits [B] i32, out
        [B, 5] f32; optional quantiles [B, 5, n_quantiles] and pooled [B, P] f32."""
        B = int(n_hits.shape[0])
        m = self.model
        if tuple(hits.shape) != (B, m.max_hits, m.n_features) or tuple(out.shape) != (B, 5):
            raise ValueError(f"forward: hits must be [{B}, {m.max_hits}, {m.n_features}] and out [{B}, 5]")
        if quantiles is not None and tuple(quantiles.shape) != (B, 5, m.n_quantiles):
            raise ValueError(f"forward: quantiles must be [{B}, 5, {m.n_quantiles}]")
        if pooled is not None and tuple(pooled.shape) != (B, m.pooled_dim):
            raise ValueError(f"forward: pooled must be [{B}, {m.pooled_dim}]")
        args = (self._h, _dev(hits, "torch.float32"), _dev(n_hits, "torch.int32"), B, _dev(out, "torch.float32"))
        if quantiles is None and pooled is None:
            st = self.lib.trackfit_forward(*args, _stream_handle(stream))
        else:
            st = self.lib.trackfit_forward_ex(*args, _dev(quantiles, "torch.float32"),
                                              _dev(pooled, "torch.float32"), _stream_handle(stream))
        if st != OK:
            raise TrackfitError(st, "trackfit_forward")

    def forward_packed(self, hits, offsets, out, stream=None) -> None:
        """Device tensors: hits [N, F] f32 (all tracks back to back, F = n_features),
        offsets [B + 1] i64 (track b = rows offsets[b] .. offsets[b + 1] - 1), out
        [B, 5] f32."""
        B = int(offsets.shape[0]) - 1
        F = self.model.n_features
        if hits.dim() != 2 or int(hits.shape[1]) != F or tuple(out.shape) != (B, 5):
            raise ValueError(f"forward_packed: hits must be [N, {F}], offsets [B + 1], out [B, 5]")
        st = self.lib.trackfit_forward_packed(self._h, _dev(hits, "torch.float32"), int(hits.shape[0]),
                                              _dev(offsets, "torch.int64"), B, _dev(out, "torch.float32"),
                                              _stream_handle(stream))
        if st != OK:
            raise TrackfitError(st, "trackfit_forward_packed")

    def forward_host(self, hits: np.ndarray, n_hits: np.ndarray, out: np.ndarray, stream=None) -> None:
        """Host arrays (ideally pinned): copies in, runs, copies out, synchronises."""
        for a, dt in ((hits, np.float32), (n_hits, np.int32), (out, np.float32)):
            if a.dtype != dt or not a.flags["C_CONTIGUOUS"]:
                raise ValueError("host buffers must be C-contiguous float32/int32/float32")
        st = self.lib.trackfit_forward_host(self._h, hits.ctypes.data, n_hits.ctypes.data, int(n_hits.shape[0]),
                                            out.ctypes.data, _stream_handle(stream))
        if st != OK:
            raise TrackfitError(st, "trackfit_forward_host")

    def forward_host_ptr(self, hits_ptr: int, n_ptr: int, B: int, out_ptr: int, stream=None) -> None:
        st = self.lib.trackfit_forward_host(self._h, hits_ptr, n_ptr, int(B), out_ptr, _stream_handle(stream))
        if st != OK:
            raise TrackfitError(st, "trackfit_forward_host")

    def device_errors(self, stream=None):
        """(status, n_bad): reads and resets the device error counters (synchronises)."""
        n = ctypes.c_int64(0)
        st = self.lib.trackfit_device_errors(self._h, _stream_handle(stream), ctypes.byref(n))
        return st, int(n.value)

    def profile(self, enable: bool) -> None:
        st = self.lib.trackfit_profile(self._h, 1 if enable else 0)
        if st != OK:
            raise TrackfitError(st, "trackfit_profile")

    def profile_read(self):
        """(summed main-kernel milliseconds, timed launches) since the last read."""
        ms, n = ctypes.c_double(0.0), ctypes.c_int64(0)
        st = self.lib.trackfit_profile_read(self._h, ctypes.byref(ms), ctypes.byref(n))
        if st != OK:
            raise TrackfitError(st, "trackfit_profile_read")
        return ms.value, n.value

    def debug_wait_limit(self, limit_ns: int, hold_tile: int = -1) -> None:
        """Test hook: bounded-wait limit of the fused kernel and a held hand-over."""
        st = self.lib.trackfit_debug_wait_limit(self._h, int(limit_ns), int(hold_tile))
        if st != OK:
            raise TrackfitError(st, "trackfit_debug_wait_limit")

    def close(self) -> None:
        if getattr(self, "_h", None) is not None and self._h.value:
            self.lib.trackfit_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()


def debug_scan(a, b, x, n_hits, h_fwd, h_bwd, stream=None) -> None:
    """Device test hook for the masked linear recurrence (both directions)."""
    B, T, C = a.shape
    st = load().trackfit_debug_scan(_dev(a, "torch.float32"), _dev(b, "torch.float32"), _dev(x, "torch.float32"),
                                    _dev(n_hits, "torch.int32"), B, T, C, _dev(h_fwd, "torch.float32"),
                                    _dev(h_bwd, "torch.float32"), _stream_handle(stream))
    if st != OK:
        raise TrackfitError(st, "trackfit_debug_scan")


def debug_umma(tf: "Trackfit", A, Bkn, D, stream=None) -> None:
    """Device test hook: D[128][128] = A[128][K] * Bkn[K][128] (bf16 bits in int16 tensors)."""
    K = int(A.shape[1])
    st = load().trackfit_debug_umma(tf._h, _dev(A, "torch.int16"), _dev(Bkn, "torch.int16"), K,
                                    _dev(D, "torch.float32"), _stream_handle(stream))
    if st != OK:
        raise TrackfitError(st, "trackfit_debug_umma")


def forward_noalloc(model: W.ModelConfig, weights, hits, n_hits, out, stream=None) -> None:
    """No-allocation forward: device fp32 weight blob, hits, n_hits and out as
    torch CUDA tensors; the library's static device scratch supplies the workspace."""
    B = int(n_hits.shape[0])
    if tuple(n_hits.shape) != (B,):
        raise ValueError(f"n_hits must be [B], got {tuple(n_hits.shape)}")
    if tuple(hits.shape) != (B, model.max_hits, model.n_features):
        raise ValueError(f"hits must be [{B}, {model.max_hits}, {model.n_features}], got {tuple(hits.shape)}")
    if tuple(out.shape) != (B, 5):
        raise ValueError(f"out must be [{B}, 5], got {tuple(out.shape)}")
    if int(weights.numel()) != weight_count(model):
        raise ValueError(f"weights hold {int(weights.numel())} values, the model needs {weight_count(model)}")
    cfg = make_config(model)
    st = load().trackfit_forward_noalloc(ctypes.byref(cfg), _dev(weights, "torch.float32"),
                                         _dev(hits, "torch.float32"), _dev(n_hits, "torch.int32"),
                                         int(n_hits.shape[0]), _dev(out, "torch.float32"), _stream_handle(stream))
    if st != OK:
        raise TrackfitError(st, "trackfit_forward_noalloc")


def debug_alloc(fail_nth: int = 0):
    """Test hook: (device allocations the library holds, allocations attempted
    since the previous call); fail_nth > 0 makes that allocation from now fail."""
    att = ctypes.c_int64(0)
    live = load().trackfit_debug_alloc(int(fail_nth), ctypes.byref(att))
    return int(live), int(att.value)


def seed(hits, n_hits, b_field: float, seed_out, features_out=None, stream=None, in_place_at=None) -> None:
    """Analytic fp64 seed (device tensors): hits [B, T, F] f32 (x, y, z first), n_hits
    [B] i32 -> seed_out [B, 5] f64 and the residual features: into features_out
    [B, T, 3] f32, or, with in_place_at = c, into columns c..c+2 of hits itself."""
    B, T, F = int(hits.shape[0]), int(hits.shape[1]), int(hits.shape[2])
    if tuple(n_hits.shape) != (B,) or tuple(seed_out.shape) != (B, 5):
        raise ValueError("seed: n_hits must be [B] and seed_out [B, 5]")
    hp = _dev(hits, "torch.float32")
    if in_place_at is not None:
        if not 3 <= in_place_at <= F - 3 or (4 * in_place_at) % 16:
            raise ValueError("seed: in_place_at must leave x, y, z alone, fit the row, and be 16-byte aligned")
        fp, fs = hp + 4 * int(in_place_at), F
    else:
        if features_out is not None and tuple(features_out.shape) != (B, T, 3):
            raise ValueError("seed: features_out must be [B, T, 3]")
        fp, fs = _dev(features_out, "torch.float32"), 3
    st = load().trackfit_seed(hp, F, _dev(n_hits, "torch.int32"), B, T, float(b_field),
                              _dev(seed_out, "torch.float64"), fp, fs, _stream_handle(stream))
    if st != OK:
        raise TrackfitError(st, "trackfit_seed")


def decode(seed_t, corrections, out, stream=None) -> None:
    """Seed decode (device tensors): seed [B, 5] f64, corrections [B, 5] f32 -> out [B, 5] f32."""
    B = int(seed_t.shape[0])
    if tuple(seed_t.shape) != (B, 5) or tuple(corrections.shape) != (B, 5) or tuple(out.shape) != (B, 5):
        raise ValueError("decode: seed, corrections and out must be [B, 5]")
    st = load().trackfit_decode(_dev(seed_t, "torch.float64"), _dev(corrections, "torch.float32"), B,
                                _dev(out, "torch.float32"), _stream_handle(stream))
    if st != OK:
        raise TrackfitError(st, "trackfit_decode")
